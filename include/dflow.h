/*
 * dflow.h -- C ABI of the DFlow speculative-decoding round on one GPU.
 *
 * One round of block-diffusion speculative decoding with DFlow's verifier
 * information relay (arXiv 2609.06498):
 *
 *   dflow_draft_block   Sec. 3 Eq. 2 with Sec. 4.2 Eq. 4-5: the drafter predicts
 *                       B future tokens in one forward pass from mask embeddings,
 *                       relayed verifier states and the fused target context.
 *   dflow_verify_block  Sec. 3 Eq. 3 (target side) and Eq. 1: one target forward
 *                       over the anchor and the B proposals against the cached
 *                       K/V; per-row greedy predictions and fused features.
 *   dflow_accept_commit Sec. 3 Eq. 3: accepted prefix, bonus token, commit of
 *                       a+1 tokens, rollback of the rest.
 *   dflow_carry_hidden  Sec. 3 (context injected into draft K/V) and Sec. 4.2
 *                       (alignment: keep the shifted verifier states of the
 *                       rejected suffix and the two boundary tokens).
 *   dflow_round         the four calls above in order, for the whole batch.
 *   dflow_round_sampled one round at temperature 1 (Sec. 5.2): sampled
 *                       proposals, speculative-sampling acceptance.
 *
 * Conventions shared by every call
 *   - Pointers in dflow_weights and dflow_state and every output pointer are
 *     DEVICE pointers, owned by the caller and never freed by the library.
 *     Structs themselves are read on the host during the call only.
 *   - The library allocates no device memory after dflow_set_workspace: all
 *     scratch lives in the caller's workspace.
 *   - Every call is asynchronous on `stream` (a cudaStream_t passed as void*).
 *     Argument errors found on the host return a nonzero status synchronously
 *     and launch nothing.  Errors found on the device (sequence capacity
 *     exhausted, token id out of range, invalid carried count, a bounded wait
 *     that timed out) are written to *state->status; every later kernel of the
 *     library that indexes memory by device state (tokens, positions, pages,
 *     counts) returns without writing once it sees a nonzero status (the
 *     dense projections keep running on their fixed workspace buffers).
 *     Read it with dflow_read_status.
 *   - A handle is not thread safe and serves one stream at a time.
 *   - dtype DFLOW_F32: weights, activations, caches in fp32, fp32 arithmetic.
 *     dtype DFLOW_BF16: weights, caches, features and carry in bf16; fp32
 *     accumulation, fp32 residual stream and fp32 norms/softmax/rotary.
 *
 * Decoding state invariants (per sequence b, n = seq_len[b] committed tokens)
 *   tokens[b][0..n-1] committed; tokens[b][n-1] is the anchor.
 *   Target K/V and drafter context K/V are valid for positions 0..n-2.
 *   carry slot j (1..n_carry[b]) holds the relayed feature for draft row j.
 *   Block row i (0..B) of a round sits at position n-1+i.
 */
#ifndef DFLOW_H
#define DFLOW_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum dflow_status {
  DFLOW_OK = 0,
  DFLOW_ERR_INVALID_ARG = 1,    /* null pointer, bad size or shape, call order */
  DFLOW_ERR_CUDA = 2,           /* a CUDA runtime call failed */
  DFLOW_ERR_CAPACITY = 3,       /* a sequence would grow past max_ctx */
  DFLOW_ERR_DEVICE_TIMEOUT = 4, /* a bounded device wait gave up */
  DFLOW_ERR_UNSUPPORTED = 5,    /* shape or device outside what the kernels cover */
  DFLOW_ERR_BAD_STATE = 6       /* token / count out of range found on the device */
} dflow_status;

enum { DFLOW_F32 = 0, DFLOW_BF16 = 1 };

#define DFLOW_MAX_FEAT 8

/* Model and workload shape.  head_dim must be 64 or 128, d_model a multiple
 * of 128, d_inter a multiple of 64.  DFLOW_BF16 runs on the tensor-core
 * kernels: head_dim 128, page_size 64 and an sm_103 device (GB300; checked by
 * dflow_set_workspace); DFLOW_F32 (a parity model) on CUDA cores.  feat_layers are 1-indexed target layers
 * (Eq. 1 takes the residual stream after each of them). */
typedef struct dflow_config {
  int32_t dtype;
  int32_t d_model, n_layers, n_q_heads, n_kv_heads, head_dim, d_inter, vocab;
  int32_t draft_layers, n_feat, feat_layers[DFLOW_MAX_FEAT];
  int32_t block;     /* B: draft tokens per round; a block has B+1 rows */
  int32_t page_size; /* tokens per KV page */
  int32_t max_batch; /* most sequences per call */
  int32_t max_ctx;   /* token capacity of one sequence (multiple of page_size) */
  int32_t num_pages; /* pages in each K/V pool */
  float rope_theta, rms_eps, ln_eps;
} dflow_config;

/* One decoder layer (Qwen3 layout).  Matrices are row-major [out][in].
 *   w_qkv     [(Hq + 2 Hkv) * hd][d]: rows of Wq, then Wk, then Wv
 *   w_o       [d][Hq * hd]
 *   w_gate_up [2 * d_inter][d]: in groups of 128 rows, rows 0..63 are gate
 *             rows 64g..64g+63 and rows 64..127 the matching up rows
 *   w_down    [d][d_inter]
 * Norm gains are fp32 vectors of d (attn_norm, mlp_norm) or hd (q/k). */
typedef struct dflow_layer_weights {
  const void *w_qkv, *w_o, *w_gate_up, *w_down;
  const float *attn_norm, *mlp_norm, *q_norm, *k_norm;
} dflow_layer_weights;

/* target: host array of n_layers layers; draft: host array of draft_layers.
 * embed, lm_head [vocab][d] (LM head shared by target and drafter);
 * w_c [d][n_feat * d] (Eq. 1); relay_w1 [d][3d], relay_w2 [2d][d] (Eq. 4);
 * e_mask, ln_w, ln_b, c_norm, final norms: fp32 [d]. */
typedef struct dflow_weights {
  const void *embed, *lm_head;
  const float *final_norm;
  const dflow_layer_weights *target;
  const dflow_layer_weights *draft;
  const float *draft_final_norm;
  const void *w_c;
  const float *c_norm;
  const float *e_mask;
  const void *relay_w1, *relay_w2;
  const float *ln_w, *ln_b;
} dflow_weights;

/* Decoding state of `batch` sequences (device memory).
 *   tokens     int32 [batch][max_ctx]
 *   seq_len    int32 [batch]           n
 *   page_table int32 [batch][max_ctx / page_size]: page id of every logical
 *              page; fixed for the life of the sequence (commit and rollback
 *              move only seq_len)
 *   kv         target pool  [n_layers][num_pages][2][Hkv][page_size][hd]
 *   draft_kv   drafter pool [draft_layers][num_pages][2][Hkv][page_size][hd]
 *   carry      [batch][B][d]  (slot j at index j-1)
 *   n_carry    int32 [batch];  boundary int32 [batch][2] = (bonus, y_{a+1})
 *   active     int32 [batch]: 0 freezes a sequence (no state writes)
 *   status     int32 [1]: 0 or a dflow_status written by the device */
typedef struct dflow_state {
  int32_t batch;
  int32_t *tokens, *seq_len;
  const int32_t *page_table;
  void *kv, *draft_kv, *carry;
  int32_t *n_carry, *boundary, *active, *status;
} dflow_state;

typedef struct dflow_handle dflow_handle;

const char *dflow_status_string(dflow_status s);

/* Validate shapes, copy the weight pointer tables, pick kernels for the
 * current device.  Allocates host memory only. */
dflow_status dflow_create(const dflow_config *cfg, const dflow_weights *w, dflow_handle **out);
/* Device bytes of scratch the handle needs (activations for max_batch rows,
 * split-K / split-KV partials, the rotary table). */
dflow_status dflow_workspace_size(const dflow_handle *h, size_t *bytes);
/* Hand over scratch (>= dflow_workspace_size bytes, 256-byte aligned).  Fills
 * constant tables with a synchronous launch on the legacy default stream.
 * DFLOW_ERR_UNSUPPORTED for a bf16 handle on a device other than sm_103. */
dflow_status dflow_set_workspace(dflow_handle *h, void *dev, size_t bytes);
dflow_status dflow_destroy(dflow_handle *h);

/* Prompt processing (setup, not part of a round; Sec. 3 committed context):
 * runs the target over prompt[b][0..len_b-1] (device int32, row stride
 * prompt_stride), writes target K/V and drafter context for positions
 * 0..len_b-1, appends the greedy next token as the anchor, sets
 * seq_len = len_b + 1, n_carry = 0.  prompt_len_host: host int32 [batch]. */
dflow_status dflow_prefill(dflow_handle *h, dflow_state *st, const int32_t *prompt,
                           int32_t prompt_stride, const int32_t *prompt_len_host,
                           void *stream);

/* Sec. 3 Eq. 2 + Sec. 4.2 Eq. 4-5.  block_tokens int32 [batch][B+1]: row 0 =
 * anchor, rows 1..B = drafter argmax.  Reads tokens, seq_len, drafter
 * context, carry, n_carry, boundary.  If logits is non-null, also the
 * drafter's fp32 logits [batch][B+1][vocab] (row 0 included; a second pass
 * over the LM head, for tests). */
dflow_status dflow_draft_block(dflow_handle *h, dflow_state *st, int32_t *block_tokens, float *logits,
                               void *stream);

/* Sec. 3 Eq. 3 (target forward) + Eq. 1.  Reads block_tokens [batch][B+1];
 * writes target K/V at positions n-1..n-1+B, target_argmax int32
 * [batch][B+1] (row i = greedy prediction for position n+i), feats
 * [batch][B+1][d] (Eq. 1, model dtype) and, if logits is non-null, fp32
 * logits [batch][B+1][vocab]. */
dflow_status dflow_verify_block(dflow_handle *h, dflow_state *st, const int32_t *block_tokens,
                                int32_t *target_argmax, void *feats, float *logits,
                                void *stream);

/* Sec. 3 Eq. 3.  a = number of leading proposals with block[i] ==
 * target_argmax[i-1]; if forced_accept (int32 [batch], values 0..B) is
 * non-null it replaces a.  Commits block[1..a] and bonus target_argmax[a] to
 * tokens[n..n+a]; seq_len += a+1.  accept_len int32 [batch] (-1 for inactive
 * sequences); committed int32 [batch][B+1], -1 padded. */
dflow_status dflow_accept_commit(dflow_handle *h, dflow_state *st, const int32_t *block_tokens,
                                 const int32_t *target_argmax, const int32_t *forced_accept,
                                 int32_t *accept_len, int32_t *committed, void *stream);

/* Sec. 3 + Sec. 4.2, after dflow_accept_commit of the same round.  Feature
 * rows 0..a join the drafter context of every draft layer (k = RoPE(k_norm(
 * W_k f)), v = W_v f at positions n_old-1..n_old-1+a); rows a+1..B-1 become
 * carry slots 1..B-a-1; boundary = (bonus, block[a+1]) (-1 when a = B). */
dflow_status dflow_carry_hidden(dflow_handle *h, dflow_state *st, const int32_t *block_tokens,
                                const void *feats, const int32_t *accept_len, void *stream);

/* One full round: draft -> verify -> accept/commit -> carry, with block
 * tokens, predictions and features in the workspace.  relay = 0 runs the
 * DFlash baseline (nothing carried, mask embeddings only). */
dflow_status dflow_round(dflow_handle *h, dflow_state *st, const int32_t *forced_accept,
                         int32_t *accept_len, int32_t *committed, int32_t relay,
                         void *stream);

/* One full round at temperature 1 (Sec. 5.2, Table 1 T = 1 rows).  The paper
 * does not print its T = 1 rule; this round applies standard speculative
 * sampling per block position:
 *   - block row i = 1..B holds a sample y_i of q_i = softmax(drafter logits
 *     of row i);
 *   - proposal i is accepted while u_i < p_i(y_i) / q_i(y_i), p_i =
 *     softmax(target logits of verify row i-1);
 *   - the token after the a accepted proposals is drawn from max(0, p_i -
 *     q_i) normalised (i = a+1 <= B), or from p_{B+1} when a = B.
 * Commit, carry and relay follow dflow_round with that token as the bonus
 * and the first rejected proposal as boundary token.  Each draw is a
 * Gumbel-max sample argmax_v(log w_v - log(-log u_v)); u_v comes from a
 * SplitMix64 counter stream keyed by (seed, sequence index b, round_index,
 * block row, purpose 0 = proposal / 1 = acceptance test / 2 = committed
 * token), u_v = (2 (splitmix64(key ^ v) >> 41) + 1) / 2^24 with
 * key = splitmix64(seed ^ splitmix64(b << 48 ^ round_index << 24 ^
 * row << 8 ^ purpose)); the acceptance uniform of row i is v = 0 of its stream.
 * The caller advances round_index (0 <= round_index < 2^24) between rounds.
 * accept_len, committed: as for dflow_accept_commit.  draft_logits,
 * verify_logits: optional device fp32 [batch][B+1][vocab]; where non-null the
 * round writes that stage's logits there (and reads them back from there),
 * else it uses workspace memory.  bf16 and fp32 handles; the round streams
 * the LM head once per stage, as the greedy round does. */
dflow_status dflow_round_sampled(dflow_handle *h, dflow_state *st, uint64_t seed, int32_t round_index,
                                 int32_t *accept_len, int32_t *committed, int32_t relay,
                                 float *draft_logits, float *verify_logits, void *stream);

/* Sec. 5.2, Table 2 "Baseline": one step of plain autoregressive greedy
 * decoding of the target, for every active sequence: the last committed token
 * (position n-1) runs through the target against the cached K/V (its K/V are
 * written), and its greedy prediction is committed: tokens[n], seq_len = n+1.
 * token_out int32 [batch] (-1 for inactive sequences).  Afterwards nothing is
 * carried (n_carry = 0, boundary = -1).  draft_context = 1 also appends the
 * row's Eq. 1 feature to the drafter context, so dflow_round may follow; with
 * 0 (the plain baseline) the drafter context falls behind and no round should
 * follow on that state.  The step runs on the block-verify launches with the
 * anchor in every row of a B+1-row block (rows 1..B are dropped), so it needs
 * the same free capacity as a round (DFLOW_ERR_CAPACITY otherwise). */
dflow_status dflow_decode_step(dflow_handle *h, dflow_state *st, int32_t *token_out, int32_t draft_context,
                               void *stream);

/* Synchronises `stream`, then copies *state->status to *host_status. */
dflow_status dflow_read_status(dflow_handle *h, const dflow_state *st, int32_t *host_status,
                               void *stream);

/* ---- measurement (not part of the method) ----------------------------------
 * With profiling enabled, the library brackets every launch of a kernel class
 * with CUDA events on the launching stream and accumulates, per class, the
 * launch count, the summed event durations and the algorithmic DRAM bytes and
 * flops of those launches (weights + activations read, outputs written; for
 * attention the K/V bytes are not known on the host and are left at 0). */
enum { DFLOW_PROF_GEMM = 0, DFLOW_PROF_ATTN = 1, DFLOW_PROF_OTHER = 2, DFLOW_PROF_N = 3 };
typedef struct dflow_kernel_profile {
  int64_t launches;
  double total_ms;
  double alg_bytes;
  double alg_flops;
} dflow_kernel_profile;

/* Turn per-launch event timing on (1) or off (0); either way clears the record. */
dflow_status dflow_profile_enable(dflow_handle *h, int32_t enable);
/* Test hook: one projection out[m][n] = sum_k X[m][k] W[n][k] through the
 * library's GEMM kernels (path 0: CUDA-core kernel of fp32 handles; bf16
 * handles: path 1 the tcgen05 kernel of one projection, path 2 the persistent
 * tcgen05 launch the round uses for 16 to 128 rows (modes 0-3, K a multiple of
 * 64 and at least 256; fewer rows are refused before any launch), path 3 the
 * one-pass tcgen05 launch the round uses above 128 rows for shapes it suits;
 * else DFLOW_ERR_UNSUPPORTED), with the epilogue `mode`: 0 store fp32 out[M][ldo];
 * 1 add into fp32 out[M][ldo]; 2 SwiGLU of 128-row [64 gate | 64 up] groups
 * into model-dtype out[M][ldo] (N/2 features); 3 SiLU into model-dtype out;
 * 4 greedy argmax over n into int32 out[M] (M <= max_batch * max(B+1, 64)).
 * Uses the handle's workspace; asynchronous on `stream`; device errors go to
 * *status (int32 device word). */
dflow_status dflow_debug_gemm(dflow_handle *h, int32_t path, const void *W, int32_t N, int32_t K,
                              const void *X, int32_t M, int32_t ldx, int32_t mode, void *out,
                              int32_t ldo, int32_t *status, void *stream);

/* Greedy tokens without any device allocation (no counterpart in the paper:
 * an integration aid for callers that cannot allocate device memory, e.g. code
 * confined to a caller-owned memory pool or a plugin whose host owns all
 * allocations).  tokens[r] = argmax_v hidden[r] . lm_head[v] (ties to the
 * lowest id; -1 if a device error occurred), computed with the round's tensor-
 * core LM-head kernels.
 *   lm_head  bf16 [vocab][d], hidden bf16 [rows][d] (already final-normalised),
 *   tokens   int32 [rows]; all device pointers owned by the caller.
 * Limits: rows <= 64, vocab <= 262144 (else DFLOW_ERR_INVALID_ARG), d a
 * multiple of 64, sm_103 devices only (else DFLOW_ERR_UNSUPPORTED).
 * Scratch lives in a ~1 MiB array compiled into the library.  It becomes
 * device memory when the library's GPU code is loaded on a device (under
 * CUDA's default lazy loading: at the first call there; CUDA_MODULE_LOADING=
 * EAGER places it at library load) and is held until exit.  The first call on
 * a device looks up the array's address (once per device, under a lock, so
 * concurrent first calls are safe): make it at set-up, before any fixed-budget
 * window or stream capture.  Calls share the array and it keeps the last
 * call's contents; calls that overlap on the GPU race.  `stream` must belong to
 * the current device (else DFLOW_ERR_INVALID_ARG).  Calls no cudaMalloc/
 * cudaFree and no allocating library routine. */
dflow_status dflow_greedy_tokens_noalloc(const void *lm_head, int32_t vocab, int32_t d, const void *hidden,
                                         int32_t rows, int32_t *tokens, void *stream);

/* Test hook, host only (no GPU needed): the schedule the persistent tcgen05
 * launch gives one GEMM of N x K weights over M rows on Q four-CTA clusters,
 * computed by the functions the kernel itself evaluates.
 *   plan  int32 [8]: padded columns, tiles T, k-blocks kb, full tiles Tf,
 *         leftover tiles Tl, clusters per leftover tile ls, completion count of
 *         the GEMM, leftover part slots available
 *   ctas  int32 [Q*4][10], per CTA (cluster c/4, rank c%4): full tiles nt, first
 *         tile t0, tile stride dt, k-block range [k0, k1), leftover tile lt (-1:
 *         none), its k-block range [lk0, lk1), the cluster's part index, bytes
 *         the CTA receives per split-K tile.
 * DFLOW_ERR_UNSUPPORTED when M or K is outside what the launch covers. */
dflow_status dflow_debug_seq_schedule(int32_t N, int32_t K, int32_t M, int32_t Q, int32_t *plan, int32_t *ctas);

/* Test hook, host only (no GPU needed): the schedule the one-pass tcgen05
 * launch (projections above 128 rows) gives N x K weights over M <= 512 rows on
 * `sms` SMs with `slot_bytes` of split-K partial slots, computed by the functions
 * the launch and the kernel evaluate.
 *   plan   int32 [10]: padded columns, tiles T, k-blocks kb, k-split P, tile
 *          groups Q, leftover tiles Tl, parts per leftover tile ls, grid (CTAs,
 *          P Q), accumulator buffers (1; 2 side by side; 3 sharing columns),
 *          ring stages
 *   items  int32 [grid][1 + 6 max_items], per CTA: its item count, then per item
 *          (in the order it runs them) tile, k-block range [k0, k1), part, parts
 *          (1: whole tile; more: the tile is reduced by that many CTAs, each
 *          finishing 1/parts of the token columns), partial slot index.
 * DFLOW_ERR_UNSUPPORTED when no schedule fits; DFLOW_ERR_CAPACITY when a CTA has
 * more than max_items items. */
dflow_status dflow_debug_wide_schedule(int32_t N, int32_t K, int32_t M, int32_t sms, int64_t slot_bytes,
                                       int32_t *plan, int32_t *items, int32_t max_items);

/* Waits for the recorded events, then fills out[DFLOW_PROF_N]. */
dflow_status dflow_profile_read(dflow_handle *h, dflow_kernel_profile *out);
/* Kernels launched by this handle since creation (always counted). */
dflow_status dflow_launch_count(const dflow_handle *h, uint64_t *count);

#ifdef __cplusplus
}
#endif
#endif /* DFLOW_H */
