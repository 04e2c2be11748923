// C ABI of the DFlow round: argument checks, workspace layout, the order of
// kernel launches for each call, and the small fused kernels of the round
// (embedding gather, norms, rotary/K-V writes, acceptance, carry, relay input).
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <cstdio>
#include <new>
#include <vector>

#include "dflow_internal.cuh"
#include "gemm_tc.cuh"
#include "sample.cuh"

using namespace dflow;

namespace {

constexpr int PF = 64;  // prompt rows per sequence per prefill step

// ---------------------------------------------------------------------------
// small kernels
// ---------------------------------------------------------------------------

__device__ __forceinline__ float block_sum(float v, float *red) {
  v = warp_sum(v);
  const int w = threadIdx.x / 32, l = threadIdx.x % 32, nw = blockDim.x / 32;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = l < nw ? red[l] : 0.f;
  return warp_sum(t);
}

// rotary table: rope[p][i] = (cos, sin)(p * theta^(-2i/hd)), angles in double
__global__ void k_rope_table(float2 *rope, int max_ctx, int hd, double theta) {
  const int half = hd / 2;
  const long long n = (long long)max_ctx * half;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < n;
       e += (long long)gridDim.x * blockDim.x) {
    const int p = (int)(e / half), i = (int)(e % half);
    const double ang = (double)p * pow(theta, -2.0 * i / hd);
    double sv, cv;
    sincos(ang, &sv, &cv);
    rope[e] = make_float2((float)cv, (float)sv);
  }
}

// device-side checks before a round touches the caches
__global__ void k_guard(const int *tokens, const int *seq_len, const int *n_carry,
                        const int *boundary, const int *active, int batch, int R, int max_ctx,
                        int vocab, int B, int *status) {
  pdl_entry();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch || !active[b]) return;
  const int n = seq_len[b];
  if (n < 1 || n - 1 + R > max_ctx) { set_status(status, DFLOW_ERR_CAPACITY); return; }
  const int anchor = tokens[(size_t)b * max_ctx + n - 1];
  const int nc = n_carry[b];
  if (anchor < 0 || anchor >= vocab || nc < 0 || nc > B - 1) { set_status(status, DFLOW_ERR_BAD_STATE); return; }
  if (nc > 0) {
    const int t0 = boundary[2 * b], t1 = boundary[2 * b + 1];
    if (t0 < 0 || t0 >= vocab || t1 < 0 || t1 >= vocab) set_status(status, DFLOW_ERR_BAD_STATE);
  }
}

// the state checks of k_guard, folded into k_rows_round
struct GuardArgs {
  const int *tokens = nullptr, *n_carry = nullptr, *boundary = nullptr;
  int max_ctx = 0, vocab = 0, B = 0;
  int *status = nullptr;  // null: no checks
};

// rows of a round: row b*R+i at position n_b-1+i; writes allowed for active
// sequences.  With gd.status set, row 0 of each sequence also runs k_guard's
// checks (the entry points whose first kernel this is launch no separate guard).
__global__ void k_rows_round(int *pos, int *wr, int *kvlen, const int *seq_len, const int *active, int batch,
                             int R, const int *status, GuardArgs gd) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= batch * R) return;
  const int b = r / R, i = r % R;
  bool ok = active[b] != 0;
  if (gd.status != nullptr && ok) {
    // every row of a sequence whose block would not fit gets no write (the
    // projections that follow place K/V by these positions and do not read the
    // status word); the block's other checks only set the status
    const int n = seq_len[b];
    const bool fits = n >= 1 && n - 1 + R <= gd.max_ctx;
    if (i == 0) {
      if (!fits) {
        set_status(gd.status, DFLOW_ERR_CAPACITY);
      } else {
        const int anchor = gd.tokens[(size_t)b * gd.max_ctx + n - 1];
        const int nc = gd.n_carry[b];
        if (anchor < 0 || anchor >= gd.vocab || nc < 0 || nc > gd.B - 1) {
          set_status(gd.status, DFLOW_ERR_BAD_STATE);
        } else if (nc > 0) {
          const int t0 = gd.boundary[2 * b], t1 = gd.boundary[2 * b + 1];
          if (t0 < 0 || t0 >= gd.vocab || t1 < 0 || t1 >= gd.vocab) set_status(gd.status, DFLOW_ERR_BAD_STATE);
        }
      }
    }
    ok = fits;
  }
  pos[r] = ok ? seq_len[b] - 1 + i : 0;
  wr[r] = ok;
  if (i == 0) kvlen[b] = ok ? seq_len[b] - 1 + R : 1;  // causal keys 0..n-2+R once the block is written
}

// block of a plain decoding step: every row of sequence b holds its last
// committed token (row 0 is the step itself; rows 1..B are computed and dropped)
__global__ void k_decode_block(int *blk, const int *tokens, const int *seq_len, const int *active, int batch, int R,
                               int max_ctx, const int *status) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= batch * R) return;
  const int b = r / R;
  blk[r] = active[b] ? tokens[(size_t)b * max_ctx + seq_len[b] - 1] : 0;
}

// after a plain decoding step: the committed token of each sequence (-1 if
// inactive), and nothing carried into a next draft block
__global__ void k_decode_finish(const int *acc, const int *comm, int R, int *token_out, int *n_carry, int *boundary,
                                int batch, const int *status) {
  pdl_entry();
  if (*status) return;
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  token_out[b] = acc[b] < 0 ? -1 : comm[(size_t)b * R];
  if (acc[b] < 0) return;
  n_carry[b] = 0;
  boundary[2 * b] = -1;
  boundary[2 * b + 1] = -1;
}

// rows of prefill step c: row b*PF+i at position c0+i if inside the prompt
__global__ void k_rows_prefill(int *pos, int *wr, int *kvlen, const int *plen, int batch, int c0,
                               const int *status) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= batch * PF) return;
  const int b = r / PF, p = c0 + r % PF;
  const bool ok = p < plen[b];
  pos[r] = ok ? p : 0;
  wr[r] = ok;
  if (r % PF == 0) kvlen[b] = plen[b] > c0 ? min(c0 + PF, plen[b]) : 1;
}

// residual-stream row finished by a small kernel: bf16(x * gain) for the next
// projection and the squared-norm partial of every 128-feature block
template <typename T>
__device__ __forceinline__ void norm_outputs(const float *xr, int r, int d, T *xn, const float *gain, float *ss,
                                             int ld_ss) {
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32, nw = blockDim.x / 32;
  for (int fb = warp; fb < d / 128; fb += nw) {
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int c = fb * 128 + lane + 32 * k;
      const float v = xr[c];
      xn[(size_t)r * d + c] = from_f<T>(v * gain[c]);
      acc += v * v;
    }
    acc = warp_sum(acc);
    if (lane == 0) ss[(size_t)fb * ld_ss + r] = acc;
  }
}

// x[r] = E[tok] (fp32 residual stream); tok = toks[b*stride + i].  With xn set,
// also the first layer's normalised input (see norm_outputs).
template <typename T>
__global__ void k_embed(const T *__restrict__ E, const int *__restrict__ toks, int stride, int R,
                        const int *__restrict__ wr, float *__restrict__ x, int d, int vocab, T *__restrict__ xn,
                        const float *__restrict__ gain, float *__restrict__ ss, int ld_ss, int *status) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x, b = r / R, i = r % R;
  int tok = (wr == nullptr || wr[r]) ? toks[(size_t)b * stride + i] : 0;
  if (tok < 0 || tok >= vocab) {
    if (threadIdx.x == 0) set_status(status, DFLOW_ERR_BAD_STATE);
    tok = 0;
  }
  for (int c = threadIdx.x; c < d; c += blockDim.x) x[(size_t)r * d + c] = to_f(E[(size_t)tok * d + c]);
  if (xn != nullptr) {
    __syncthreads();
    norm_outputs<T>(x + (size_t)r * d, r, d, xn, gain, ss, ld_ss);
  }
}

// y[r] = x[r] / rms(x[r]) * w   (fp32 in, model dtype out)
template <typename T>
__global__ void k_rmsnorm(const float *__restrict__ x, int ldx, const float *__restrict__ w,
                          T *__restrict__ y, int ldy, int d, float eps, const int *status) {
  pdl_entry();
  if (*status) return;
  __shared__ float red[32];
  const float *xr = x + (size_t)blockIdx.x * ldx;
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) ss += xr[c] * xr[c];
  ss = block_sum(ss, red);
  const float inv = rsqrtf(ss / d + eps);
  for (int c = threadIdx.x; c < d; c += blockDim.x)
    y[(size_t)blockIdx.x * ldy + c] = from_f<T>(xr[c] * inv * w[c]);
}

// per (row, head): q/k RMSNorm over hd, rotary at pos[r], then write q to
// q_out, k/v either into a paged pool at pos[r] (when wr[r]) or into block
// buffers.  The source buffer holds nq query heads, then hkv key heads, then
// hkv value heads.
template <typename T, int HD>
__global__ void __launch_bounds__(128)
k_qkv_post(Dims D, const float *__restrict__ src, int ld, int nq, const float *__restrict__ qn,
           const float *__restrict__ kn, const float2 *__restrict__ rope,
           const int *__restrict__ pos, const int *__restrict__ wr, int R, T *__restrict__ q_out,
           T *__restrict__ pool, const int *__restrict__ page_table, T *__restrict__ bk,
           T *__restrict__ bv, const int *status) {
  pdl_entry();
  if (*status) return;
  constexpr int J = HD / 32, H2 = HD / 64;
  const int r = blockIdx.x, lane = threadIdx.x % 32;
  const int head = blockIdx.y * 4 + threadIdx.x / 32;
  if (head >= nq + 2 * D.hkv) return;
  const float *s = src + (size_t)r * ld + (size_t)head * HD;
  float v[J];
#pragma unroll
  for (int j = 0; j < J; ++j) v[j] = s[lane + 32 * j];
  const bool is_q = head < nq, is_k = !is_q && head < nq + D.hkv;
  if (is_q || is_k) {
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < J; ++j) ss += v[j] * v[j];
    ss = warp_sum(ss);
    const float inv = rsqrtf(ss / HD + D.rms_eps);
    const float *g = is_q ? qn : kn;
#pragma unroll
    for (int j = 0; j < J; ++j) v[j] *= inv * g[lane + 32 * j];
    const float2 *cs = rope + (size_t)pos[r] * (HD / 2);
#pragma unroll
    for (int j = 0; j < H2; ++j) {
      const float2 t = cs[lane + 32 * j];
      const float x1 = v[j], x2 = v[j + H2];
      v[j] = x1 * t.x - x2 * t.y;
      v[j + H2] = x2 * t.x + x1 * t.y;
    }
  }
  T *dst;
  if (is_q) {
    dst = q_out + ((size_t)r * nq + head) * HD;
  } else {
    const int kvh = is_k ? head - nq : head - nq - D.hkv;
    if (bk != nullptr) {
      dst = (is_k ? bk : bv) + ((size_t)r * D.hkv + kvh) * HD;
    } else {
      if (!wr[r]) return;
      const int b = r / R, p = pos[r];
      const int page = page_table[(size_t)b * D.pages_per_seq + p / D.page_size];
      dst = pool + pool_off(D, page, is_k ? 0 : 1, kvh, p % D.page_size);
    }
  }
#pragma unroll
  for (int j = 0; j < J; ++j) dst[lane + 32 * j] = from_f<T>(v[j]);
}

// stash[r][f*d + c] = x[r][c]: residual stream after a feature layer (Eq. 1 input)
template <typename T>
__global__ void k_stash(const float *__restrict__ x, T *__restrict__ stash, int d, int m, int f,
                        const int *status) {
  pdl_entry();
  if (*status) return;
  const size_t r = blockIdx.x;
  for (int c = threadIdx.x; c < d; c += blockDim.x) stash[r * m * d + (size_t)f * d + c] = from_f<T>(x[r * d + c]);
}

// g[r] = argmax over the per-tile partials (ties: lowest token id)
// the drafter's block tokens written straight from the argmax: row 0 of each
// sequence is its anchor, rows 1..R-1 the predictions
struct BlockOut {
  int *blk = nullptr;
  const int *tokens = nullptr, *seq_len = nullptr;
  int max_ctx = 0, R = 1;
};

__global__ void k_argmax_reduce(const float *__restrict__ pv, const int *__restrict__ pi, int n_tiles,
                                int rows, int *__restrict__ g, const int *status, BlockOut bo) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32, lane = threadIdx.x % 32;
  if (r >= rows) return;
  float v = -INFINITY;
  int idx = 0x7fffffff;
  for (int t = lane; t < n_tiles; t += 32) argmax_merge(v, idx, pv[(size_t)r * n_tiles + t], pi[(size_t)r * n_tiles + t]);
  warp_argmax(v, idx);
  if (lane == 0) {
    g[r] = idx;
    if (bo.blk != nullptr) {
      const int b = r / bo.R, i = r % bo.R;
      bo.blk[r] = i == 0 ? bo.tokens[(size_t)b * bo.max_ctx + bo.seq_len[b] - 1] : idx;
    }
  }
}

// relay MLP input (Eq. 4): u = [E(b); E(y_{a+1}); h_j] for each of the B slots
template <typename T>
__global__ void k_relay_u(const T *__restrict__ E, const int *__restrict__ boundary,
                          const T *__restrict__ carry, T *__restrict__ u, int d, int B, int vocab,
                          const int *status) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x, b = r / B, s = r % B;
  int t0 = boundary[2 * b], t1 = boundary[2 * b + 1];
  t0 = (t0 < 0 || t0 >= vocab) ? 0 : t0;
  t1 = (t1 < 0 || t1 >= vocab) ? 0 : t1;
  T *ur = u + (size_t)r * 3 * d;
  const T *h = carry + ((size_t)b * B + s) * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    ur[c] = E[(size_t)t0 * d + c];
    ur[d + c] = E[(size_t)t1 * d + c];
    ur[2 * d + c] = h[c];
  }
}

// Eq. 5 for one carried slot j of sequence b
template <typename T>
__device__ void draft_relay_row(const T *__restrict__ E, const float *__restrict__ e_mask, const T *__restrict__ carry,
                                const float *__restrict__ bg, const float *__restrict__ ln_w,
                                const float *__restrict__ ln_b, float ln_eps, float *__restrict__ xr, int d, int B,
                                int b, int j, float *red) {
  (void)E;
  const T *h = carry + ((size_t)b * B + j - 1) * d;
  float s1 = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) s1 += to_f(h[c]);
  const float mu = block_sum(s1, red) / d;
  float s2 = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float t = to_f(h[c]) - mu;
    s2 += t * t;
  }
  const float inv = rsqrtf(block_sum(s2, red) / d + ln_eps);
  const float *beta = bg + ((size_t)b * B + j - 1) * 2 * d, *gamma = beta + d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float ln = (to_f(h[c]) - mu) * inv * ln_w[c] + ln_b[c];
    xr[c] = e_mask[c] + beta[c] * ln + gamma[c];
  }
}

// drafter inputs (Eq. 5): row 0 = E(anchor); slot j <= n_carry:
// E_mask + beta * LN(h_j) + gamma; other slots E_mask
template <typename T>
__global__ void k_draft_input(const T *__restrict__ E, const float *__restrict__ e_mask,
                              const int *__restrict__ tokens, const int *__restrict__ seq_len,
                              int max_ctx, const T *__restrict__ carry, const int *__restrict__ n_carry,
                              const float *__restrict__ bg, const float *__restrict__ ln_w,
                              const float *__restrict__ ln_b, float ln_eps, int relay,
                              float *__restrict__ x, int d, int B, T *__restrict__ xn,
                              const float *__restrict__ gain, float *__restrict__ ss, int ld_ss,
                              const int *status) {
  pdl_entry();
  if (*status) return;
  __shared__ float red[32];
  const int R = B + 1, r = blockIdx.x, b = r / R, j = r % R;
  float *xr = x + (size_t)r * d;
  if (j == 0) {
    const int tok = tokens[(size_t)b * max_ctx + seq_len[b] - 1];
    for (int c = threadIdx.x; c < d; c += blockDim.x) xr[c] = to_f(E[(size_t)tok * d + c]);
  } else if (!relay || j > n_carry[b]) {
    for (int c = threadIdx.x; c < d; c += blockDim.x) xr[c] = e_mask[c];
  } else {
    draft_relay_row(E, e_mask, carry, bg, ln_w, ln_b, ln_eps, xr, d, B, b, j, red);
  }
  if (xn != nullptr) {
    __syncthreads();
    norm_outputs<T>(xr, r, d, xn, gain, ss, ld_ss);
  }
}

// Eq. 3: a, bonus, commit (one thread per sequence)
// pos2 / wr2 (optional): the positions of the rows that join the drafter context
// (what k_carry_rows computes from acc), filled here inside a round
__global__ void k_accept(const int *__restrict__ blk, const int *__restrict__ g,
                         const int *__restrict__ forced, int *__restrict__ tokens,
                         int *__restrict__ seq_len, const int *__restrict__ active, int batch, int B,
                         int max_ctx, int *__restrict__ acc, int *__restrict__ comm, int *status,
                         int *__restrict__ pos2 = nullptr, int *__restrict__ wr2 = nullptr) {
  pdl_entry();
  if (*status) return;
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  const int R = B + 1;
  const int *bb = blk + (size_t)b * R, *gb = g + (size_t)b * R;
  int *cb = comm + (size_t)b * R;
  if (!active[b]) {
    acc[b] = -1;
    for (int i = 0; i < R; ++i) cb[i] = -1;
    if (pos2 != nullptr)
      for (int i = 0; i < R; ++i) {
        pos2[(size_t)b * R + i] = 0;
        wr2[(size_t)b * R + i] = 0;
      }
    return;
  }
  int a = 0;
  while (a < B && bb[a + 1] == gb[a]) ++a;
  if (forced != nullptr) {
    const int f = forced[b];
    if (f < 0 || f > B) { set_status(status, DFLOW_ERR_BAD_STATE); return; }
    a = f;
  }
  const int n = seq_len[b];
  if (n + a + 1 > max_ctx) { set_status(status, DFLOW_ERR_CAPACITY); return; }
  for (int i = 0; i < R; ++i) {
    const int t = i < a ? bb[i + 1] : (i == a ? gb[a] : -1);
    cb[i] = t;
    if (i <= a) tokens[(size_t)b * max_ctx + n + i] = t;
  }
  seq_len[b] = n + a + 1;
  acc[b] = a;
  if (pos2 != nullptr)  // rows 0..a at positions n-1..n-1+a join the drafter context
    for (int i = 0; i < R; ++i) {
      pos2[(size_t)b * R + i] = i <= a ? n - 1 + i : 0;
      wr2[(size_t)b * R + i] = i <= a ? 1 : 0;
    }
}

// positions of the rows that join the drafter context after a commit
__global__ void k_carry_rows(const int *__restrict__ acc, const int *__restrict__ seq_len, int batch,
                             int R, int *__restrict__ pos, int *__restrict__ wr, const int *status) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= batch * R) return;
  const int b = r / R, i = r % R, a = acc[b];
  const bool ok = a >= 0 && i <= a;
  pos[r] = ok ? seq_len[b] - a - 2 + i : 0;
  wr[r] = ok;
}

// Sec. 4.2 alignment: slot j = s+1 <- feature row a+j, for j <= B-a-1
template <typename T>
__global__ void k_carry(const T *__restrict__ feats, const int *__restrict__ acc,
                        const int *__restrict__ blk, const int *__restrict__ tokens,
                        const int *__restrict__ seq_len, int max_ctx, T *__restrict__ carry,
                        int *__restrict__ n_carry, int *__restrict__ boundary, int d, int B,
                        int relay, const int *status) {
  pdl_entry();
  if (*status) return;
  const int b = blockIdx.x, s = blockIdx.y, R = B + 1, a = acc[b];
  if (a < 0) return;
  const int nc = relay ? max(0, B - a - 1) : 0;
  if (s == 0 && threadIdx.x == 0) {
    n_carry[b] = nc;
    boundary[2 * b] = tokens[(size_t)b * max_ctx + seq_len[b] - 1];
    boundary[2 * b + 1] = a < B ? blk[(size_t)b * R + a + 1] : -1;
  }
  if (s >= nc) return;
  const T *src = feats + ((size_t)b * R + a + 1 + s) * d;
  T *dst = carry + ((size_t)b * B + s) * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) dst[c] = src[c];
}

// prefill bookkeeping for step c: commit prompt tokens, anchor = argmax at len-1
__global__ void k_prefill_commit(const int *__restrict__ prompt, int stride,
                                 const int *__restrict__ plen, const int *__restrict__ pos,
                                 const int *__restrict__ wr, const int *__restrict__ g, int batch,
                                 int max_ctx, int *__restrict__ tokens, int *__restrict__ seq_len,
                                 int *__restrict__ n_carry, int *__restrict__ boundary,
                                 const int *status) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= batch * PF || !wr[r]) return;
  const int b = r / PF, p = pos[r], len = plen[b];
  tokens[(size_t)b * max_ctx + p] = prompt[(size_t)b * stride + p];
  if (p == len - 1) {
    tokens[(size_t)b * max_ctx + len] = g[r];
    seq_len[b] = len + 1;
    n_carry[b] = 0;
    boundary[2 * b] = -1;
    boundary[2 * b + 1] = -1;
  }
}

// ---------------------------------------------------------------------------
// host helpers
// ---------------------------------------------------------------------------

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

struct dflow_handle {
  dflow_config cfg;
  dflow_weights w;
  std::vector<dflow_layer_weights> tl, dl;
  Dims D;
  int dtype, esz, R, rows_round, rows_max, vocab_tiles, sm_count, gld;
  int attn_split_round, attn_split_pf;
  size_t attn_entries;
  bool use_tc;
  bool fused;  // tensor-core GEMMs with folded norms and the fused Q/K/V epilogue
  size_t ws_need = 0, ws_bytes = 0;
  char *ws = nullptr;
  // workspace views
  float *x, *gf32, *apart, *am_val, *ss;
  float2 *rope;
  void *xn, *q, *bk, *bv, *ao, *mlp, *stash, *feats, *relay_u, *relay_h;
  int *pos, *wr, *pos2, *wr2, *am_idx, *blk, *g, *gd, *acc, *comm, *plen, *kvlen, *zeros;
  float *qlog, *plog;  // T = 1 round: drafter and target logits [rows_round][vocab]
  SampWs samp;
  TcWorkspace tcw;
  DepChain dep;  // completion counters between consecutive tensor-core launches
  // measurement
  uint64_t n_launch = 0;
  bool prof = false;
  struct ProfRec { cudaEvent_t e0, e1; int kind; double bytes, flops; };
  std::vector<ProfRec> prof_recs;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_next = 0;
};

namespace {

// a failed CUDA call; with DFLOW_DEBUG set, the call and the error go to stderr
dflow_status cuda_failed(const char *what, cudaError_t e) {
  static const bool dbg = getenv("DFLOW_DEBUG") != nullptr;
  if (dbg) fprintf(stderr, "dflow: %s: %s\n", what, cudaGetErrorString(e));
  return DFLOW_ERR_CUDA;
}
#define CK(expr)                                           \
  do {                                                     \
    cudaError_t e_ = (expr);                               \
    if (e_ != cudaSuccess) return cuda_failed(#expr, e_);  \
  } while (0)

// a launch outside the counting chain: the next counting launch waits for its grid
#define KL(...)          \
  do {                   \
    __VA_ARGS__;         \
    ++k.h->n_launch;     \
    k.h->dep.brk();      \
  } while (0)

struct Call {
  dflow_handle *h;
  const int *status;
  int *status_w;
  cudaStream_t s;
};

size_t layout(dflow_handle *h, char *base) {
  const dflow_config &c = h->cfg;
  const Dims &D = h->D;
  size_t off = 0;
  auto take = [&](size_t bytes) -> char * {
    char *p = base ? base + off : nullptr;
    off += align256(bytes);
    return p;
  };
  const size_t rm = h->rows_max, es = h->esz;
  const int qd = D.hq * D.hd, kvd = D.hkv * D.hd;
  h->x = (float *)take(rm * D.d * 4);
  h->ss = (float *)take(rm * (D.d / 128) * 4);
  h->gf32 = (float *)take(rm * h->gld * 4);
  h->xn = take(rm * D.d * es);
  h->q = take(rm * qd * es);
  h->bk = take(rm * kvd * es);
  h->bv = take(rm * kvd * es);
  h->ao = take(rm * qd * es);
  h->mlp = take(rm * D.inter * es);
  h->stash = take(rm * (size_t)D.n_feat * D.d * es);
  h->feats = take(rm * D.d * es);
  h->relay_u = take((size_t)c.max_batch * D.B * 3 * D.d * es);
  h->relay_h = take((size_t)c.max_batch * D.B * D.d * es);
  h->apart = (float *)take(h->attn_entries * (D.hd + 2) * 4);
  h->am_val = (float *)take(rm * h->vocab_tiles * 4);
  h->am_idx = (int *)take(rm * h->vocab_tiles * 4);
  h->pos = (int *)take(rm * 4);
  h->wr = (int *)take(rm * 4);
  h->pos2 = (int *)take(rm * 4);
  h->wr2 = (int *)take(rm * 4);
  h->blk = (int *)take(rm * 4);
  h->g = (int *)take(rm * 4);
  h->gd = (int *)take(rm * 4);
  h->acc = (int *)take((size_t)c.max_batch * 4);
  h->comm = (int *)take(rm * 4);
  h->plen = (int *)take((size_t)c.max_batch * 4);
  h->kvlen = (int *)take((size_t)c.max_batch * 4);
  h->zeros = (int *)take((size_t)c.max_batch * 4);
  const size_t rr = h->rows_round;
  h->qlog = (float *)take(rr * D.vocab * 4);
  h->plog = (float *)take(rr * D.vocab * 4);
  h->samp.nch = samp_chunks(D.vocab);
  h->samp.part = (float2 *)take(rr * h->samp.nch * 8);
  h->samp.gv = (float *)take(rr * h->samp.nch * 4);
  h->samp.gi = (int *)take(rr * h->samp.nch * 4);
  h->samp.lse_q = (float *)take(rr * 4);
  h->samp.lse_p = (float *)take(rr * 4);
  h->samp.a = (int *)take((size_t)c.max_batch * 4);
  h->rope = (float2 *)take((size_t)c.max_ctx * (D.hd / 2) * 8);
  h->dep.dev = (unsigned int *)take(kDepSlots * sizeof(unsigned int));
  const int max_n = std::max(std::max(D.vocab, 2 * D.inter), std::max(h->gld, D.d));
  tc_layout(h->tcw, base, off, h->sm_count, rm, (max_n + 127) / 128);
  return off;
}

int pick_splits(const dflow_handle *h, int batch, int rows) {
  int want = (2 * h->sm_count + h->D.hkv * batch - 1) / (h->D.hkv * batch);
  const int cap = (int)(h->attn_entries / ((size_t)rows * h->D.hq));
  return std::max(1, std::min(std::min(want, cap), 64));
}

cudaEvent_t prof_event(dflow_handle *h) {
  if (h->ev_next == h->ev_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    h->ev_pool.push_back(e);
  }
  return h->ev_pool[h->ev_next++];
}

// brackets one launch of class `kind` with events when profiling is on
struct ProfScope {
  dflow_handle *h;
  cudaStream_t s;
  cudaEvent_t e0 = nullptr;
  int kind;
  double bytes, flops;
  ProfScope(dflow_handle *h_, cudaStream_t s_, int kind_, double bytes_, double flops_)
      : h(h_), s(s_), kind(kind_), bytes(bytes_), flops(flops_) {
    if (h->prof && (e0 = prof_event(h))) cudaEventRecord(e0, s);
  }
  ~ProfScope() {
    if (!e0) return;
    cudaEvent_t e1 = prof_event(h);
    if (!e1) return;
    cudaEventRecord(e1, s);
    h->prof_recs.push_back({e0, e1, kind, bytes, flops});
  }
};

double ep_out_bytes(const EpArgs &ep, int M, int N, int esz) {
  switch (ep.mode) {
    case EP_STORE_F32: return 4.0 * M * N;
    case EP_RESID: return 8.0 * M * N;
    case EP_SWIGLU: return (double)esz * M * N / 2;
    case EP_SILU: return (double)esz * M * N;
    case EP_ARGMAX: return 8.0 * M * ((N + 127) / 128);
  }
  return 0.0;
}

cudaError_t gemm(const Call &k, const void *W, int N, int K, const void *X, int M, int ldx,
                 const EpArgs &ep) {
  dflow_handle *h = k.h;
  const double es = h->esz;
  ProfScope ps(h, k.s, DFLOW_PROF_GEMM, es * N * K + es * M * K + ep_out_bytes(ep, M, N, h->esz), 2.0 * M * N * K);
  ++h->n_launch;
  if (!h->use_tc) {  // the fp32 parity model
    h->dep.brk();
    return gemm_simt(h->dtype, W, N, K, X, M, ldx, ep, k.status, k.s);
  }
  // few rows: the persistent kernel, one GEMM (all clusters, balanced tiles)
  const bool seq_mode = ep.mode == EP_STORE_F32 || ep.mode == EP_RESID || ep.mode == EP_SWIGLU ||
                        ep.mode == EP_QKV || ep.mode == EP_SILU;
  if (seq_mode && h->dep.dev != nullptr && K % 64 == 0 && K / 64 >= 4 && ldx % 8 == 0 && seq_supported(M)) {
    const SeqSpec sp{W, N, K, X, ldx, ep};
    return gemm_seq(h->tcw, 1, &sp, M, k.status_w, k.s, &h->dep);
  }
  if (!tc_supports(N, K, M, ldx, ep)) return cudaErrorInvalidValue;
  // more rows than the persistent launch takes: one pass over the weights for up
  // to 512 rows where its schedule suits the shape, else 128-row tiles
  if (M > 128 && gemm_wide_suits(h->tcw, N, K, M))
    return gemm_wide(h->tcw, W, N, K, X, M, ldx, ep, k.status_w, k.s, &h->dep);
  return gemm_tc(h->tcw, W, N, K, X, M, ldx, ep, k.status_w, k.s, true, &h->dep);
}

EpArgs ep_f32(float *out, int ldo, int mode = EP_STORE_F32) {
  EpArgs e{};
  e.mode = mode;
  e.out_f32 = out;
  e.ldo = ldo;
  return e;
}
EpArgs ep_t(int mode, void *out, int ldt) {
  EpArgs e{};
  e.mode = mode;
  e.out_t = out;
  e.ldt = ldt;
  return e;
}

template <typename T>
cudaError_t rmsnorm(const Call &k, const float *x, int ldx, const float *w, void *y, int ldy, int rows) {
  const Dims &D = k.h->D;
  KL(klaunch(k_rmsnorm<T>, rows, 256, 0, k.s, x, ldx, w, static_cast<T *>(y), ldy, D.d, D.rms_eps, k.status));
  return cudaGetLastError();
}

template <typename T>
cudaError_t qkv_post(const Call &k, const Dims &D, int rows, const float *src, int ld, int nq,
                     const float *qn, const float *kn, const int *pos, const int *wr, void *q_out,
                     void *pool, const int *pt, void *bk, void *bv) {
  const int heads = nq + 2 * D.hkv;
  dim3 grid(rows, (heads + 3) / 4);
  if (D.hd == 128)
    KL(klaunch(k_qkv_post<T, 128>, grid, 128, 0, k.s, D, src, ld, nq, qn, kn, k.h->rope, pos, wr, D.R,
                                               (T *)q_out, (T *)pool, pt, (T *)bk, (T *)bv, k.status));
  else
    KL(klaunch(k_qkv_post<T, 64>, grid, 128, 0, k.s, D, src, ld, nq, qn, kn, k.h->rope, pos, wr, D.R,
                                              (T *)q_out, (T *)pool, pt, (T *)bk, (T *)bv, k.status));
  return cudaGetLastError();
}

// One Qwen3 decoder layer over `rows` rows held in h->x (fp32 residual).
//   causal = 1: target layer; K/V written to the paged pool (rows with wr),
//               attention over positions 0..pos.
//   causal = 0: drafter layer; block K/V kept in bk/bv, attention over the
//               drafter context pool (0..n-2) and the block rows.
// the input RMSNorm of a projection, folded into its epilogue (fused path)
EpArgs in_norm(EpArgs e, const dflow_handle *h) {
  e.in_ss = h->ss;
  e.in_ss_n = h->D.d / 128;
  e.ld_ss = h->rows_max;
  e.in_inv_d = 1.0f / h->D.d;
  e.in_eps = h->D.rms_eps;
  return e;
}

// residual add that also leaves bf16(x * next_gain), the squared-norm
// partials of x and (optionally) the Eq. 1 stash copy of x
EpArgs resid_norm(const dflow_handle *h, const float *next_gain, void *stash) {
  EpArgs e = ep_f32(h->x, h->D.d, EP_RESID);
  e.out_ss = h->ss;
  e.ld_ss = h->rows_max;
  e.out_xn = h->xn;
  e.ld_xn = h->D.d;
  e.out_gain = next_gain;
  e.out_stash = stash;
  e.ld_stash = h->D.n_feat * h->D.d;
  return e;
}

// fused Q/K/V epilogue targets: q to h->q, k/v to the paged pool (pool set) or
// to the block buffers (pool null)
EpArgs qkv_ep(const dflow_handle *h, const Dims &D, int nq, const float *qn, const float *kn, const int *pos,
              const int *wr, void *pool, const int *page_table, bool block) {
  EpArgs e{};
  e.mode = EP_QKV;
  QkvOut &o = e.qkv;
  o.nq = nq;
  o.hkv = D.hkv;
  o.hq_row = D.hq;
  o.eps = D.rms_eps;
  o.qn = qn;
  o.kn = kn;
  o.rope = h->rope;
  o.pos = pos;
  o.wr = wr;
  o.R = D.R;
  o.q_out = h->q;
  o.pool = pool;
  o.page_table = page_table;
  o.pages_per_seq = D.pages_per_seq;
  o.page_size = D.page_size;
  o.num_pages = D.num_pages;
  o.bk = block ? h->bk : nullptr;
  o.bv = block ? h->bv : nullptr;
  return e;
}

// attention of one layer: q (h->q) against the layer's pool (and, drafter, the
// block's own K/V) into h->ao
AttnArgs layer_attn_args(const dflow_handle *h, void *pool_layer, const dflow_state *st, int causal, int splits) {
  AttnArgs a{};
  a.q = h->q;
  a.pool = pool_layer;
  a.page_table = st->page_table;
  a.bk = causal ? nullptr : h->bk;
  a.bv = causal ? nullptr : h->bv;
  a.pos = h->pos;
  a.seq_len = st->seq_len;
  a.kvlen = h->kvlen;
  a.causal = causal;
  a.n_splits = splits;
  a.part = h->apart;
  a.out = h->ao;
  return a;
}

cudaError_t layer_attention(const Call &k, const Dims &D, int batch, void *pool_layer, const dflow_state *st,
                            int causal, int splits) {
  dflow_handle *h = k.h;
  const int rows = batch * D.R;
  AttnArgs a{};
  a.q = h->q;
  a.pool = pool_layer;
  a.page_table = st->page_table;
  a.bk = causal ? nullptr : h->bk;
  a.bv = causal ? nullptr : h->bv;
  a.pos = h->pos;
  a.seq_len = st->seq_len;
  a.kvlen = h->kvlen;
  a.causal = causal;
  a.n_splits = splits;
  a.part = h->apart;
  a.out = h->ao;
  ProfScope ps(h, k.s, DFLOW_PROF_ATTN, 0.0, 4.0 * rows * D.hq * D.hd);
  h->n_launch += 1;
  return attention(h->dtype, D, batch, a, k.status_w, k.s, &h->dep);
}

// One Qwen3 decoder layer over `rows` rows held in h->x (fp32 residual).
//   causal = 1: target layer; K/V written to the paged pool (rows with wr),
//               attention over positions 0..pos.
//   causal = 0: drafter layer; block K/V kept in bk/bv, attention over the
//               drafter context pool (0..n-2) and the block rows.
// Fused path (tensor-core GEMMs, 128-dim heads): h->xn / h->ss already hold
// bf16(x * attn_norm) and the squared norms of x; the layer leaves
// bf16(x * next_gain) and the new norms for whatever projection comes next.
template <typename T>
cudaError_t layer_forward(const Call &k, const Dims &D, int batch, const dflow_layer_weights &L,
                          void *pool_layer, const dflow_state *st, int causal, int splits, const float *next_gain,
                          void *stash) {
  dflow_handle *h = k.h;
  const int rows = batch * D.R, qkv_dim = (D.hq + 2 * D.hkv) * D.hd, qd = D.hq * D.hd;
  cudaError_t e;
  if (h->fused) {
    EpArgs eq = in_norm(qkv_ep(h, D, D.hq, L.q_norm, L.k_norm, h->pos, h->wr, causal ? pool_layer : nullptr,
                               st->page_table, !causal),
                        h);
    if ((e = gemm(k, L.w_qkv, qkv_dim, D.d, h->xn, rows, D.d, eq))) return e;
  } else {
    if ((e = rmsnorm<T>(k, h->x, D.d, L.attn_norm, h->xn, D.d, rows))) return e;
    if ((e = gemm(k, L.w_qkv, qkv_dim, D.d, h->xn, rows, D.d, ep_f32(h->gf32, h->gld)))) return e;
    if ((e = qkv_post<T>(k, D, rows, h->gf32, h->gld, D.hq, L.q_norm, L.k_norm, h->pos, h->wr, h->q,
                         causal ? pool_layer : nullptr, st->page_table, causal ? nullptr : h->bk,
                         causal ? nullptr : h->bv)))
      return e;
  }
  if ((e = layer_attention(k, D, batch, pool_layer, st, causal, splits))) return e;
  if (h->fused) {
    if ((e = gemm(k, L.w_o, D.d, qd, h->ao, rows, qd, resid_norm(h, L.mlp_norm, nullptr)))) return e;
    if ((e = gemm(k, L.w_gate_up, 2 * D.inter, D.d, h->xn, rows, D.d, in_norm(ep_t(EP_SWIGLU, h->mlp, D.inter), h))))
      return e;
    return gemm(k, L.w_down, D.d, D.inter, h->mlp, rows, D.inter, resid_norm(h, next_gain, stash));
  }
  if ((e = gemm(k, L.w_o, D.d, qd, h->ao, rows, qd, ep_f32(h->x, D.d, EP_RESID)))) return e;
  if ((e = rmsnorm<T>(k, h->x, D.d, L.mlp_norm, h->xn, D.d, rows))) return e;
  if ((e = gemm(k, L.w_gate_up, 2 * D.inter, D.d, h->xn, rows, D.d, ep_t(EP_SWIGLU, h->mlp, D.inter)))) return e;
  if ((e = gemm(k, L.w_down, D.d, D.inter, h->mlp, rows, D.inter, ep_f32(h->x, D.d, EP_RESID)))) return e;
  if (stash) {
    KL(klaunch(k_stash<T>, rows, 256, 0, k.s, h->x, (T *)h->stash, D.d, D.n_feat,
               (int)(((T *)stash - (T *)h->stash) / D.d), k.status));
    return cudaGetLastError();
  }
  return cudaSuccess;
}

// final RMSNorm -> LM head -> greedy token per row (g non-null) and fp32 logits
// (logits non-null): one pass over the LM head per output asked for
template <typename T>
cudaError_t lm_head_argmax(const Call &k, const Dims &D, int rows, const float *norm, int *g,
                           float *logits, BlockOut bo = BlockOut{}) {
  dflow_handle *h = k.h;
  cudaError_t e;
  if (!h->fused && (e = rmsnorm<T>(k, h->x, D.d, norm, h->xn, D.d, rows))) return e;
  EpArgs ep{};
  ep.mode = EP_ARGMAX;
  ep.part_val = h->am_val;
  ep.part_idx = h->am_idx;
  ep.n_tiles = h->vocab_tiles;
  if (h->fused) ep = in_norm(ep, h);
  if (g) {
    if ((e = gemm(k, h->w.lm_head, D.vocab, D.d, h->xn, rows, D.d, ep))) return e;
    KL(klaunch(k_argmax_reduce, (rows + 7) / 8, 256, 0, k.s, h->am_val, h->am_idx, h->vocab_tiles, rows, g,
               k.status, bo));
    if ((e = cudaGetLastError())) return e;
  }
  if (logits) {
    EpArgs el = ep_f32(logits, D.vocab);
    if (h->fused) el = in_norm(el, h);
    return gemm(k, h->w.lm_head, D.vocab, D.d, h->xn, rows, D.d, el);
  }
  return cudaSuccess;
}

// feature slot of target layer l+1 in the Eq. 1 stash, or null
template <typename T>
void *stash_slot(const dflow_handle *h, int l) {
  for (int fi = 0; fi < h->D.n_feat; ++fi)
    if (h->cfg.feat_layers[fi] == l + 1) return static_cast<T *>(h->stash) + (size_t)fi * h->D.d;
  return nullptr;
}

// The decoder layers [0, nL) of one stack (target: causal, K/V to its pool and
// the Eq. 1 stash; drafter: block K/V) over the rows in h->x.  On the fused
// tensor-core path with few rows the first QKV projection runs alone, then each
// layer is its attention plus one persistent launch of its O, gate/up and down
// projections and the next layer's QKV; otherwise (or with
// DFLOW_SEPARATE_GEMMS set) layer by layer, one launch per projection.
template <typename T>
cudaError_t stack_forward(const Call &k, const Dims &D, int batch, const dflow_layer_weights *Ls, int nL,
                          T *pool_base, const dflow_state *st, int causal, int splits, const float *final_gain) {
  dflow_handle *h = k.h;
  const int rows = batch * D.R, qkv_dim = (D.hq + 2 * D.hkv) * D.hd, qd = D.hq * D.hd;
  auto pool = [&](int l) { return pool_base + (size_t)l * pool_layer_elems(D); };
  auto next_gain = [&](int l) { return l + 1 < nL ? Ls[l + 1].attn_norm : final_gain; };
  auto stash = [&](int l) { return causal ? stash_slot<T>(h, l) : nullptr; };
  const bool seq =
      h->fused && h->dep.dev != nullptr && seq_supported(rows) && getenv("DFLOW_SEPARATE_GEMMS") == nullptr;
  cudaError_t e;
  if (!seq) {
    for (int l = 0; l < nL; ++l)
      if ((e = layer_forward<T>(k, D, batch, Ls[l], pool(l), st, causal, splits, next_gain(l), stash(l)))) return e;
    return cudaSuccess;
  }
  auto qkv_args = [&](int l) {
    return in_norm(qkv_ep(h, D, D.hq, Ls[l].q_norm, Ls[l].k_norm, h->pos, h->wr, causal ? (void *)pool(l) : nullptr,
                          st->page_table, !causal),
                   h);
  };
  if ((e = gemm(k, Ls[0].w_qkv, qkv_dim, D.d, h->xn, rows, D.d, qkv_args(0)))) return e;
  // DFLOW_FUSED_ATTENTION: the attention as the first phase of each layer's
  // persistent launch instead of its own launch (same results; at batch 1 the
  // separate launch is faster: its start overlaps the previous launch's tail and
  // it uses twice the key splits, while in the fused launch the attention
  // clusters join the gate/up projection late)
  const bool fuse_attn = seq_attn_supported(D, batch, rows) && getenv("DFLOW_FUSED_ATTENTION") != nullptr;
  for (int l = 0; l < nL; ++l) {
    if (!fuse_attn && (e = layer_attention(k, D, batch, pool(l), st, causal, splits))) return e;
    const dflow_layer_weights &L = Ls[l];
    SeqSpec sp[4];
    int n = 0;
    sp[n++] = SeqSpec{L.w_o, D.d, qd, h->ao, qd, resid_norm(h, L.mlp_norm, nullptr)};
    sp[n++] = SeqSpec{L.w_gate_up, 2 * D.inter, D.d, h->xn, D.d, in_norm(ep_t(EP_SWIGLU, h->mlp, D.inter), h)};
    sp[n++] = SeqSpec{L.w_down, D.d, D.inter, h->mlp, D.inter, resid_norm(h, next_gain(l), stash(l))};
    if (l + 1 < nL) sp[n++] = SeqSpec{Ls[l + 1].w_qkv, qkv_dim, D.d, h->xn, D.d, qkv_args(l + 1)};
    double bytes = 0.0, flops = 0.0;
    for (int j = 0; j < n; ++j) {
      bytes += (double)h->esz * sp[j].N * sp[j].K + (double)h->esz * rows * sp[j].K + ep_out_bytes(sp[j].ep, rows, sp[j].N, h->esz);
      flops += 2.0 * rows * sp[j].N * sp[j].K;
    }
    ProfScope ps(h, k.s, DFLOW_PROF_GEMM, bytes, flops);
    ++h->n_launch;
    if (fuse_attn) {
      const SeqAttnSpec as{D, batch, layer_attn_args(h, pool(l), st, causal, splits)};
      if ((e = gemm_seq(h->tcw, n, sp, rows, k.status_w, k.s, &h->dep, false, &as))) return e;
    } else if ((e = gemm_seq(h->tcw, n, sp, rows, k.status_w, k.s, &h->dep))) {
      return e;
    }
  }
  return cudaSuccess;
}

// target forward over h->x (embeddings) at h->pos; writes K/V, g, Eq. 1 features
template <typename T>
cudaError_t target_forward(const Call &k, const Dims &D, int batch, const dflow_state *st, int *g,
                           void *feats, float *logits, int splits) {
  dflow_handle *h = k.h;
  const int rows = batch * D.R;
  const int L = h->cfg.n_layers;
  cudaError_t e;
  if ((e = stack_forward<T>(k, D, batch, h->tl.data(), L, static_cast<T *>(st->kv), st, 1, splits,
                            h->w.final_norm)))
    return e;
  if ((e = lm_head_argmax<T>(k, D, rows, h->w.final_norm, g, logits))) return e;
  // Eq. 1: H_T = RMSNorm(W_c [H^l1; ...; H^lm])
  if ((e = gemm(k, h->w.w_c, D.d, D.n_feat * D.d, h->stash, rows, D.n_feat * D.d, ep_f32(h->gf32, h->gld)))) return e;
  return rmsnorm<T>(k, h->gf32, h->gld, h->w.c_norm, feats, D.d, rows);
}

// drafter context injection: K/V of feature rows (wr2) at pos2 in every draft layer
template <typename T>
cudaError_t ctx_append(const Call &k, const Dims &D, int rows, const dflow_state *st, const void *feats) {
  dflow_handle *h = k.h;
  cudaError_t e;
  const size_t qoff = (size_t)D.hq * D.hd * D.d;  // K and V rows follow the Q rows of w_qkv
  const int nkv = 2 * D.hkv * D.hd;
  if (h->fused && h->dep.dev != nullptr && seq_supported(rows) && D.d % 64 == 0 && D.d / 64 >= 4) {
    // the draft layers' projections are independent: up to four per persistent launch
    for (int l0 = 0; l0 < h->cfg.draft_layers; l0 += 4) {
      SeqSpec sp[4];
      int n = 0;
      double bytes = 0.0, flops = 0.0;
      for (int l = l0; l < std::min(l0 + 4, h->cfg.draft_layers); ++l) {
        const dflow_layer_weights &L = h->dl[l];
        T *pool_l = static_cast<T *>(st->draft_kv) + (size_t)l * pool_layer_elems(D);
        sp[n++] = SeqSpec{static_cast<const T *>(L.w_qkv) + qoff, nkv, D.d, feats, D.d,
                          qkv_ep(h, D, 0, nullptr, L.k_norm, h->pos2, h->wr2, pool_l, st->page_table, false)};
        bytes += (double)h->esz * nkv * D.d + (double)h->esz * rows * D.d;
        flops += 2.0 * rows * nkv * D.d;
      }
      ProfScope ps(h, k.s, DFLOW_PROF_GEMM, bytes, flops);
      ++h->n_launch;
      if ((e = gemm_seq(h->tcw, n, sp, rows, k.status_w, k.s, &h->dep, true))) return e;
    }
    return cudaSuccess;
  }
  for (int l = 0; l < h->cfg.draft_layers; ++l) {
    const dflow_layer_weights &L = h->dl[l];
    const T *wkv = static_cast<const T *>(L.w_qkv) + qoff;
    T *pool_l = static_cast<T *>(st->draft_kv) + (size_t)l * pool_layer_elems(D);
    if (h->fused) {
      if ((e = gemm(k, wkv, 2 * D.hkv * D.hd, D.d, feats, rows, D.d,
                    qkv_ep(h, D, 0, nullptr, L.k_norm, h->pos2, h->wr2, pool_l, st->page_table, false))))
        return e;
      continue;
    }
    if ((e = gemm(k, wkv, 2 * D.hkv * D.hd, D.d, feats, rows, D.d, ep_f32(h->gf32, h->gld)))) return e;
    if ((e = qkv_post<T>(k, D, rows, h->gf32, h->gld, 0, nullptr, L.k_norm, h->pos2, h->wr2, nullptr,
                         pool_l, st->page_table, nullptr, nullptr)))
      return e;
  }
  return cudaSuccess;
}

// the round's device-side state checks, run by its first kernel (k_rows_round)
GuardArgs guard_args(const Call &k, const dflow_state *st) {
  GuardArgs g;
  g.tokens = st->tokens;
  g.n_carry = st->n_carry;
  g.boundary = st->boundary;
  g.max_ctx = k.h->cfg.max_ctx;
  g.vocab = k.h->D.vocab;
  g.B = k.h->D.B;
  g.status = k.status_w;
  return g;
}

Dims round_dims(const dflow_handle *h) {
  Dims D = h->D;
  D.R = h->R;
  return D;
}

template <typename T>
dflow_status do_draft(const Call &k, dflow_state *st, int *blk, int relay, float *logits = nullptr,
                      const SampRound *sr = nullptr) {
  dflow_handle *h = k.h;
  const Dims D = round_dims(h);
  const int batch = st->batch, rows = batch * D.R, B = D.B;
  KL(klaunch(k_rows_round, (rows + 127) / 128, 128, 0, k.s, h->pos, h->wr, h->kvlen, st->seq_len, st->active, batch,
             D.R, k.status, guard_args(k, st)));
  CK(cudaGetLastError());
  if (relay) {
    // Eq. 4 for every slot of every sequence; Eq. 5 keeps slots j <= n_carry
    KL(klaunch(k_relay_u<T>, batch * B, 256, 0, k.s, (const T *)h->w.embed, st->boundary, (const T *)st->carry,
                                             (T *)h->relay_u, D.d, B, D.vocab, k.status));
    CK(cudaGetLastError());
    const int rr = batch * B;
    if (h->use_tc && h->dep.dev != nullptr && seq_supported(rr) && D.d % 64 == 0) {
      // both relay GEMMs in one persistent launch (the second reads the first's SiLU output)
      const SeqSpec sp[2] = {{h->w.relay_w1, D.d, 3 * D.d, h->relay_u, 3 * D.d, ep_t(EP_SILU, h->relay_h, D.d)},
                             {h->w.relay_w2, 2 * D.d, D.d, h->relay_h, D.d, ep_f32(h->gf32, 2 * D.d)}};
      ProfScope ps(h, k.s, DFLOW_PROF_GEMM,
                   (double)h->esz * (3.0 * D.d * D.d + 2.0 * D.d * D.d) + (double)h->esz * rr * 4.0 * D.d,
                   2.0 * rr * 5.0 * D.d * D.d);
      ++h->n_launch;
      CK(gemm_seq(h->tcw, 2, sp, rr, k.status_w, k.s, &h->dep));
    } else {
      CK(gemm(k, h->w.relay_w1, D.d, 3 * D.d, h->relay_u, rr, 3 * D.d, ep_t(EP_SILU, h->relay_h, D.d)));
      CK(gemm(k, h->w.relay_w2, 2 * D.d, D.d, h->relay_h, rr, D.d, ep_f32(h->gf32, 2 * D.d)));
    }
  }
  KL(klaunch(k_draft_input<T>, rows, 256, 0, k.s, (const T *)h->w.embed, h->w.e_mask, st->tokens, st->seq_len,
                                          h->cfg.max_ctx, (const T *)st->carry, st->n_carry, h->gf32,
                                          h->w.ln_w, h->w.ln_b, D.ln_eps, relay, h->x, D.d, B,
                                          h->fused ? (T *)h->xn : nullptr, h->dl[0].attn_norm, h->ss, h->rows_max,
                                          k.status));
  CK(cudaGetLastError());
  const int splits = pick_splits(h, batch, rows);
  CK(stack_forward<T>(k, D, batch, h->dl.data(), h->cfg.draft_layers, static_cast<T *>(st->draft_kv), st, 0, splits,
                      h->w.draft_final_norm));
  if (sr != nullptr) {
    // T = 1: logits only, then a Gumbel-max sample per block row
    CK(lm_head_argmax<T>(k, D, rows, h->w.draft_final_norm, nullptr, logits));
    int n = 0;
    const cudaError_t e = samp_draft(logits, D.vocab, D.R, batch, *sr, h->samp, st->tokens, st->seq_len, st->active,
                                     h->cfg.max_ctx, blk, k.status, k.s, &n);
    h->n_launch += n;
    h->dep.brk();
    CK(e);
    CK(cudaGetLastError());
    return DFLOW_OK;
  }
  BlockOut bo;
  bo.blk = blk;
  bo.tokens = st->tokens;
  bo.seq_len = st->seq_len;
  bo.max_ctx = h->cfg.max_ctx;
  bo.R = D.R;
  CK(lm_head_argmax<T>(k, D, rows, h->w.draft_final_norm, h->gd, logits, bo));
  return DFLOW_OK;
}

template <typename T>
// rows_ready: the round's drafting already wrote pos / wr / kvlen for these rows
// (seq_len is unchanged in between), so k_rows_round is not run again
dflow_status do_verify(const Call &k, dflow_state *st, const int *blk, int *g, void *feats, float *logits,
                       bool rows_ready = false) {
  dflow_handle *h = k.h;
  const Dims D = round_dims(h);
  const int batch = st->batch, rows = batch * D.R;
  if (!rows_ready) {
    KL(klaunch(k_rows_round, (rows + 127) / 128, 128, 0, k.s, h->pos, h->wr, h->kvlen, st->seq_len, st->active, batch,
               D.R, k.status, guard_args(k, st)));
    CK(cudaGetLastError());
  }
  KL(klaunch(k_embed<T>, rows, 256, 0, k.s, (const T *)h->w.embed, blk, D.R, D.R, (const int *)nullptr, h->x, D.d,
             D.vocab, h->fused ? (T *)h->xn : nullptr, h->tl[0].attn_norm, h->ss, h->rows_max, k.status_w));
  CK(cudaGetLastError());
  CK(target_forward<T>(k, D, batch, st, g, feats, logits, pick_splits(h, batch, rows)));
  return DFLOW_OK;
}

// carry_rows: also write the context rows' positions for the do_carry that follows
dflow_status do_accept(const Call &k, dflow_state *st, const int *blk, const int *g, const int *forced,
                       int *acc, int *comm, bool carry_rows = false) {
  dflow_handle *h = k.h;
  KL(klaunch(k_accept, (st->batch + 31) / 32, 32, 0, k.s, blk, g, forced, st->tokens, st->seq_len, st->active,
                                                 st->batch, h->D.B, h->cfg.max_ctx, acc, comm, k.status_w,
                                                 carry_rows ? h->pos2 : nullptr, carry_rows ? h->wr2 : nullptr));
  CK(cudaGetLastError());
  return DFLOW_OK;
}

template <typename T>
// rows_ready: the accept kernel of the same round already wrote pos2 / wr2
dflow_status do_carry(const Call &k, dflow_state *st, const int *blk, const void *feats, const int *acc,
                      int relay, bool rows_ready = false) {
  dflow_handle *h = k.h;
  const Dims D = round_dims(h);
  const int batch = st->batch, rows = batch * D.R;
  if (!rows_ready) {
    KL(klaunch(k_carry_rows, (rows + 127) / 128, 128, 0, k.s, acc, st->seq_len, batch, D.R, h->pos2, h->wr2,
               k.status));
    CK(cudaGetLastError());
  }
  CK(ctx_append<T>(k, D, rows, st, feats));
  KL(klaunch(k_carry<T>, dim3(batch, D.B), 256, 0, k.s, (const T *)feats, acc, blk, st->tokens, st->seq_len,
                                               h->cfg.max_ctx, (T *)st->carry, st->n_carry, st->boundary,
                                               D.d, D.B, relay, k.status));
  CK(cudaGetLastError());
  return DFLOW_OK;
}

// Sec. 5.2, T = 1: draft (samples) -> verify (logits) -> speculative sampling
// (acceptance length and the token after it) -> Eq. 3 commit with that
// acceptance forced -> carry
template <typename T>
dflow_status do_round_sampled(const Call &k, dflow_state *st, SampRound sr, int *acc, int *comm, int relay,
                              float *qlog, float *plog) {
  dflow_handle *h = k.h;
  const int batch = st->batch, R = h->R;
  dflow_status r;
  if ((r = do_draft<T>(k, st, h->blk, relay, qlog, &sr))) return r;
  if ((r = do_verify<T>(k, st, h->blk, nullptr, h->feats, plog, true))) return r;
  int n = 0;
  const cudaError_t e = samp_verify(plog, qlog, h->D.vocab, R, batch, sr, h->samp, h->blk, st->active, h->g,
                                    k.status, k.s, &n);
  h->n_launch += n;
  h->dep.brk();
  CK(e);
  CK(cudaGetLastError());
  if ((r = do_accept(k, st, h->blk, h->g, h->samp.a, acc, comm, true))) return r;
  return do_carry<T>(k, st, h->blk, h->feats, acc, relay, true);
}

// Sec. 5.2 baseline: one greedy step of the target alone.  The step runs on the
// block-verify launches of a round: every row of the block holds the anchor, row
// 0 is the step (the anchor at position n-1: its K/V, its Eq. 1 feature and its
// prediction) and rows 1..B are computed and dropped (their K/V lie past the
// committed length).  At batch 1 every projection streams the same weights for
// one row or B+1, so the step costs about one verify pass.
template <typename T>
dflow_status do_decode(const Call &k, dflow_state *st, int *token_out, int draft_context) {
  dflow_handle *h = k.h;
  const int batch = st->batch, R = h->R, rows = batch * R;
  KL(klaunch(k_decode_block, (rows + 127) / 128, 128, 0, k.s, h->blk, st->tokens, st->seq_len, st->active, batch, R,
             h->cfg.max_ctx, k.status));
  CK(cudaGetLastError());
  dflow_status r;
  if ((r = do_verify<T>(k, st, h->blk, h->g, h->feats, nullptr))) return r;
  // commit the prediction of row 0: Eq. 3 with the acceptance forced to 0 commits exactly that token
  if ((r = do_accept(k, st, h->blk, h->g, h->zeros, h->acc, h->comm))) return r;
  if (draft_context && (r = do_carry<T>(k, st, h->blk, h->feats, h->acc, 0))) return r;
  KL(klaunch(k_decode_finish, (batch + 127) / 128, 128, 0, k.s, h->acc, h->comm, R, token_out, st->n_carry,
             st->boundary, batch, k.status));
  CK(cudaGetLastError());
  return DFLOW_OK;
}

// device-side checks of the state before a call that writes `rows` rows per sequence
dflow_status guard_rows(const Call &k, dflow_state *st, int rows) {
  dflow_handle *h = k.h;
  KL(klaunch(k_guard, (st->batch + 127) / 128, 128, 0, k.s, st->tokens, st->seq_len, st->n_carry, st->boundary,
                                                   st->active, st->batch, rows, h->cfg.max_ctx,
                                                   h->D.vocab, h->D.B, k.status_w));
  CK(cudaGetLastError());
  return DFLOW_OK;
}
dflow_status guard(const Call &k, dflow_state *st) { return guard_rows(k, st, k.h->R); }

template <typename T>
dflow_status do_prefill(const Call &k, dflow_state *st, const int *prompt, int stride, const int *plen_host) {
  dflow_handle *h = k.h;
  Dims D = h->D;
  D.R = PF;
  const int batch = st->batch, rows = batch * PF;
  int maxlen = 0;
  for (int b = 0; b < batch; ++b) maxlen = std::max(maxlen, plen_host[b]);
  CK(cudaMemcpyAsync(h->plen, plen_host, sizeof(int) * batch, cudaMemcpyHostToDevice, k.s));
  const int splits = pick_splits(h, batch, rows);
  for (int c0 = 0; c0 < maxlen; c0 += PF) {
    KL(klaunch(k_rows_prefill, (rows + 127) / 128, 128, 0, k.s, h->pos, h->wr, h->kvlen, h->plen, batch, c0, k.status));
    CK(cudaGetLastError());
    KL(klaunch(k_embed<T>, rows, 256, 0, k.s, (const T *)h->w.embed, prompt + c0, stride, PF, (const int *)h->wr,
               h->x, D.d, D.vocab, h->fused ? (T *)h->xn : nullptr, h->tl[0].attn_norm, h->ss, h->rows_max,
               k.status_w));
    CK(cudaGetLastError());
    CK(target_forward<T>(k, D, batch, st, h->g, h->feats, nullptr, splits));
    KL(klaunch(k_prefill_commit, (rows + 127) / 128, 128, 0, k.s, prompt, stride, h->plen, h->pos, h->wr, h->g, batch,
                                                          h->cfg.max_ctx, st->tokens, st->seq_len,
                                                          st->n_carry, st->boundary, k.status));
    CK(cudaGetLastError());
    CK(cudaMemcpyAsync(h->pos2, h->pos, sizeof(int) * rows, cudaMemcpyDeviceToDevice, k.s));
    CK(cudaMemcpyAsync(h->wr2, h->wr, sizeof(int) * rows, cudaMemcpyDeviceToDevice, k.s));
    CK(ctx_append<T>(k, D, rows, st, h->feats));
  }
  return DFLOW_OK;
}

dflow_status check_call(dflow_handle *h, const dflow_state *st) {
  if (!h || !st) return DFLOW_ERR_INVALID_ARG;
  if (!h->ws) return DFLOW_ERR_INVALID_ARG;
  if (st->batch < 1 || st->batch > h->cfg.max_batch) return DFLOW_ERR_INVALID_ARG;
  if (!st->tokens || !st->seq_len || !st->page_table || !st->kv || !st->draft_kv || !st->carry ||
      !st->n_carry || !st->boundary || !st->active || !st->status)
    return DFLOW_ERR_INVALID_ARG;
  return DFLOW_OK;
}

// start of a call: its first counting launch waits for the previous grid; after a
// failed call the counters are zeroed (a launch may have been counted but not run)
void prep_chain(dflow_handle *h, void *stream) {
  DepChain &d = h->dep;
  if (d.dirty && d.dev != nullptr) {
    // with the counters, the persistent GEMM's leftover sums (a failed launch may have left partials)
    if (cudaMemsetAsync(d.dev, 0, kDepSlots * sizeof(unsigned int), (cudaStream_t)stream) == cudaSuccess &&
        (!h->use_tc || tc_init(h->tcw, (cudaStream_t)stream) == cudaSuccess)) {
      for (int i = 0; i < kDepSlots; ++i) d.shadow[i] = 0;
      d.next = 0;
      d.dirty = false;
    } else {
      cudaGetLastError();
      d.dev = nullptr;  // counting off for this handle: every launch waits for its predecessor's grid
    }
  }
  d.brk();
}

Call make_call(dflow_handle *h, dflow_state *st, void *stream) {
  prep_chain(h, stream);
  return Call{h, st->status, st->status, (cudaStream_t)stream};
}

// a failed call leaves the counters unknown
dflow_status finish(dflow_handle *h, dflow_status r) {
  if (r != DFLOW_OK) h->dep.dirty = true;
  return r;
}

bool valid_layer(const dflow_layer_weights &L) {
  return L.w_qkv && L.w_o && L.w_gate_up && L.w_down && L.attn_norm && L.mlp_norm && L.q_norm && L.k_norm;
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

extern "C" {

const char *dflow_status_string(dflow_status s) {
  switch (s) {
    case DFLOW_OK: return "ok";
    case DFLOW_ERR_INVALID_ARG: return "invalid argument";
    case DFLOW_ERR_CUDA: return "CUDA runtime error";
    case DFLOW_ERR_CAPACITY: return "sequence capacity exhausted";
    case DFLOW_ERR_DEVICE_TIMEOUT: return "bounded device wait timed out";
    case DFLOW_ERR_UNSUPPORTED: return "unsupported shape or device";
    case DFLOW_ERR_BAD_STATE: return "token or count out of range";
  }
  return "unknown status";
}

dflow_status dflow_create(const dflow_config *cfg, const dflow_weights *w, dflow_handle **out) {
  if (!cfg || !w || !out) return DFLOW_ERR_INVALID_ARG;
  *out = nullptr;
  const dflow_config &c = *cfg;
  if (c.dtype != DFLOW_F32 && c.dtype != DFLOW_BF16) return DFLOW_ERR_INVALID_ARG;
  if (c.d_model <= 0 || c.n_layers <= 0 || c.n_q_heads <= 0 || c.n_kv_heads <= 0 || c.d_inter <= 0 ||
      c.vocab <= 0 || c.draft_layers <= 0 || c.block <= 0 || c.page_size <= 0 || c.max_batch <= 0 ||
      c.max_ctx <= 0 || c.num_pages <= 0)
    return DFLOW_ERR_INVALID_ARG;
  if (c.head_dim != 64 && c.head_dim != 128) return DFLOW_ERR_UNSUPPORTED;
  if (c.dtype == DFLOW_BF16 && (c.head_dim != 128 || c.page_size != 64)) return DFLOW_ERR_UNSUPPORTED;
  if (c.d_model % 128 || c.d_inter % 64 || c.n_q_heads % c.n_kv_heads || c.max_ctx % c.page_size)
    return DFLOW_ERR_UNSUPPORTED;
  if (c.n_feat < 1 || c.n_feat > DFLOW_MAX_FEAT) return DFLOW_ERR_INVALID_ARG;
  for (int i = 0; i < c.n_feat; ++i)
    if (c.feat_layers[i] < 1 || c.feat_layers[i] > c.n_layers) return DFLOW_ERR_INVALID_ARG;
  if (!w->embed || !w->lm_head || !w->final_norm || !w->target || !w->draft || !w->draft_final_norm ||
      !w->w_c || !w->c_norm || !w->e_mask || !w->relay_w1 || !w->relay_w2 || !w->ln_w || !w->ln_b)
    return DFLOW_ERR_INVALID_ARG;
  for (int l = 0; l < c.n_layers; ++l)
    if (!valid_layer(w->target[l])) return DFLOW_ERR_INVALID_ARG;
  for (int l = 0; l < c.draft_layers; ++l)
    if (!valid_layer(w->draft[l])) return DFLOW_ERR_INVALID_ARG;

  dflow_handle *h = new (std::nothrow) dflow_handle();
  if (!h) return DFLOW_ERR_INVALID_ARG;
  h->cfg = c;
  h->w = *w;
  h->tl.assign(w->target, w->target + c.n_layers);
  h->dl.assign(w->draft, w->draft + c.draft_layers);
  h->w.target = h->tl.data();
  h->w.draft = h->dl.data();
  Dims &D = h->D;
  D.d = c.d_model;
  D.hq = c.n_q_heads;
  D.hkv = c.n_kv_heads;
  D.hd = c.head_dim;
  D.inter = c.d_inter;
  D.vocab = c.vocab;
  D.B = c.block;
  D.R = c.block + 1;
  D.page_size = c.page_size;
  D.num_pages = c.num_pages;
  D.max_ctx = c.max_ctx;
  D.pages_per_seq = c.max_ctx / c.page_size;
  D.n_feat = c.n_feat;
  D.rms_eps = c.rms_eps;
  D.ln_eps = c.ln_eps;
  h->dtype = c.dtype;
  h->esz = c.dtype == DFLOW_BF16 ? 2 : 4;
  h->R = c.block + 1;
  h->rows_round = c.max_batch * h->R;
  h->rows_max = c.max_batch * std::max(h->R, PF);
  h->vocab_tiles = (c.vocab + 127) / 128;
  h->gld = std::max((c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim, 2 * c.d_model);
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaGetLastError();
  h->sm_count = sms > 0 ? sms : 148;
  const int sr = std::min(64, std::max(1, (2 * h->sm_count + c.n_kv_heads * c.max_batch - 1) / (c.n_kv_heads * c.max_batch)));
  h->attn_entries = std::max((size_t)h->rows_round * c.n_q_heads * sr, (size_t)h->rows_max * c.n_q_heads * std::min(sr, 4));
  // bf16 models run on the tensor-core kernels (sm_103, checked when the
  // workspace is handed over); fp32 (the parity model) on CUDA cores
  h->use_tc = c.dtype == DFLOW_BF16;
  h->fused = h->use_tc;
  h->ws_need = layout(h, nullptr);
  *out = h;
  return DFLOW_OK;
}

dflow_status dflow_workspace_size(const dflow_handle *h, size_t *bytes) {
  if (!h || !bytes) return DFLOW_ERR_INVALID_ARG;
  *bytes = h->ws_need;
  return DFLOW_OK;
}

dflow_status dflow_set_workspace(dflow_handle *h, void *dev, size_t bytes) {
  if (!h || !dev || bytes < h->ws_need || ((uintptr_t)dev & 255)) return DFLOW_ERR_INVALID_ARG;
  if (h->use_tc) {
    int dev_id = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev_id) != cudaSuccess ||
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev_id) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev_id) != cudaSuccess) {
      cudaGetLastError();
      return DFLOW_ERR_CUDA;
    }
    if (major != 10 || minor != 3) return DFLOW_ERR_UNSUPPORTED;
  }
  h->ws = static_cast<char *>(dev);
  h->ws_bytes = bytes;
  layout(h, h->ws);
  const long long n = (long long)h->cfg.max_ctx * (h->D.hd / 2);
  k_rope_table<<<(int)std::min<long long>((n + 255) / 256, 4096), 256>>>(h->rope, h->cfg.max_ctx, h->D.hd,
                                                                          (double)h->cfg.rope_theta);
  CK(cudaGetLastError());
  CK(cudaMemset(h->zeros, 0, sizeof(int) * h->cfg.max_batch));
  if (h->use_tc) CK(tc_init(h->tcw, 0));
  CK(cudaDeviceSynchronize());
  return DFLOW_OK;
}

dflow_status dflow_destroy(dflow_handle *h) {
  if (!h) return DFLOW_ERR_INVALID_ARG;
  for (cudaEvent_t e : h->ev_pool) cudaEventDestroy(e);
  delete h;
  return DFLOW_OK;
}

dflow_status dflow_prefill(dflow_handle *h, dflow_state *st, const int32_t *prompt, int32_t prompt_stride,
                           const int32_t *prompt_len_host, void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!prompt || !prompt_len_host || prompt_stride < 1) return DFLOW_ERR_INVALID_ARG;
  for (int b = 0; b < st->batch; ++b) {
    const int len = prompt_len_host[b];
    if (len < 1 || len > prompt_stride) return DFLOW_ERR_INVALID_ARG;
    if (len + 1 + h->R > h->cfg.max_ctx) return DFLOW_ERR_CAPACITY;
  }
  Call k = make_call(h, st, stream);
  return finish(h, h->dtype == DFLOW_BF16 ? do_prefill<bf16>(k, st, prompt, prompt_stride, prompt_len_host)
                                          : do_prefill<float>(k, st, prompt, prompt_stride, prompt_len_host));
}

dflow_status dflow_draft_block(dflow_handle *h, dflow_state *st, int32_t *block_tokens, float *logits,
                               void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!block_tokens) return DFLOW_ERR_INVALID_ARG;
  Call k = make_call(h, st, stream);
  return finish(h, h->dtype == DFLOW_BF16 ? do_draft<bf16>(k, st, block_tokens, 1, logits)
                                          : do_draft<float>(k, st, block_tokens, 1, logits));
}

dflow_status dflow_verify_block(dflow_handle *h, dflow_state *st, const int32_t *block_tokens,
                                int32_t *target_argmax, void *feats, float *logits, void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!block_tokens || !target_argmax || !feats) return DFLOW_ERR_INVALID_ARG;
  Call k = make_call(h, st, stream);
  return finish(h, h->dtype == DFLOW_BF16 ? do_verify<bf16>(k, st, block_tokens, target_argmax, feats, logits)
                                          : do_verify<float>(k, st, block_tokens, target_argmax, feats, logits));
}

dflow_status dflow_accept_commit(dflow_handle *h, dflow_state *st, const int32_t *block_tokens,
                                 const int32_t *target_argmax, const int32_t *forced_accept,
                                 int32_t *accept_len, int32_t *committed, void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!block_tokens || !target_argmax || !accept_len || !committed) return DFLOW_ERR_INVALID_ARG;
  Call k = make_call(h, st, stream);
  return finish(h, do_accept(k, st, block_tokens, target_argmax, forced_accept, accept_len, committed));
}

dflow_status dflow_carry_hidden(dflow_handle *h, dflow_state *st, const int32_t *block_tokens,
                                const void *feats, const int32_t *accept_len, void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!block_tokens || !feats || !accept_len) return DFLOW_ERR_INVALID_ARG;
  Call k = make_call(h, st, stream);
  return finish(h, h->dtype == DFLOW_BF16 ? do_carry<bf16>(k, st, block_tokens, feats, accept_len, 1)
                                          : do_carry<float>(k, st, block_tokens, feats, accept_len, 1));
}

dflow_status dflow_round(dflow_handle *h, dflow_state *st, const int32_t *forced_accept, int32_t *accept_len,
                         int32_t *committed, int32_t relay, void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!accept_len || !committed) return DFLOW_ERR_INVALID_ARG;
  Call k = make_call(h, st, stream);
  if (h->dtype == DFLOW_BF16) {
    if ((r = do_draft<bf16>(k, st, h->blk, relay))) return finish(h, r);
    if ((r = do_verify<bf16>(k, st, h->blk, h->g, h->feats, nullptr, true))) return finish(h, r);
    if ((r = do_accept(k, st, h->blk, h->g, forced_accept, accept_len, committed, true))) return finish(h, r);
    return finish(h, do_carry<bf16>(k, st, h->blk, h->feats, accept_len, relay, true));
  }
  if ((r = do_draft<float>(k, st, h->blk, relay))) return finish(h, r);
  if ((r = do_verify<float>(k, st, h->blk, h->g, h->feats, nullptr, true))) return finish(h, r);
  if ((r = do_accept(k, st, h->blk, h->g, forced_accept, accept_len, committed, true))) return finish(h, r);
  return finish(h, do_carry<float>(k, st, h->blk, h->feats, accept_len, relay, true));
}

dflow_status dflow_round_sampled(dflow_handle *h, dflow_state *st, uint64_t seed, int32_t round_index,
                                 int32_t *accept_len, int32_t *committed, int32_t relay, float *draft_logits,
                                 float *verify_logits, void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!accept_len || !committed || round_index < 0 || round_index >= (1 << 24)) return DFLOW_ERR_INVALID_ARG;
  Call k = make_call(h, st, stream);
  const SampRound sr{seed, round_index};
  float *q = draft_logits ? draft_logits : h->qlog, *p = verify_logits ? verify_logits : h->plog;
  return finish(h, h->dtype == DFLOW_BF16 ? do_round_sampled<bf16>(k, st, sr, accept_len, committed, relay, q, p)
                                          : do_round_sampled<float>(k, st, sr, accept_len, committed, relay, q, p));
}

dflow_status dflow_decode_step(dflow_handle *h, dflow_state *st, int32_t *token_out, int32_t draft_context,
                               void *stream) {
  dflow_status r = check_call(h, st);
  if (r) return r;
  if (!token_out) return DFLOW_ERR_INVALID_ARG;
  Call k = make_call(h, st, stream);
  if ((r = guard(k, st))) return finish(h, r);
  return finish(h, h->dtype == DFLOW_BF16 ? do_decode<bf16>(k, st, token_out, draft_context)
                                          : do_decode<float>(k, st, token_out, draft_context));
}

dflow_status dflow_profile_enable(dflow_handle *h, int32_t enable) {
  if (!h) return DFLOW_ERR_INVALID_ARG;
  h->prof = enable != 0;
  h->prof_recs.clear();
  h->ev_next = 0;
  return DFLOW_OK;
}

dflow_status dflow_profile_read(dflow_handle *h, dflow_kernel_profile *out) {
  if (!h || !out) return DFLOW_ERR_INVALID_ARG;
  for (int i = 0; i < DFLOW_PROF_N; ++i) out[i] = dflow_kernel_profile{0, 0.0, 0.0, 0.0};
  for (auto &r : h->prof_recs) {
    CK(cudaEventSynchronize(r.e1));
    float ms = 0.f;
    CK(cudaEventElapsedTime(&ms, r.e0, r.e1));
    dflow_kernel_profile &o = out[r.kind];
    o.launches += 1;
    o.total_ms += ms;
    o.alg_bytes += r.bytes;
    o.alg_flops += r.flops;
  }
  return DFLOW_OK;
}

dflow_status dflow_debug_gemm(dflow_handle *h, int32_t path, const void *W, int32_t N, int32_t K, const void *X,
                              int32_t M, int32_t ldx, int32_t mode, void *out, int32_t ldo, int32_t *status,
                              void *stream) {
  if (!h || !h->ws || !W || !X || !out || !status || N < 1 || K < 1 || M < 1 || ldx < K) return DFLOW_ERR_INVALID_ARG;
  if ((path >= 1) != (h->dtype == DFLOW_BF16) || path < 0 || path > 3) return DFLOW_ERR_UNSUPPORTED;
  if (path == 2 && (mode == EP_ARGMAX || K % 64 || K / 64 < 4 || ldx % 8 || !seq_supported(M)))
    return DFLOW_ERR_UNSUPPORTED;
  if (mode < 0 || mode > 4) return DFLOW_ERR_INVALID_ARG;
  if (mode == EP_ARGMAX && ((N + 127) / 128 > h->vocab_tiles || M > h->rows_max)) return DFLOW_ERR_INVALID_ARG;
  if (K % 32) return DFLOW_ERR_UNSUPPORTED;
  cudaStream_t s = (cudaStream_t)stream;
  EpArgs ep{};
  ep.mode = mode;
  if (mode == EP_STORE_F32 || mode == EP_RESID) {
    ep.out_f32 = static_cast<float *>(out);
    ep.ldo = ldo;
  } else if (mode == EP_SWIGLU || mode == EP_SILU) {
    ep.out_t = out;
    ep.ldt = ldo;
  } else {
    ep.part_val = h->am_val;
    ep.part_idx = h->am_idx;
    ep.n_tiles = (N + 127) / 128;
  }
  cudaError_t e;
  if (path == 2) {
    // the persistent launch the round uses for few-row projections, as one GEMM
    prep_chain(h, stream);
    if (h->dep.dev == nullptr) return DFLOW_ERR_UNSUPPORTED;
    const SeqSpec sp{W, N, K, X, ldx, ep};
    e = gemm_seq(h->tcw, 1, &sp, M, status, s, &h->dep);
    h->dep.brk();
    if (e != cudaSuccess) h->dep.dirty = true;
  } else if (path == 3) {
    e = gemm_wide(h->tcw, W, N, K, X, M, ldx, ep, status, s);
  } else if (path == 1) {
    e = tc_supports(N, K, M, ldx, ep) ? gemm_tc(h->tcw, W, N, K, X, M, ldx, ep, status, s) : cudaErrorNotSupported;
  } else {
    e = gemm_simt(h->dtype, W, N, K, X, M, ldx, ep, status, s);
  }
  if (e == cudaErrorNotSupported) return DFLOW_ERR_UNSUPPORTED;
  CK(e);
  if (mode == EP_ARGMAX) {
    klaunch(k_argmax_reduce, (M + 7) / 8, 256, 0, s, h->am_val, h->am_idx, ep.n_tiles, M, static_cast<int *>(out), status,
            BlockOut{});
    CK(cudaGetLastError());
  }
  return DFLOW_OK;
}

dflow_status dflow_launch_count(const dflow_handle *h, uint64_t *count) {
  if (!h || !count) return DFLOW_ERR_INVALID_ARG;
  *count = h->n_launch;
  return DFLOW_OK;
}

dflow_status dflow_read_status(dflow_handle *h, const dflow_state *st, int32_t *host_status, void *stream) {
  if (!h || !st || !st->status || !host_status) return DFLOW_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize((cudaStream_t)stream));
  CK(cudaMemcpy(host_status, st->status, sizeof(int32_t), cudaMemcpyDeviceToHost));
  return DFLOW_OK;
}

}  // extern "C"
