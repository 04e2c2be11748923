// tcgen05 (5th-generation tensor core) weight-streaming GEMM for bf16.
#pragma once
#include <cuda.h>

#include "dflow_internal.cuh"

namespace dflow {

// 2D tensor map of a bf16 row-major [rows][ld] matrix, box 64 columns x box_rows
// rows, 128-byte swizzle (cached by arguments).
bool tensor_map(CUtensorMap *out, const void *ptr, int rows, int cols, int ld, int box_rows, bool use_cache = true);
// 3D tensor map of a bf16 [d2][d1][d0] array (d0 contiguous), box 64 x b1 x b2,
// 128-byte swizzle (not cached)
bool tensor_map_3d(CUtensorMap *out, const void *ptr, int d0, int d1, int d2, int b1, int b2);

// Scratch of the tensor-core GEMM inside the handle's workspace.
struct TcWorkspace {
  int sm_count = 0;
  // persistent launch: fp32 sums and arrival counts of tiles split over several
  // clusters (zero between uses; tc_init zeroes them)
  float *lacc = nullptr;
  unsigned int *lctr = nullptr;
  // wide launch (more than 128 token rows): per-tile arrival counts (zero
  // between uses, right after lctr) and the fp32 split-K partial slots
  unsigned int *wctr = nullptr;
  float *wslots = nullptr;
  size_t wslot_bytes = 0;
  size_t left_bytes = 0;  // lacc, lctr and wctr: zeroed by tc_init
};

// Reserve the GEMM scratch at byte offset `off` of `base` (null base: size only).
void tc_layout(TcWorkspace &w, char *base, size_t &off, int sm_count, size_t rows_max, int max_tiles);
// True when the tensor-core kernel covers this problem (bf16, alignment, sizes).
bool tc_supports(int N, int K, int M, int ldx, const EpArgs &ep);
// Zero the counters once after the workspace is handed over.
cudaError_t tc_init(const TcWorkspace &w, cudaStream_t s);
// use_caches = false: tensor maps are encoded on the stack and the launch plan
// is recomputed, so the call touches no host heap
// chain: completion counters of the caller's launch sequence, or null (grid waits)
cudaError_t gemm_tc(const TcWorkspace &w, const void *W, int N, int K, const void *X, int M,
                    int ldx, const EpArgs &ep, int *status, cudaStream_t s, bool use_caches = true,
                    DepChain *chain = nullptr);

// One projection over up to 512 token rows per pass in a single stream of the
// weights (any M: passes of 512 rows), split over k in independent CTAs when
// the tiles are too few to fill the GPU; modes as gemm_tc.
// whether gemm_wide has a schedule for this shape (above 128 rows it beats the
// row-tiled launches on every projection shape measured, k-split or not: its
// split's partial tiles are reduced by all CTAs of the tile, each finishing its
// share of the token columns)
bool gemm_wide_suits(const TcWorkspace &w, int N, int K, int M);
cudaError_t gemm_wide(const TcWorkspace &w, const void *W, int N, int K, const void *X, int M, int ldx,
                      const EpArgs &ep, int *status, cudaStream_t s, DepChain *chain = nullptr);

// One GEMM of a persistent sequence (out[m][n] = X[m][:] . W[n][:] with a
// fused epilogue; modes EP_STORE_F32, EP_RESID, EP_SWIGLU, EP_QKV).
struct SeqSpec {
  const void *W;
  int N, K;
  const void *X;
  int ldx;
  EpArgs ep;
};
// True when up to 4 GEMMs over M rows can run as one persistent launch.
bool seq_supported(int M);
// The attention of one layer, run as the first phase of a persistent launch
// whose first GEMM reads its output (the O projection).
struct SeqAttnSpec {
  Dims D;     // D.R: rows per sequence
  int batch;
  AttnArgs a;  // q, pool (this layer), page table, block K/V (drafter), pos, seq_len, kvlen, causal, out
};
// True when the attention can be such a phase: 128-dim heads, 64-token pages,
// one 128-row group of query rows per (kv head, sequence), M <= 128 rows.
bool seq_attn_supported(const Dims &D, int batch, int M);
// The GEMMs of `sp` in order, in one launch: GEMM j's activations are read once
// every tile of GEMM j - 1 is finished; the first waits for the previous launch
// in `chain` (required), the next launch waits for the last GEMM.  independent:
// no GEMM reads another's output (all wait only for the previous launch; the next
// launch waits for all of them); Q/K/V epilogues may then appear more than once
// if they share their column table.
// att: the attention phase ahead of the first GEMM (not with independent), or null.
cudaError_t gemm_seq(const TcWorkspace &w, int n, const SeqSpec *sp, int M, int *status, cudaStream_t s,
                     DepChain *chain, bool independent = false, const SeqAttnSpec *att = nullptr);

}  // namespace dflow
