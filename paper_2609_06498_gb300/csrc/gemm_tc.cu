// Weight-streaming GEMM on the 5th-generation tensor cores (tcgen05 + TMEM),
// fed by TMA, for the dense projections of the round (Qwen3 QKV / O / gate-up /
// down, the Eq. 1 feature projection, the Eq. 4 relay MLP, the drafter context
// K/V projection and the LM head).
//
// out[m][n] = sum_k X[m][k] W[n][k] with few rows m (the B+1 block rows of each
// sequence) and many output features n.  The kernel computes the transposed
// product D[n][m] = W[n][:] . X[m][:] so the weight tile is the 128-row A
// operand and the token rows are the MMA's N dimension (padded to 16).
//
//   * The grid is Q clusters of P CTAs (one CTA per SM).  Cluster q owns the
//     128-feature weight tiles q, q+Q, q+2Q, ...; inside a tile the P CTAs of
//     the cluster split the K range (split-K) so that P*Q SMs stream weights.
//   * In each CTA, warp 0 streams W and X k-blocks with TMA (128-byte swizzle)
//     into a ring of shared-memory stages; warp 1 issues tcgen05.mma
//     (128 x Npad x 16) into a TMEM accumulator (two buffers, so one tile's
//     reduction overlaps the next tile's MMAs); warps 2-5 drain the
//     accumulator with tcgen05.ld.
//   * Split-K partials meet in distributed shared memory: each CTA parks its
//     fp32 partial in its own shared memory, signals its peers' mbarriers,
//     and sums one slice of the token columns over the P partials (in rank
//     order, so the result is deterministic) before running the fused
//     epilogue on that slice.  No partial leaves the cluster.
//   * Every mbarrier wait is bounded (about 2 s of globaltimer); on expiry the
//     kernel records DFLOW_ERR_DEVICE_TIMEOUT, drains its own copies and MMAs,
//     frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <map>
#include <mutex>
#include <tuple>
#include <unordered_map>

#include "attn_t5.cuh"
#include "gemm_tc.cuh"
#include "ptx.cuh"

namespace dflow {

namespace {

using namespace ptx;

constexpr int BM = 128;           // weight rows per tile (MMA M)
constexpr int BK = 64;            // k elements per k-block (128 bytes of bf16: one swizzle row)
constexpr int A_BYTES = BM * BK * 2;
constexpr int MAX_NPAD = 256;    // token columns of one k_gemm_tc pass (one MMA's N)
constexpr int MAX_COLS = 512;    // token columns of the per-column tables (k_gemm_wide: two MMAs per k-step)
constexpr int MAX_SPLIT_NPAD = 64;  // split-K (P > 1) only for up to 64 token columns
constexpr int SEQ_MAX_NPAD = 128;   // token columns of the persistent layer-segment kernel
constexpr int THREADS = 192;
constexpr int SMEM_BUDGET = 224 * 1024;

struct Params {
  int N, K, M, npad, T, kb, P, Q, stages, tmem_cols, rx_bytes;
  uint32_t idesc;
  EpArgs ep;
  int *status;
  Dep dep;
};

struct Smem {
  // recv: this CTA's slice of the split-K partials has arrived (armed by the CTA
  // itself, completed by its peers' bytes); rfree: every owner has consumed
  // this CTA's previous pushes (one arrival per peer)
  // ovf (one-pass GEMM with overlapping accumulators): the epilogue has read the
  // columns its buffer shares with the other one
  uint64_t full[16], empty[16], accf[2], acce[2], recv, rfree, drain, ovf;
  uint32_t tmem;
  int flag;
  int abort;
  int left_last;  // the leftover part just finished completed its columns' count
  alignas(16) float xch[16][64];  // also the QKV epilogue's bf16 staging tile [16][128]
  float rv[4][16];
  int ri[4][16];
  float ssred[4][16];
  float col_scale[MAX_COLS];
  long long qkv_base[MAX_COLS];  // EP_QKV, paged pool: element offset of the column's K slot of kv head 0, or -1
  int qkv_pos[MAX_COLS];         // EP_QKV: position of the column's row
};

// epilogue inputs that do not depend on the product, loaded while the MMAs run
struct EpPre {
  float x[16];    // EP_RESID: residual stream values of this row's feature at the chunk's columns
  float gain;     // EP_RESID: next RMSNorm gain of the feature (out_xn)
  float2 cs[16];  // EP_QKV: rotary (cos, sin) of pair r at the chunk's columns' positions
  float gn;       // EP_QKV: q or k RMSNorm gain of row r
};

// SiLU from the fast exponential and division intrinsics (the result is rounded to bf16)
__device__ __forceinline__ float silu_fast(float x) { return __fdividef(x, 1.0f + __expf(-x)); }

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// sums of x[0..15] over the warp's 32 lanes by recursive halving: at each step a
// lane keeps half of its columns and adds the partner's copy of them, so 16
// shuffles do the work of 16 butterfly reductions (80).  Returns the sum of
// column (lane >> 1) & 15 (lanes 2c and 2c + 1 both hold column c).
__device__ __forceinline__ float warp_column_sums16(const float *x, int lane) {
  constexpr unsigned FULL = 0xffffffffu;
  float a[8], b[4], c[2];
  const bool h16 = lane & 16, h8 = lane & 8, h4 = lane & 4, h2 = lane & 2;
#pragma unroll
  for (int k = 0; k < 8; ++k)
    a[k] = (h16 ? x[k + 8] : x[k]) + __shfl_xor_sync(FULL, h16 ? x[k] : x[k + 8], 16);
#pragma unroll
  for (int k = 0; k < 4; ++k)
    b[k] = (h8 ? a[k + 4] : a[k]) + __shfl_xor_sync(FULL, h8 ? a[k] : a[k + 4], 8);
#pragma unroll
  for (int k = 0; k < 2; ++k)
    c[k] = (h4 ? b[k + 2] : b[k]) + __shfl_xor_sync(FULL, h4 ? b[k] : b[k + 2], 4);
  float d = (h2 ? c[1] : c[0]) + __shfl_xor_sync(FULL, h2 ? c[0] : c[1], 2);
  return d + __shfl_xor_sync(FULL, d, 1);
}

// per-column sum over the tile's 128 rows (all epilogue threads call it)
__device__ __forceinline__ void column_sums(Smem &sm, int sub, int lane, const float *x, float *out) {
  const float d = warp_column_sums16(x, lane);
  if (!(lane & 1)) sm.ssred[sub][(lane >> 1) & 15] = d;
  epi_bar();
#pragma unroll
  for (int j = 0; j < 16; ++j) out[j] = sm.ssred[0][j] + sm.ssred[1][j] + sm.ssred[2][j] + sm.ssred[3][j];
  epi_bar();
}

// sm.col_scale[c] = rsqrt(sum_e in_ss[e][c] / d + eps) for the M columns: the
// input rows' RMSNorm folded into the product.  All 128 epilogue threads load
// (a column and a stride of the partials each, so the L2 loads overlap), then
// the groups' sums are added in a fixed order.
__device__ __forceinline__ void col_scales(const EpArgs &ep, Smem &sm, int M, int r) {
  if (M > 64) {
    for (int c = r; c < M; c += BM) {
      float acc0 = 0.f, acc1 = 0.f;
      int e = 0;
#pragma unroll 4
      for (; e + 1 < ep.in_ss_n; e += 2) {
        acc0 += __ldcg(ep.in_ss + (size_t)e * ep.ld_ss + c);
        acc1 += __ldcg(ep.in_ss + (size_t)(e + 1) * ep.ld_ss + c);
      }
      if (e < ep.in_ss_n) acc0 += __ldcg(ep.in_ss + (size_t)e * ep.ld_ss + c);
      sm.col_scale[c] = rsqrtf((acc0 + acc1) * ep.in_inv_d + ep.in_eps);
    }
    epi_bar();
    return;
  }
  const int cols = M <= 32 ? 32 : 64, groups = BM / cols;
  const int c = r % cols, q = r / cols;
  const float *const src = ep.in_ss + c;
  const int n = ep.in_ss_n;
  const size_t ld = ep.ld_ss;
  float acc0 = 0.f, acc1 = 0.f;
  if (c < M) {
    int e = q;
#pragma unroll 4
    for (; e + groups < n; e += 2 * groups) {
      acc0 += __ldcg(src + (size_t)e * ld);
      acc1 += __ldcg(src + (size_t)(e + groups) * ld);
    }
    if (e < n) acc0 += __ldcg(src + (size_t)e * ld);
  }
  float *const part = &sm.xch[0][0];  // [groups][cols]
  part[q * cols + c] = acc0 + acc1;
  epi_bar();
  if (r < M) {
    float tot = 0.f;
    for (int g = 0; g < groups; ++g) tot += part[g * cols + r];
    sm.col_scale[r] = rsqrtf(tot * ep.in_inv_d + ep.in_eps);
  }
  epi_bar();
}

// token column -> position and paged-pool slot of the Q/K/V epilogue
__device__ __forceinline__ void qkv_table(const QkvOut &o, Smem &sm, int M, int r) {
  for (int c = r; c < M; c += BM) {
    const int grow = o.row0 + c, pp = o.pos[grow];
    long long base = -1;
    if (o.bk == nullptr && o.wr[grow]) {
      const int page = o.page_table[(size_t)(grow / o.R) * o.pages_per_seq + pp / o.page_size];
      base = ((long long)page * 2 * o.hkv * o.page_size + pp % o.page_size) * BM;
    }
    sm.qkv_pos[c] = pp;
    sm.qkv_base[c] = base;
  }
}

// prefetch of the inputs epilogue_chunk(t, c0, nc) will need (PT: any parameter
// block with the GEMM's N, M and ep)
template <int EP, typename PT, int NC = 16>
__device__ __forceinline__ void epilogue_prefetch(const PT &p, const Smem &sm, int t, int r, int c0, int nc,
                                                  EpPre &pre) {
  const EpArgs &ep = p.ep;
  const int n = t * BM + r, ncol = min(c0 + nc, p.M) - c0;
  if constexpr (EP == EP_RESID) {
#pragma unroll
    for (int j = 0; j < NC; ++j)
      pre.x[j] = (n < p.N && j < ncol) ? __ldcg(ep.out_f32 + (size_t)(c0 + j) * ep.ldo + n) : 0.f;
    pre.gain = (ep.out_xn != nullptr && n < p.N) ? ep.out_gain[n] : 0.f;
  } else if constexpr (EP == EP_QKV) {
    const QkvOut &o = ep.qkv;
    pre.gn = t < o.nq + o.hkv ? (t < o.nq ? o.qn : o.kn)[r] : 0.f;
    if (t < o.nq + o.hkv && r < 64) {
#pragma unroll
      for (int j = 0; j < NC; ++j)
        pre.cs[j] = j < ncol ? o.rope[(size_t)sm.qkv_pos[c0 + j] * (BM / 2) + r] : make_float2(0.f, 0.f);
    }
  }
}

// epilogue on token columns c0 .. c0+nc-1 (nc <= NC <= 16) of tile t; v[j] = D[row r][c0+j].
// Every argument a loop needs is read into a register before the first store
// (a store through a generic pointer could alias the parameter block, which
// would make the compiler re-read it after each store).
template <int EP, typename PT, int NC = 16>
__device__ __forceinline__ void epilogue_chunk(const PT &p, Smem &sm, int t, int r, int sub, int lane, int c0,
                                               int nc, float *v, const EpPre &pre) {
  static_assert(NC >= 1 && NC <= 16, "chunk width");
  const int n = t * BM + r;
  const EpArgs &ep = p.ep;
  const int cend = min(c0 + nc, p.M);
  if (ep.in_ss) {
#pragma unroll
    for (int j = 0; j < NC; ++j) v[j] *= sm.col_scale[min(c0 + j, MAX_COLS - 1)];
  }
  if constexpr (EP == EP_STORE_F32 || EP == EP_SILU) {
    if (n < p.N) {
      float *const out_f32 = ep.out_f32 + n;
      bf16 *const out_t = reinterpret_cast<bf16 *>(ep.out_t) + n;
      const size_t ldo = ep.ldo, ldt = ep.ldt;
#pragma unroll
      for (int j = 0; j < NC; ++j) {
        const int col = c0 + j;
        if (col < cend) {
          if constexpr (EP == EP_STORE_F32) out_f32[(size_t)col * ldo] = v[j];
          if constexpr (EP == EP_SILU) out_t[(size_t)col * ldt] = __float2bfloat16_rn(silu_fast(v[j]));
        }
      }
    }
  } else if constexpr (EP == EP_RESID) {
    // arguments in registers before the first store (a store could alias them)
    float *const out_f32 = ep.out_f32 + n;
    bf16 *const out_xn = ep.out_xn ? reinterpret_cast<bf16 *>(ep.out_xn) + n : nullptr;
    bf16 *const out_stash = ep.out_stash ? reinterpret_cast<bf16 *>(ep.out_stash) + n : nullptr;
    float *const out_ss = ep.out_ss;
    const size_t ldo = ep.ldo, ld_xn = ep.ld_xn, ld_stash = ep.ld_stash;
    const int ld_ss = ep.ld_ss;
    float x[16];
    const bool row_ok = n < p.N, has_xn = out_xn != nullptr, has_stash = out_stash != nullptr;
#pragma unroll
    for (int j = NC; j < 16; ++j) x[j] = 0.f;
#pragma unroll
    for (int j = 0; j < NC; ++j) {
      const int col = c0 + j;
      x[j] = pre.x[j] + v[j];
      if (row_ok && col < cend) {
        out_f32[(size_t)col * ldo] = x[j];
        if (has_xn) out_xn[(size_t)col * ld_xn] = __float2bfloat16_rn(x[j] * pre.gain);
        if (has_stash) out_stash[(size_t)col * ld_stash] = __float2bfloat16_rn(x[j]);
      } else {
        x[j] = 0.f;
      }
    }
    if (out_ss) {
      // squared-norm partial of this tile's 128 features; thread r < 16 owns column c0 + r
#pragma unroll
      for (int j = 0; j < NC; ++j) x[j] *= x[j];
      const float d = warp_column_sums16(x, lane);
      if (!(lane & 1)) sm.ssred[sub][(lane >> 1) & 15] = d;
      epi_bar();
      if (r < 16 && c0 + r < cend)
        out_ss[(size_t)t * ld_ss + c0 + r] = sm.ssred[0][r] + sm.ssred[1][r] + sm.ssred[2][r] + sm.ssred[3][r];
      epi_bar();
    }
  } else if constexpr (EP == EP_QKV) {
    // arguments in registers before the first store (a store could alias them)
    const QkvOut &o = ep.qkv;
    const int head = t, nq = o.nq, hkv = o.hkv, row0 = o.row0;
    const int kind = head < nq ? 0 : (head < nq + hkv ? 1 : 2);  // q, k, v
    const int kvh = kind == 1 ? head - nq : head - nq - hkv;
    // the head's 128 values of token column c go to dst0 + off(c): q rows, the
    // drafter's block K/V, or the column's slot in the paged pool (off < 0: none)
    const bool paged = kind != 0 && o.bk == nullptr;
    const long long rstride = kind == 0 ? (long long)o.hq_row * BM : (long long)hkv * BM;
    bf16 *const dst0 = kind == 0 ? static_cast<bf16 *>(o.q_out) + (size_t)head * BM
                       : !paged  ? static_cast<bf16 *>(kind == 1 ? o.bk : o.bv) + (size_t)kvh * BM
                                 : static_cast<bf16 *>(o.pool) + (size_t)((kind == 1 ? 0 : hkv) + kvh) * o.page_size * BM;
    const float eps = o.eps;
    // the chunk's bf16 results, [16 columns][128 dims], in the exchange area
    bf16 *const stage = reinterpret_cast<bf16 *>(&sm.xch[0][0]);
    if (kind != 2) {
      // per-head RMSNorm over the 128 rows of the column, then rotary on pairs (r, r + 64)
      float sq[16], tot[16], y[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) sq[j] = j < NC ? v[j] * v[j] : 0.f;
      column_sums(sm, sub, lane, sq, tot);
      const float gn = pre.gn;
#pragma unroll
      for (int j = 0; j < NC; ++j) y[j] = v[j] * rsqrtf(tot[j] * (1.0f / BM) + eps) * gn;
      if (r >= 64) {
#pragma unroll
        for (int j = 0; j < NC; ++j) sm.xch[j][r - 64] = y[j];
      }
      epi_bar();
      uint32_t lohi[16];  // bf16 pair (dim r, dim r + 64)
      if (r < 64) {
#pragma unroll
        for (int j = 0; j < NC; ++j) {
          const float2 cs = pre.cs[j];
          const float x1 = y[j], x2 = sm.xch[j][r];
          const __nv_bfloat162 b2 = __floats2bfloat162_rn(x1 * cs.x - x2 * cs.y, x2 * cs.x + x1 * cs.y);
          lohi[j] = *reinterpret_cast<const uint32_t *>(&b2);
        }
      }
      epi_bar();  // every read of the exchange area is done before it becomes the staging tile
      if (r < 64) {
#pragma unroll
        for (int j = 0; j < NC; ++j) {
          const __nv_bfloat162 b2 = *reinterpret_cast<const __nv_bfloat162 *>(&lohi[j]);
          stage[j * BM + r] = b2.x;
          stage[j * BM + r + 64] = b2.y;
        }
      }
    } else {
#pragma unroll
      for (int j = 0; j < NC; ++j) stage[j * BM + r] = __float2bfloat16_rn(v[j]);
    }
    epi_bar();
    // 16-byte stores: vector e holds dims 8 (e % 16) .. of column c0 + e / 16
    const int nv = (cend - c0) * 16;
    for (int e = r; e < nv; e += BM) {
      const int jc = e >> 4, part = e & 15, col = c0 + jc;
      const long long off = paged ? sm.qkv_base[col] : (long long)(row0 + col) * rstride;
      if (off >= 0)
        *reinterpret_cast<uint4 *>(dst0 + off + part * 8) = *reinterpret_cast<const uint4 *>(stage + jc * BM + part * 8);
    }
    epi_bar();  // the staging tile is rewritten by the next chunk
  } else if constexpr (EP == EP_SWIGLU) {
    // rows 0..63 of the tile are gate features 64t.., rows 64..127 the matching up features
    bf16 *const out_t = reinterpret_cast<bf16 *>(ep.out_t) + t * 64 + r;
    const size_t ldt = ep.ldt;
    if (r >= 64) {
#pragma unroll
      for (int j = 0; j < NC; ++j) sm.xch[j][r - 64] = v[j];
    }
    epi_bar();
    if (r < 64 && t * BM + 64 + r < p.N) {
      float up[NC];
#pragma unroll
      for (int j = 0; j < NC; ++j) up[j] = sm.xch[j][r];
#pragma unroll
      for (int j = 0; j < NC; ++j) {
        const int col = c0 + j;
        if (col < cend) out_t[(size_t)col * ldt] = __float2bfloat16_rn(silu_fast(v[j]) * up[j]);
      }
    }
    epi_bar();
  } else if constexpr (EP == EP_ARGMAX) {
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float bv = n < p.N ? v[j] : -INFINITY;
      int bi = n < p.N ? n : 0x7fffffff;
      warp_argmax(bv, bi);
      if (lane == 0) {
        sm.rv[sub][j] = bv;
        sm.ri[sub][j] = bi;
      }
    }
    epi_bar();
    if (sub == 0 && lane < 16) {
      float bv = sm.rv[0][lane];
      int bi = sm.ri[0][lane];
#pragma unroll
      for (int s = 1; s < 4; ++s) argmax_merge(bv, bi, sm.rv[s][lane], sm.ri[s][lane]);
      const int col = c0 + lane;
      float *const part_val = ep.part_val;
      int *const part_idx = ep.part_idx;
      const size_t n_tiles = ep.n_tiles;
      if (col < cend) {
        part_val[(size_t)col * n_tiles + t] = bv;
        part_idx[(size_t)col * n_tiles + t] = bi;
      }
    }
    epi_bar();
  }
}

// 16 bytes into a peer CTA's shared memory, counted on the peer's barrier
__device__ __forceinline__ void st_async_f4(uint32_t caddr, const float4 &v, uint32_t cbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(caddr),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(cbar)
               : "memory");
}
// split-K: token columns [s0, s1) of rank `rank` out of P (4-column groups)
__host__ __device__ __forceinline__ int splitk_w4(int M, int P) { return ((M + 4 * P - 1) / (4 * P)) * 4; }
// bytes the owner of [s0, s1) receives per tile: a float4 per row and column group from each peer
__host__ __device__ __forceinline__ uint32_t splitk_recv_bytes(int P, int s0, int s1) {
  return s1 > s0 ? (uint32_t)((P - 1) * BM * ((s1 - s0 + 3) / 4) * 16) : 0u;
}

// A cluster's part of a tile that several clusters share: the tile's part slots
// ([parts][BM][npad] fp32, slot `part` this cluster's), the arrival count of
// this CTA's columns, and the number of parts.
struct LeftPart {
  float *acc = nullptr;
  unsigned int *ctr = nullptr;
  unsigned int parts = 0;
  int part = 0;
  bool first = false;  // the group's first part: counts the tile for an owner without columns
};
__device__ __forceinline__ unsigned int atom_add_acq_rel(unsigned int *a, unsigned int v) {
  unsigned int old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
  return old;
}

// One tile of a P-way split-K GEMM (P > 1) done by the P CTAs at cluster ranks
// rbase .. rbase + P - 1 (this CTA is the rr-th).  Every one holds a partial of
// the whole [128 x M] tile; the rr-th finishes token columns [s0, s1).
// Each thread pushes its row's partial, 4-column group by group, into the
// receive area of the group's owner (st.async, counted on the owner's recv
// barrier; its own groups locally), frees the TMEM buffer, then waits for its
// own recv barrier alone, sums the P partials in rank order (deterministic) and
// runs the fused epilogue.  It re-arms recv with next_bytes (what its next
// split-K tile will receive) before telling the senders (rfree, rfree_n
// arrivals each) that they may push again.  False when a wait expired.
// CW4 > 0: the split is 4-way over npad = 4 CW4 columns (each owner finishes
// CW4 of them), known at compile time: every loop has a fixed trip count, the
// owner of a column group is a constant, and the epilogue covers CW4 columns.
// lp.acc set (0 < CW4 <= 16 only): the cluster holds one part of the tile; each owner
// stores its columns' sum in its part's slot, and only the one completing the
// count adds the parts (in part order, so the result does not depend on the
// arrival order) and runs their epilogue (sm.left_last = 1 in that CTA).
template <int EP, typename PT, int CW4 = 0>
__device__ __forceinline__ bool splitk_tile(const PT &g, Smem &sm, float *rx, int P_, int npad_, int M,
                                            uint32_t lane_addr, int i, int t, int r, int sub, int lane, int rr,
                                            int rbase, bool leader, uint32_t next_bytes, uint32_t rfree_n,
                                            const LeftPart lp = LeftPart{}) {
  static_assert(CW4 % 4 == 0 && CW4 <= 32, "owner width");
  constexpr int NC = CW4 > 0 && CW4 < 16 ? CW4 : 16;  // epilogue columns per chunk
  const int P = CW4 ? 4 : P_, npad = CW4 ? 4 * CW4 : npad_;
  const int w4 = CW4 ? CW4 : splitk_w4(M, P);
  const int s0 = min(rr * w4, M), s1 = min((rr + 1) * w4, M);
  const int buf = i & 1;
  EpPre pre;
  epilogue_prefetch<EP, PT, NC>(g, sm, t, r, s0, min(NC, s1 - s0), pre);
  if (leader) {
    int ok = mbar_wait(&sm.accf[buf], (i >> 1) & 1) ? 1 : 0;
    if (ok && i > 0) ok = mbar_wait_cluster(&sm.rfree, (i - 1) & 1) ? 1 : 0;
    sm.flag = ok;
  }
  __syncwarp();
  epi_bar();
  if (!sm.flag) return false;
  tc_fence_after();
  const uint32_t acc_addr = lane_addr + buf * npad;
  const uint32_t rx_s = smem_u32(rx), recv_s = smem_u32(&sm.recv);
  float v[16];
  // the row's partial of columns c0 .. c0 + 15, pushed group by group to the groups' owners
  auto push16 = [&](int c0) {
    tmem_ld16(acc_addr + c0, v);
#pragma unroll
    for (int q4 = 0; q4 < 4; ++q4) {
      const int col = c0 + 4 * q4;
      if (col >= M) break;
      const int owner = col / w4;
      const int e = (rr * BM + r) * w4 + (col - owner * w4);  // the sender's slot in the owner's area
      const float4 x = make_float4(v[4 * q4], v[4 * q4 + 1], v[4 * q4 + 2], v[4 * q4 + 3]);
      if (owner == rr)
        *reinterpret_cast<float4 *>(rx + e) = x;
      else
        st_async_f4(mapa(rx_s + (uint32_t)e * 4, (uint32_t)(rbase + owner)), x, mapa(recv_s, (uint32_t)(rbase + owner)));
    }
  };
  if constexpr (CW4 > 0) {
#pragma unroll
    for (int c0 = 0; c0 < 4 * CW4; c0 += 16)
      if (c0 < M) push16(c0);
  } else {
    for (int c0 = 0; c0 < npad && c0 < M; c0 += 16) push16(c0);
  }
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(&sm.acce[buf]);
  if (leader) sm.flag = mbar_wait(&sm.recv, i & 1) ? 1 : 0;
  __syncwarp();
  epi_bar();
  const bool ok = sm.flag != 0;
  // a shared tile counts once per column owner: for an owner without columns, in its first part
  if (leader) sm.left_last = (lp.acc != nullptr && s0 >= s1 && lp.first) ? 1 : 0;
  // re-arm recv for the next tile, then let the senders push again; done right
  // after the last read of the receive area, before the epilogue's global
  // stores (which a release arrive issued after them would wait for)
  auto release = [&]() {
    epi_bar();  // every thread has read the receive area
    if (leader) {
      mbar_expect_tx(&sm.recv, next_bytes);
#pragma unroll 1
      for (int pr = 0; pr < P; ++pr)
        if (pr != rr) mbar_arrive_remote_relaxed(&sm.rfree, (uint32_t)(rbase + pr), rfree_n);
    }
  };
  bool released = false;
  if (ok) {
    for (int c0 = s0; c0 < s1; c0 += 16) {
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = 0.f;
      // the P partials of the row, in rank order
      auto add_partial = [&](int sp) {
        const float *src = rx + (sp * BM + r) * w4 + (c0 - s0);
#pragma unroll
        for (int q4 = 0; q4 < NC / 4; ++q4) {
          if (c0 + 4 * q4 >= s1) break;
          const float4 y = *reinterpret_cast<const float4 *>(src + 4 * q4);
          v[4 * q4] += y.x;
          v[4 * q4 + 1] += y.y;
          v[4 * q4 + 2] += y.z;
          v[4 * q4 + 3] += y.w;
        }
      };
      if constexpr (CW4 > 0) {
#pragma unroll
        for (int sp = 0; sp < 4; ++sp) add_partial(sp);
      } else {
        for (int sp = 0; sp < P; ++sp) add_partial(sp);
      }
      if (c0 + 16 >= s1) {
        release();
        released = true;
      }
      if (c0 > s0) epilogue_prefetch<EP, PT, NC>(g, sm, t, r, c0, min(NC, s1 - c0), pre);
      if constexpr (CW4 > 0 && CW4 <= 16) {
        if (lp.acc != nullptr) {
          // one chunk (CW4 <= 16): this cluster's part of the columns into its slot
          const size_t slot = (size_t)BM * npad;
          float *const a = lp.acc + (size_t)r * npad + c0;
#pragma unroll
          for (int q4 = 0; q4 < NC / 4; ++q4)
            if (c0 + 4 * q4 < s1)
              __stcg(reinterpret_cast<float4 *>(a + lp.part * slot + 4 * q4),
                     make_float4(v[4 * q4], v[4 * q4 + 1], v[4 * q4 + 2], v[4 * q4 + 3]));
          // the leader's count is a release at GPU scope that follows every thread's
          // additions through the barrier (the pattern of a block-wide result
          // published by one thread), and an acquire for the last part's reads
          epi_bar();
          if (leader) sm.left_last = atom_add_acq_rel(lp.ctr, 1u) == lp.parts - 1 ? 1 : 0;
          epi_bar();
          if (!sm.left_last) continue;
          // every part is in (the leader's acquire, ordered before these reads by the
          // barrier): their sum in part order; the count is left at zero
#pragma unroll
          for (int q4 = 0; q4 < NC / 4; ++q4) {
            if (c0 + 4 * q4 >= s1) break;
            float4 x = __ldcg(reinterpret_cast<const float4 *>(a + 4 * q4));
            for (int pp = 1; pp < (int)lp.parts; ++pp) {
              const float4 y = __ldcg(reinterpret_cast<const float4 *>(a + pp * slot + 4 * q4));
              x.x += y.x;
              x.y += y.y;
              x.z += y.z;
              x.w += y.w;
            }
            v[4 * q4] = x.x;
            v[4 * q4 + 1] = x.y;
            v[4 * q4 + 2] = x.z;
            v[4 * q4 + 3] = x.w;
          }
          if (leader) *reinterpret_cast<volatile unsigned int *>(lp.ctr) = 0u;
        }
      }
      epilogue_chunk<EP, PT, NC>(g, sm, t, r, sub, lane, c0, min(NC, s1 - c0), v, pre);
    }
  }
  if (!released) release();
  return ok;
}

template <int EP>
__global__ void __launch_bounds__(THREADS, 1)
k_gemm_tc(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, const Params p) {
  // the next kernel may launch once every CTA of this one runs; inputs produced by
  // the previous launch are read only after dep_wait() (weights are prefetched before it)
  pdl_trigger();
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(dsm) + 1023) & ~(uintptr_t)1023);
  const int stage_bytes = A_BYTES + p.npad * BK * 2;
  float *rx = reinterpret_cast<float *>(ring + (size_t)p.stages * stage_bytes);  // [P][BM][w4] split-K receive area
  Smem &sm = *reinterpret_cast<Smem *>(reinterpret_cast<uint8_t *>(rx) + p.rx_bytes);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int rank = p.P > 1 ? (int)cluster_rank() : 0;
  const int q = blockIdx.x / p.P;
  const int kr0 = rank * p.kb / p.P, kr1 = (rank + 1) * p.kb / p.P;

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.accf[b], 1);
      mbar_init(&sm.acce[b], 4);
    }
    mbar_init(&sm.recv, 1);
    mbar_init(&sm.rfree, p.P > 1 ? p.P - 1 : 1);
    mbar_init(&sm.drain, 1);
    sm.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (p.P > 1) {
      // armed for the first tile before the cluster barrier below lets any peer push
      const int w4 = splitk_w4(p.M, p.P);
      mbar_expect_tx(&sm.recv, splitk_recv_bytes(p.P, min(rank * w4, p.M), min((rank + 1) * w4, p.M)));
    }
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&sm.tmem)),
                 "r"(p.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  if (p.P > 1) cluster_sync();  // peers' barriers are initialised before anyone signals them
  tc_fence_after();
  const uint32_t tmem = sm.tmem;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint64_t pw = policy_evict_first(), px = policy_evict_last();
      int stage = 0;
      uint32_t ph = 0;
      int n_issued = 0;  // (tile, k-block) units whose copies were started, in ring order
      bool ok = true;
      const int nk = kr1 - kr0;
      const int n_units = ((p.T - q + p.Q - 1) / p.Q) * nk;  // (tile, k-block) pairs of this CTA, in order
      // weight tiles of the first ring do not depend on the previous kernel: start them now
      const int pre = n_units < p.stages ? n_units : p.stages;
      for (int u = 0; u < pre; ++u) {
        mbar_expect_tx(&sm.full[u], stage_bytes);
        tma_load_2d(ring + (size_t)u * stage_bytes, &tmW, (kr0 + u % nk) * BK, (q + (u / nk) * p.Q) * BM, &sm.full[u], pw);
      }
      n_issued = pre;
      dep_wait(p.dep, p.status);
      if (p.dep.wait) fence_proxy_async_global();
      for (int u = 0; u < pre; ++u)
        tma_load_2d(ring + (size_t)u * stage_bytes + A_BYTES, &tmX, (kr0 + u % nk) * BK, 0, &sm.full[u], px);
      stage = pre % p.stages;
      ph = pre == p.stages ? 1 : 0;
      for (int u = pre; u < n_units; ++u) {
        const int t = q + (u / nk) * p.Q, k = kr0 + u % nk;
        if (!mbar_wait(&sm.empty[stage], ph ^ 1) || *(volatile int *)&sm.abort) {
          ok = false;
          break;
        }
        uint8_t *a = ring + (size_t)stage * stage_bytes;
        mbar_expect_tx(&sm.full[stage], stage_bytes);
        tma_load_2d(a, &tmW, k * BK, t * BM, &sm.full[stage], pw);
        tma_load_2d(a + A_BYTES, &tmX, k * BK, 0, &sm.full[stage], px);
        n_issued = u + 1;
        if (++stage == p.stages) {
          stage = 0;
          ph ^= 1;
        }
      }
      if (!ok) {
        set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
        atomicExch(&sm.abort, 1);
      }
      // every copy this thread started has landed before the CTA may exit: the
      // last fill of each stage is one of the last `stages` units
      for (int u = n_issued > p.stages ? n_issued - p.stages : 0; u < n_issued; ++u)
        if (!mbar_wait(&sm.full[u % p.stages], (uint32_t)((u / p.stages) & 1)))
          set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      bool ok = true;
      int i = 0;
      for (int t = q; t < p.T && ok; t += p.Q, ++i) {
        const int buf = i & 1;
        if (!mbar_wait(&sm.acce[buf], ((i >> 1) & 1) ^ 1)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem + buf * p.npad;
        for (int k = kr0; k < kr1; ++k) {
          if (!mbar_wait(&sm.full[stage], ph) || *(volatile int *)&sm.abort) { ok = false; break; }
          tc_fence_after();
          const uint32_t a = smem_u32(ring + (size_t)stage * stage_bytes);
          const uint64_t ad = smem_desc(a), bd = smem_desc(a + A_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            mma_bf16(d, ad + 2 * kk, bd + 2 * kk, p.idesc, (k > kr0 || kk > 0) ? 1u : 0u);
          mma_commit(&sm.empty[stage]);
          if (++stage == p.stages) {
            stage = 0;
            ph ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(&sm.accf[buf]);
      }
      if (!ok) {
        set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
        atomicExch(&sm.abort, 1);
      }
      // all MMAs of this thread complete before TMEM is released
      mma_commit(&sm.drain);
      if (!mbar_wait(&sm.drain, 0)) set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
  } else {
    // ---------------- epilogue warps 2..5 ----------------
    const int sub = warp & 3;  // TMEM sub-partition this warp may read
    const int r = sub * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(sub * 32) << 16);
    const bool leader = threadIdx.x == 64;
    if (leader) dep_wait(p.dep, p.status);
    epi_bar();  // the other epilogue threads read the previous launch's outputs after the leader's wait
    if (p.ep.in_ss) col_scales(p.ep, sm, p.M, r);
    if constexpr (EP == EP_QKV) {
      // per token column: position, and the paged-pool slot its K/V rows go to
      qkv_table(p.ep.qkv, sm, p.M, r);
      epi_bar();
    }
    int i = 0;
    for (int t = q; t < p.T; t += p.Q, ++i) {
      const int buf = i & 1;
      if (p.P == 1) {
        EpPre pre;
        epilogue_prefetch<EP>(p, sm, t, r, 0, 16, pre);
        if (leader) sm.flag = mbar_wait(&sm.accf[buf], (i >> 1) & 1) ? 1 : 0;
        __syncwarp();
        epi_bar();
        if (!sm.flag) {
          if (leader) {
            set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
            atomicExch(&sm.abort, 1);
          }
          break;
        }
        tc_fence_after();
        const uint32_t acc_addr = lane_addr + buf * p.npad;
        float v[16];
        for (int c0 = 0; c0 < p.npad && c0 < p.M; c0 += 16) {
          if (c0 > 0) epilogue_prefetch<EP>(p, sm, t, r, c0, 16, pre);
          tmem_ld16(acc_addr + c0, v);
          epilogue_chunk<EP>(p, sm, t, r, sub, lane, c0, 16, v, pre);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.acce[buf]);
      } else {
        const int w4 = splitk_w4(p.M, p.P);
        const uint32_t nb = splitk_recv_bytes(p.P, min(rank * w4, p.M), min((rank + 1) * w4, p.M));
        if (!splitk_tile<EP>(p, sm, rx, p.P, p.npad, p.M, lane_addr, i, t, r, sub, lane, rank, 0, leader, nb, 1u)) {
          if (leader) {
            set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
            atomicExch(&sm.abort, 1);
          }
          break;
        }
      }
      epi_bar();  // sm.flag is rewritten by the leader at the top of the next tile
    }
  }

  __syncwarp();  // lanes that skipped a single-thread role wait for it here
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) dep_signal(p.dep);  // every global write of this CTA is done
  if (p.P > 1) cluster_sync();  // no CTA leaves while a peer may still read its shared memory
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(p.tmem_cols) : "memory");
  }
}

// ===========================================================================
// Wide weight-streaming GEMM: up to 512 token rows in one pass over the weights
// (two MMAs per k-step once the padded rows exceed one MMA's N of 256), for the
// blocks of large batches.  The grid is Q tile groups x P k-splits of CTAs:
// CTA (q, r) takes tiles q, q + Q, ... over k-blocks [r kb / P, (r + 1) kb / P)
// (or, with leftovers, whole tiles and then one k part of a leftover tile; see
// wide_item).  A tile split over several CTAs is reduced by all of them: each
// stores its fp32 partial in an L2 slot and counts it, waits until the tile's
// parts are all in (the grid is at most one CTA per SM, so they are resident
// together), adds the slots in part order (so the result does not depend on the
// arrival order) for its share of the token columns and runs the fused epilogue
// on them; a second count lets the last one leave the counter at zero.
// ===========================================================================
constexpr int WIDE_MAX_NPAD = 512;
constexpr int WIDE_MAX_TILES = 4096;                    // 128-row tiles of one projection (N <= 524288)
constexpr size_t WIDE_SLOT_BYTES = (size_t)48 << 20;   // split-K partials, kept well inside L2

struct WideParams {
  int N, K, M, npad, T, kb, P, Q, stages, tmem_cols, nbuf;
  int Tl, ls;               // leftover tiles and the parts each is split into (P = 1 only; Tl = 0: none)
  uint32_t idesc1, idesc2;  // MMA N = min(npad, 256), and npad - 256
  EpArgs ep;
  int *status;
  Dep dep;
  float *slots;       // partials of the split tiles: [T][P][BM][npad], or [Tl][ls][BM][npad] for the leftovers
  unsigned int *ctr;  // [T] arrivals per tile (zero between uses)
};

// The tiles ("items") of CTA c of the one-pass GEMM, in order.  Without
// leftovers, CTA c = q P + rank takes tiles q, q + Q, ..., each over the k range
// `rank` of P.  With leftovers (P = 1), CTA c takes tiles c, c + Q, ... below
// Tf = T - Tl whole, then, for c < Tl ls, the k range c % ls of ls of leftover
// tile Tf + c / ls: every CTA streams about the same number of k-blocks.
struct WideItem {
  int t, k0, k1, part, parts;
  int slot;  // index of this part's partial slot (parts > 1)
};
__host__ __device__ __forceinline__ int wide_n_items(const WideParams &p, int c) {
  if (p.Tl == 0) {
    const int q = c / p.P;
    return q < p.T ? (p.T - q + p.Q - 1) / p.Q : 0;
  }
  const int Tf = p.T - p.Tl;
  return (c < Tf ? (Tf - c + p.Q - 1) / p.Q : 0) + (c < p.Tl * p.ls ? 1 : 0);
}
__host__ __device__ __forceinline__ WideItem wide_item(const WideParams &p, int c, int i) {
  WideItem it;
  if (p.Tl == 0) {
    const int q = c / p.P, rank = c % p.P;
    it.t = q + i * p.Q;
    it.part = rank;
    it.parts = p.P;
    it.slot = it.t * p.P + rank;
  } else {
    const int Tf = p.T - p.Tl, nf = c < Tf ? (Tf - c + p.Q - 1) / p.Q : 0;
    if (i < nf) {
      it.t = c + i * p.Q;
      it.part = 0;
      it.parts = 1;
      it.slot = 0;
    } else {
      it.t = Tf + c / p.ls;
      it.part = c % p.ls;
      it.parts = p.ls;
      it.slot = c;
    }
  }
  it.k0 = it.part * p.kb / it.parts;
  it.k1 = (it.part + 1) * p.kb / it.parts;
  return it;
}

template <int EP>
__global__ void __launch_bounds__(THREADS, 1)
k_gemm_wide(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX1,
            const __grid_constant__ CUtensorMap tmX2, const WideParams p) {
  // the next kernel may launch once every CTA of this one runs; inputs produced by
  // the previous launch are read only after dep_wait() (weights are prefetched before it)
  pdl_trigger();
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(dsm) + 1023) & ~(uintptr_t)1023);
  const int stage_bytes = A_BYTES + p.npad * BK * 2;
  Smem &sm = *reinterpret_cast<Smem *>(ring + (size_t)p.stages * stage_bytes);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int cta = (int)blockIdx.x;
  const bool two = p.npad > 256;  // a second MMA (and X box) for rows 256..npad-1

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.accf[b], 1);
      mbar_init(&sm.acce[b], 4);
    }
    mbar_init(&sm.drain, 1);
    mbar_init(&sm.ovf, 4);
    sm.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&sm.tmem)),
                 "r"(p.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem;
  const int n_tiles = wide_n_items(p, cta);  // tiles (whole or a k range) of this CTA
  // accumulator buffers: nbuf 1: one; 2: two side by side; 3: two that share the
  // TMEM columns [512 - npad, npad) (npad > 256): buffer 0 at column 0, buffer 1
  // at 512 - npad.  With 3 the epilogue reads the shared columns first and
  // arrives on ovf, and the next tile's MMAs wait for that instead of the whole
  // epilogue.
  const bool ovl = p.nbuf == 3;
  auto acc_col = [&](int buf) -> uint32_t {
    return buf == 0 ? 0u : (uint32_t)(p.nbuf == 2 ? p.npad : 512 - p.npad);
  };

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint64_t pw = policy_evict_first(), px = policy_evict_last();
      auto load_x = [&](uint8_t *a, int k, uint64_t *bar) {
        tma_load_2d(a + A_BYTES, &tmX1, k * BK, 0, bar, px);
        if (two) tma_load_2d(a + A_BYTES + 256 * 128, &tmX2, k * BK, 256, bar, px);
      };
      // the CTA's (tile, k-block) units in order
      int wi = 0, wk = 0;
      WideItem cur{};
      if (n_tiles > 0) {
        cur = wide_item(p, cta, 0);
        wk = cur.k0;
      }
      auto next_unit = [&](int &t, int &k) -> bool {
        if (wi >= n_tiles) return false;
        t = cur.t;
        k = wk;
        if (++wk >= cur.k1 && ++wi < n_tiles) {
          cur = wide_item(p, cta, wi);
          wk = cur.k0;
        }
        return true;
      };
      int n_issued = 0;
      bool ok = true;
      // weight tiles of the first ring do not depend on the previous kernel: start them now
      int pre_k[16];
      int pre = 0, t = 0, k = 0;
      while (pre < p.stages && next_unit(t, k)) {
        mbar_expect_tx(&sm.full[pre], stage_bytes);
        tma_load_2d(ring + (size_t)pre * stage_bytes, &tmW, k * BK, t * BM, &sm.full[pre], pw);
        pre_k[pre++] = k;
      }
      n_issued = pre;
      dep_wait(p.dep, p.status);
      if (p.dep.wait) fence_proxy_async_global();
      for (int u = 0; u < pre; ++u) load_x(ring + (size_t)u * stage_bytes, pre_k[u], &sm.full[u]);
      int stage = pre % p.stages;
      uint32_t ph = pre == p.stages ? 1 : 0;
      for (int u = pre; next_unit(t, k); ++u) {
        if (!mbar_wait(&sm.empty[stage], ph ^ 1) || *(volatile int *)&sm.abort) {
          ok = false;
          break;
        }
        uint8_t *a = ring + (size_t)stage * stage_bytes;
        mbar_expect_tx(&sm.full[stage], stage_bytes);
        tma_load_2d(a, &tmW, k * BK, t * BM, &sm.full[stage], pw);
        load_x(a, k, &sm.full[stage]);
        n_issued = u + 1;
        if (++stage == p.stages) {
          stage = 0;
          ph ^= 1;
        }
      }
      if (!ok) {
        set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
        atomicExch(&sm.abort, 1);
      }
      // every copy this thread started has landed before the CTA may exit
      for (int u = n_issued > p.stages ? n_issued - p.stages : 0; u < n_issued; ++u)
        if (!mbar_wait(&sm.full[u % p.stages], (uint32_t)((u / p.stages) & 1)))
          set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int i = 0; i < n_tiles && ok; ++i) {
        const int buf = p.nbuf >= 2 ? (i & 1) : 0;
        const uint32_t par = p.nbuf >= 2 ? (uint32_t)((i >> 1) & 1) : (uint32_t)(i & 1);
        if (!mbar_wait(&sm.acce[buf], par ^ 1)) { ok = false; break; }
        // the previous tile's epilogue has read the columns the two buffers share
        if (ovl && i > 0 && !mbar_wait(&sm.ovf, (uint32_t)((i - 1) & 1))) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem + acc_col(buf);
        const WideItem it = wide_item(p, cta, i);
        const int kr0 = it.k0;
        for (int k = it.k0; k < it.k1; ++k) {
          if (!mbar_wait(&sm.full[stage], ph) || *(volatile int *)&sm.abort) { ok = false; break; }
          tc_fence_after();
          const uint32_t a = smem_u32(ring + (size_t)stage * stage_bytes);
          const uint64_t ad = smem_desc(a), bd1 = smem_desc(a + A_BYTES), bd2 = smem_desc(a + A_BYTES + 256 * 128);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint32_t acc = (k > kr0 || kk > 0) ? 1u : 0u;
            mma_bf16(d, ad + 2 * kk, bd1 + 2 * kk, p.idesc1, acc);
            if (two) mma_bf16(d + 256, ad + 2 * kk, bd2 + 2 * kk, p.idesc2, acc);
          }
          mma_commit(&sm.empty[stage]);
          if (++stage == p.stages) {
            stage = 0;
            ph ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(&sm.accf[buf]);
      }
      if (!ok) {
        set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
        atomicExch(&sm.abort, 1);
      }
      mma_commit(&sm.drain);
      if (!mbar_wait(&sm.drain, 0)) set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
  } else {
    // ---------------- epilogue warps 2..5 ----------------
    const int sub = warp & 3;
    const int r = sub * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(sub * 32) << 16);
    const bool leader = threadIdx.x == 64;
    if (leader) dep_wait(p.dep, p.status);
    epi_bar();
    if (p.ep.in_ss) col_scales(p.ep, sm, p.M, r);
    if constexpr (EP == EP_QKV) {
      qkv_table(p.ep.qkv, sm, p.M, r);
      epi_bar();
    }
    const int cols = p.npad < p.M ? p.npad : p.M;
    for (int i = 0; i < n_tiles; ++i) {
      const WideItem it = wide_item(p, cta, i);
      const int t = it.t, rank = it.part, P = it.parts;
      const int buf = p.nbuf >= 2 ? (i & 1) : 0;
      const uint32_t par = p.nbuf >= 2 ? (uint32_t)((i >> 1) & 1) : (uint32_t)(i & 1);
      // 16-column chunks in the order c(0), c(1), ...: with shared columns, the
      // chunks that hold them first (buffer 0: its last ones; buffer 1: its first),
      // then ovf
      const int nch = (cols + 15) / 16;
      const int c_first = ovl && buf == 0 ? (512 - p.npad) / 16 : 0;
      const int rot = c_first < nch ? c_first : 0;
      const int n_shared = !ovl ? -1 : buf == 0 ? (c_first < nch ? nch - c_first : 0)
                                                : min((2 * p.npad - 512 + 15) / 16, nch);
      auto chunk_col = [&](int k) { return 16 * ((rot + k) % nch); };
      auto shared_read = [&](int k) {  // after the k-th chunk in this order (k = -1: before the first)
        if (k + 1 == n_shared) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.ovf);
        }
      };
      EpPre pre;
      if (P == 1) epilogue_prefetch<EP>(p, sm, t, r, chunk_col(0), 16, pre);
      if (leader) sm.flag = mbar_wait(&sm.accf[buf], par) ? 1 : 0;
      __syncwarp();
      epi_bar();
      if (!sm.flag) {
        if (leader) {
          set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
          atomicExch(&sm.abort, 1);
        }
        break;
      }
      tc_fence_after();
      const uint32_t acc_addr = lane_addr + acc_col(buf);
      float v[16];
      shared_read(-1);
      if (P == 1) {
        for (int k = 0; k < nch; ++k) {
          const int c0 = chunk_col(k);
          if (k > 0) epilogue_prefetch<EP>(p, sm, t, r, c0, 16, pre);
          tmem_ld16(acc_addr + c0, v);
          epilogue_chunk<EP>(p, sm, t, r, sub, lane, c0, 16, v, pre);
          shared_read(k);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.acce[buf]);
      } else {
        // this CTA's partial of row r into its slot, then free the accumulator
        // a slot is [npad / 16 column chunks][BM rows][16]: a warp's stores of one
        // chunk are one contiguous 2 KB run
        float *const mine = p.slots + (size_t)it.slot * BM * p.npad + (size_t)r * 16;
        for (int k = 0; k < nch; ++k) {
          const int c0 = chunk_col(k);
          tmem_ld16(acc_addr + c0, v);
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4)
            __stcg(reinterpret_cast<float4 *>(mine + (size_t)c0 * BM + 4 * q4),
                   make_float4(v[4 * q4], v[4 * q4 + 1], v[4 * q4 + 2], v[4 * q4 + 3]));
          shared_read(k);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.acce[buf]);
        // The leader's count is a release at GPU scope after every thread's stores
        // (through the barrier); its wait for all P counts an acquire for every
        // thread's reads after the next barrier.  The P CTAs of the tile are all
        // resident (grid <= SMs, one CTA per SM, and no later launch starts before
        // every CTA of this one has), so the wait ends; it is bounded all the same.
        epi_bar();
        if (leader) {
          atom_add_acq_rel(p.ctr + t, 1u);
          int ok = 1;
          const unsigned long long t0 = gtime();
          for (int it = 0;; ++it) {
            unsigned int v;
            asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p.ctr + t) : "memory");
            if (v >= (unsigned)P) break;
            if ((it & 15) == 15 && gtime() - t0 > WAIT_NS) {
              ok = 0;
              break;
            }
          }
          sm.flag = ok;
        }
        epi_bar();
        if (!sm.flag) {
          if (leader) {
            set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
            atomicExch(&sm.abort, 1);
          }
          break;
        }
        // this CTA's share of the token columns: chunks [rank nch / P, (rank + 1) nch / P)
        {
          const float *const row0 = p.slots + (size_t)(it.slot - rank) * BM * p.npad + (size_t)r * 16;
          const size_t rstride = (size_t)BM * p.npad;  // one rank's slot
          const int k0 = rank * nch / P, k1 = (rank + 1) * nch / P;
          for (int k = k0; k < k1; ++k) {
            const int c0 = 16 * k;
            epilogue_prefetch<EP>(p, sm, t, r, c0, 16, pre);
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] = 0.f;
            for (int rr = 0; rr < P; ++rr) {
#pragma unroll
              for (int q4 = 0; q4 < 4; ++q4) {
                const float4 y = __ldcg(reinterpret_cast<const float4 *>(row0 + rr * rstride + (size_t)c0 * BM + 4 * q4));
                v[4 * q4] += y.x;
                v[4 * q4 + 1] += y.y;
                v[4 * q4 + 2] += y.z;
                v[4 * q4 + 3] += y.w;
              }
            }
            epilogue_chunk<EP>(p, sm, t, r, sub, lane, c0, 16, v, pre);
          }
        }
        // every CTA of the tile counts again once its reads are done; the last
        // one leaves the count at zero for the next use
        epi_bar();
        if (leader && atom_add_acq_rel(p.ctr + t, 1u) == (unsigned)(2 * P - 1))
          *reinterpret_cast<volatile unsigned int *>(p.ctr + t) = 0u;
      }
      epi_bar();  // sm.flag is rewritten at the next tile
    }
  }

  __syncwarp();  // lanes that skipped a single-thread role wait for it here
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) dep_signal(p.dep);  // every global write of this CTA is done
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(p.tmem_cols) : "memory");
  }
}

// ===========================================================================
// Persistent sequence of weight-streaming GEMMs: one launch per layer segment
// (O, gate/up, down projections and the next layer's QKV projection).  One
// cluster of SEQ_P CTAs owns 128-row tiles q, q + Q, ... of every GEMM and
// splits their K range as k_gemm_tc does.  The producer streams weight
// k-blocks without a break across the GEMM boundaries; a unit's activation
// k-block is issued once every tile of the previous GEMM is finished (one
// completion counter per GEMM, one release add per CTA and tile), so the next
// GEMM's weights fill the ring while the epilogue warps finish the current
// GEMM.  Every CTA of the grid is resident at once (the grid is sized by the
// cluster occupancy), which the cross-CTA waits rely on.
// ===========================================================================
constexpr int SEQ_MAX = 4;  // GEMMs per launch
constexpr int SEQ_P = 4;    // cluster size = split-K ways of a tile inside a cluster
constexpr int SEQ_LEFT_MAX = 40;  // leftover tiles of one GEMM and part slots (one per cluster; at most 38)

// Tiles 0 .. Tf-1 go to the Q clusters round robin (cluster q: q, q + Q, ...),
// each split 4 ways over the cluster's CTAs and reduced in shared memory.  The
// Tl = T - Tf leftover tiles (T mod Q of them, when Q is a multiple) are each
// split over ls = Q / Tl clusters, 4 ls ways: every CTA then streams the same
// number of weight k-blocks.  A cluster reduces its part of a leftover tile in
// shared memory like any tile; each column owner then stores its columns in
// its cluster's fp32 slot of lacc (L2), and the owner whose arrival completes
// the count of its columns adds the slots in part order, runs their epilogue
// and leaves the count at zero again.
struct SeqGemm {
  int N, K, M, T, kb, mode;
  int q0, Qg;  // clusters q0 .. q0+Qg-1 take this GEMM's tiles (tile stride Qg)
  int Tf, Tl, ls;
  // the per-CTA schedule without runtime divisions: cluster q has nt_a + (q < nt_b)
  // full tiles; x / ls and x / (SEQ_P ls) are umulhi(x, ls_mag), umulhi(x, parts_mag)
  // (exact: every dividend here times its divisor is below 2^32)
  int nt_a, nt_b;
  unsigned int ls_mag, parts_mag;
  uint32_t idesc;
  EpArgs ep;
  unsigned int *done;   // completion counter: each CTA adds 1 per tile whose columns it finished
  unsigned int done_n;  // its value once every tile of this GEMM is finished
  float *lacc;          // [Q][BM][npad] leftover part slots, one per cluster
  unsigned int *lctr;   // [Tl][SEQ_P] leftover contributions per column owner (zero between uses)
};
struct SeqMaps {
  CUtensorMap w[SEQ_MAX], x[SEQ_MAX];  // weights [N][K], activations [M][K]
  CUtensorMap akv, aq;                 // attention phase: one layer of the K/V pool; the query rows (3D)
};
// the attention phase ahead of the first GEMM: units u = (kv head u % hkv,
// sequence u / hkv), unit u on cluster u % n_clusters (its four CTAs are the
// unit's key splits)
struct SeqAttnPhase {
  int on, block, q_tma, n_units, n_clusters;
  Dims D;
  AttnArgs a;
  unsigned int *done;   // each CTA adds 1 per unit it finished
  unsigned int done_n;  // its value once every unit is finished
};
struct SeqParams {
  int n, M, npad, Q, stages, tmem_cols, rx_bytes;
  int independent;  // 1: no GEMM reads another's output; they share the launch's completion counter
  int *status;
  Dep dep;  // the previous launch: inputs of the first GEMM (and of the attention phase)
  SeqAttnPhase att;
  SeqGemm g[SEQ_MAX];
};
constexpr int SEQ_ATT_KVS = 3;  // K/V pages in flight in the attention phase

// bounded wait on a completion counter (acquire); false on expiry.  The counter
// holds exactly n once its GEMM is complete (its slot is not reused in the same
// launch), so a value past n means a miscount: it would have released this wait
// early, and it is recorded in *status.
__device__ __forceinline__ bool counter_wait(const unsigned int *c, unsigned int n, int *status) {
  const unsigned long long t0 = gtime();
  for (int i = 0;; ++i) {
    unsigned int v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(c) : "memory");
    if ((int)(v - n) >= 0) {
      if (v != n) set_status(status, DFLOW_ERR_BAD_STATE);
      return true;
    }
    if ((i & 15) == 15 && gtime() - t0 > WAIT_NS) return false;
  }
}
__device__ __forceinline__ void counter_add(unsigned int *c, unsigned int n) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(c), "r"(n) : "memory");
}

// the tensor maps of GEMM j, addressed with constant offsets into the parameter block
__device__ __forceinline__ const CUtensorMap *seq_wmap(const SeqMaps &m, int j) {
  switch (j) {
    case 0: return &m.w[0];
    case 1: return &m.w[1];
    case 2: return &m.w[2];
    default: return &m.w[3];
  }
}
__device__ __forceinline__ const CUtensorMap *seq_xmap(const SeqMaps &m, int j) {
  switch (j) {
    case 0: return &m.x[0];
    case 1: return &m.x[1];
    case 2: return &m.x[2];
    default: return &m.x[3];
  }
}

// this CTA's tile count, first tile, tile stride, k-block range and split of
// every GEMM, read once from the parameter block with constant indices and kept
// in registers (the unit loops index them through sel4, never with a runtime
// array index)
struct SeqTab {
  int n, nt[SEQ_MAX], t0[SEQ_MAX], dt[SEQ_MAX], k0[SEQ_MAX], k1[SEQ_MAX];
  int lt[SEQ_MAX], lk0[SEQ_MAX], lk1[SEQ_MAX];  // leftover tile (index among the leftovers, or -1) and k range
  int lpart[SEQ_MAX];                           // the cluster's part index in its leftover tile
};
__device__ __forceinline__ int sel4(const int (&a)[SEQ_MAX], int j) {
  return j == 0 ? a[0] : j == 1 ? a[1] : j == 2 ? a[2] : a[3];
}
// high 32 bits of a 32 x 32-bit product (the schedule's divisions by runtime values)
__host__ __device__ __forceinline__ unsigned int umulhi32(unsigned int a, unsigned int b) {
#ifdef __CUDA_ARCH__
  return __umulhi(a, b);
#else
  return (unsigned int)(((unsigned long long)a * b) >> 32);
#endif
}
__host__ __device__ __forceinline__ int imin(int a, int b) { return a < b ? a : b; }
// cta: this CTA's index in the grid (clusters are SEQ_P consecutive CTAs).  Also
// evaluated on the host, where a test checks the schedule for every shape.
__host__ __device__ __forceinline__ SeqTab seq_tab(const SeqParams &p, int cta) {
  SeqTab t;
  t.n = p.n;
  const int q = cta / SEQ_P, rr = cta % SEQ_P;  // cluster, rank in the cluster
#pragma unroll
  for (int j = 0; j < SEQ_MAX; ++j) {
    const SeqGemm &g = p.g[j];
    const int qj = q - (j < p.n ? g.q0 : 0);  // the cluster's index among the GEMM's clusters
    const bool on = j < p.n && qj >= 0 && qj < g.Qg;
    const int kb = on ? g.kb : 0;
    t.t0[j] = on ? qj : 0;
    t.dt[j] = on ? g.Qg : 1;
    t.nt[j] = on ? g.nt_a + (qj < g.nt_b ? 1 : 0) : 0;
    t.k0[j] = rr * kb / SEQ_P;
    t.k1[j] = (rr + 1) * kb / SEQ_P;
    const bool left = on && qj < g.Tl * g.ls;
    const int lt = left ? (int)umulhi32((unsigned)qj, g.ls_mag) : 0;
    const int m = (qj - lt * g.ls) * SEQ_P + rr;  // this CTA's part of its leftover tile
    t.lt[j] = left ? lt : -1;
    t.lpart[j] = left ? qj - lt * g.ls : 0;
    t.lk0[j] = left ? (int)umulhi32((unsigned)(m * kb), g.parts_mag) : 0;
    t.lk1[j] = left ? (int)umulhi32((unsigned)((m + 1) * kb), g.parts_mag) : 0;
  }
  return t;
}
// bytes this CTA receives in a split-K tile of GEMM j
__host__ __device__ __forceinline__ uint32_t seq_recv_bytes(int M, int npad, int rank) {
  const int w4 = npad / SEQ_P;
  return splitk_recv_bytes(SEQ_P, imin(rank * w4, M), imin((rank + 1) * w4, M));
}
// true when this CTA has another tile after tile ti of GEMM j (ti = -1: its leftover part)
__device__ __forceinline__ bool seq_more(const SeqTab &tb, int j, int ti) {
  if (ti + 1 < sel4(tb.nt, j)) return true;
  for (++j; j < tb.n; ++j)
    if (sel4(tb.nt, j) > 0 || sel4(tb.lt, j) >= 0) return true;
  return false;
}

// one tile of GEMM g (split-K over the SEQ_P CTAs of the cluster, NPAD token
// columns); false when a bounded wait expired.  rfree counts SEQ_P - 1
// arrivals per tile, one from each other owner.
// lt >= 0: t is leftover tile lt, the cluster holds one part of it (the host
// splits tiles over clusters only for NPAD <= MAX_SPLIT_NPAD: one epilogue chunk
// per owner).
template <int EP, int NPAD>
__device__ __forceinline__ bool seq_tile(const SeqGemm &g, Smem &sm, float *rx, uint32_t lane_addr, int i, int t, int lt,
                                         int part, int r, int sub, int lane, int rank, bool leader,
                                         uint32_t next_bytes) {
  static_assert(SEQ_P == 4, "the compile-time split of splitk_tile is 4-way");
  LeftPart lp;
  if (lt >= 0) {
    // slots of clusters lt ls .. lt ls + ls - 1 (one per cluster of the GEMM)
    lp.acc = g.lacc + (size_t)lt * g.ls * BM * NPAD;
    lp.ctr = g.lctr + lt * SEQ_P + rank;
    lp.parts = (unsigned int)g.ls;
    lp.part = part;
    lp.first = part == 0;
  }
  const bool ok = splitk_tile<EP, SeqGemm, NPAD / 4>(g, sm, rx, SEQ_P, NPAD, g.M, lane_addr, i, t, r, sub, lane, rank, 0,
                                                     leader, next_bytes, 1u, lp);
  epi_bar();  // sm.flag is rewritten at the top of the next tile
  return ok;
}

constexpr int SEQ_THREADS = THREADS + 32;  // warp 6: the activation producer

// one unit of the attention phase, out of line so that the phase's registers
// (a softmax row of 128 O values) do not crowd the GEMM roles'
__device__ __noinline__ void seq_attn_unit(const SeqMaps &maps, const SeqParams &p, uint8_t *region,
                                           t5::T5Bars<SEQ_ATT_KVS> &ab, uint32_t tmem, int kvh, int b, int rank,
                                           const Dep *dep) {
  if (p.att.block)
    t5::t5_unit<true, SEQ_P, SEQ_ATT_KVS, SEQ_THREADS>(&maps.akv, &maps.aq, p.att.D, p.att.a, p.att.q_tma, region, ab,
                                                      tmem, kvh, b, 0, rank, dep, p.status);
  else
    t5::t5_unit<false, SEQ_P, SEQ_ATT_KVS, SEQ_THREADS>(&maps.akv, &maps.aq, p.att.D, p.att.a, p.att.q_tma, region, ab,
                                                       tmem, kvh, b, 0, rank, dep, p.status);
}
// the CTA's schedule in shared memory, after the Smem block
constexpr size_t SEQ_SMEM_TAB_OFF = (sizeof(Smem) + 15) & ~(size_t)15;
// after the schedule: the attention phase's barriers and per-row results
constexpr size_t SEQ_SMEM_ATT_OFF = (SEQ_SMEM_TAB_OFF + sizeof(SeqTab) + 15) & ~(size_t)15;

// NPAD: the token columns (p.npad, seq_npad), a compile-time constant so that
// the split-K epilogue has fixed trip counts
template <int NPAD>
__global__ void __launch_bounds__(SEQ_THREADS, 1)
k_gemm_seq(const __grid_constant__ SeqMaps maps, const __grid_constant__ SeqParams p) {
  // the next launch may start once every CTA of this one runs; it waits on the
  // last GEMM's completion counter
  pdl_trigger();
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(dsm) + 1023) & ~(uintptr_t)1023);
  const int stage_bytes = A_BYTES + p.npad * BK * 2;
  float *rx = reinterpret_cast<float *>(ring + (size_t)p.stages * stage_bytes);  // [SEQ_P][BM][w4] split-K receive area
  Smem &sm = *reinterpret_cast<Smem *>(reinterpret_cast<uint8_t *>(rx) + p.rx_bytes);
  SeqTab *const stab = reinterpret_cast<SeqTab *>(reinterpret_cast<uint8_t *>(&sm) + SEQ_SMEM_TAB_OFF);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int rank = (int)cluster_rank();

  if (threadIdx.x == 0) {
    // this CTA's schedule, once, for every role
    *stab = seq_tab(p, (int)blockIdx.x);
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(&sm.full[s], 2);  // one arrival (with its byte count) from each producer
      mbar_init(&sm.empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sm.accf[b], 1);
      mbar_init(&sm.acce[b], 4);
    }
    mbar_init(&sm.recv, 1);
    mbar_init(&sm.rfree, SEQ_P - 1);
    mbar_init(&sm.drain, 1);
    sm.abort = 0;
    sm.left_last = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    // armed for this CTA's first split-K tile before the cluster barrier below
    const SeqTab tb = *stab;
    bool any = false;
    for (int j = 0; j < tb.n; ++j) any = any || sel4(tb.nt, j) > 0 || sel4(tb.lt, j) >= 0;
    mbar_expect_tx(&sm.recv, any ? seq_recv_bytes(p.M, NPAD, rank) : 0u);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&sm.tmem)),
                 "r"(p.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // peers' barriers are initialised before anyone signals them
  tc_fence_after();
  const uint32_t tmem = sm.tmem;

  // ---------------- attention phase (clusters 0 .. n_clusters - 1) ----------------
  // The ring and the receive area hold the units' Q, K/V pages and P tiles; this
  // CTA's weight stream starts after it.  The first GEMM's activations are the
  // phase's output: its activation producer waits for the phase's count.
  if (p.att.on) {
    const int q = (int)blockIdx.x / SEQ_P;
    if (q < p.att.n_clusters) {
      t5::T5Bars<SEQ_ATT_KVS> &ab =
          *reinterpret_cast<t5::T5Bars<SEQ_ATT_KVS> *>(reinterpret_cast<uint8_t *>(&sm) + SEQ_SMEM_ATT_OFF);
      const Dep *dep = &p.dep;
      for (int u = q; u < p.att.n_units; u += p.att.n_clusters) {
        const int kvh = u % p.att.D.hkv, b = u / p.att.D.hkv;
        seq_attn_unit(maps, p, ring, ab, tmem, kvh, b, rank, dep);
        dep = nullptr;
        if (threadIdx.x == 0) counter_add(p.att.done, 1u);  // after the unit's closing cluster barrier
      }
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      // the weight copies that now refill the ring follow the phase's own accesses to it
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
  }

  if (warp == 0 || warp == 6) {
    // ---------------- TMA producers: warp 0 streams every unit's weight k-block
    // (nothing to wait for but a free stage, so the next GEMM's weights fill the
    // ring ahead of time); warp 6 its activation k-block, once the GEMM's inputs
    // are complete.  Each arrives on the stage's full barrier with its own bytes.
    if (lane == 0) {
      const bool wp = warp == 0;
      const SeqTab tb = *stab;
      const uint64_t pol = wp ? policy_evict_first() : policy_evict_last();
      const uint32_t bytes = wp ? (uint32_t)A_BYTES : (uint32_t)(stage_bytes - A_BYTES);
      if (wp)
        for (int j = 0; j < tb.n; ++j) prefetch_tensormap(seq_wmap(maps, j));
      int stage = 0, u = 0;
      uint32_t ph = 0;
      bool ok = true, dep_done = false;
      for (int j = 0; j < tb.n && ok; ++j) {
        const int nt = sel4(tb.nt, j), k0 = sel4(tb.k0, j), k1 = sel4(tb.k1, j), lt = sel4(tb.lt, j);
        if (nt == 0 && lt < 0) continue;
        const CUtensorMap *map = wp ? seq_wmap(maps, j) : seq_xmap(maps, j);
        if (!wp) {
          // GEMM j reads what GEMM j - 1 (or the previous launch) wrote
          if (j == 0 && p.att.on) {
            // the attention phase's output (it waited for the launch's inputs itself)
            if (!counter_wait(p.att.done, p.att.done_n, p.status)) {
              ok = false;
              break;
            }
            dep_done = true;
          } else if (j == 0 || p.independent) {
            // the launch's inputs: once, before this producer's first copy
            if (!dep_done) dep_wait(p.dep, p.status);
            dep_done = true;
          } else if (!counter_wait(p.g[j - 1].done, p.g[j - 1].done_n, p.status)) {
            ok = false;
            break;
          }
          if ((j > 0 && !p.independent) || p.dep.wait || (j == 0 && p.att.on)) fence_proxy_async_global();
          prefetch_tensormap(map);
        }
        // the leftover part first, then the full tiles
        for (int ti = lt >= 0 ? -1 : 0; ti < nt && ok; ++ti) {
          const int tile = ti < 0 ? p.g[j].Tf + lt : sel4(tb.t0, j) + ti * sel4(tb.dt, j);
          const int row = wp ? tile * BM : 0;
          const int kb0 = ti < 0 ? sel4(tb.lk0, j) : k0, kb1 = ti < 0 ? sel4(tb.lk1, j) : k1;
          for (int k = kb0; k < kb1; ++k, ++u) {
            if (!mbar_wait(&sm.empty[stage], ph ^ 1) || *(volatile int *)&sm.abort) {
              ok = false;
              break;
            }
            mbar_expect_tx(&sm.full[stage], bytes);
            tma_load_2d(ring + (size_t)stage * stage_bytes + (wp ? 0 : A_BYTES), map, k * BK, row, &sm.full[stage], pol);
            if (++stage == p.stages) {
              stage = 0;
              ph ^= 1;
            }
          }
        }
      }
      if (!ok) {
        set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
        atomicExch(&sm.abort, 1);
      }
      // this producer's copies have landed before the CTA may exit: each of the
      // last `stages` units' full barrier completes once both producers' bytes are in
      if (wp && ok) {
        for (int v = u > p.stages ? u - p.stages : 0; v < u; ++v)
          if (!mbar_wait(&sm.full[v % p.stages], (uint32_t)((v / p.stages) & 1)))
            set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
      } else if (!ok) {
        // an aborted launch: stages may lack the other producer's copy, so give
        // this producer's copies a bounded time to land
        const unsigned long long t0 = gtime();
        while (gtime() - t0 < 200000ull) {
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      bool ok = true;
      int i = 0;
      const SeqTab tb = *stab;
      const uint32_t idesc = p.g[0].idesc;  // one row count, so one instruction descriptor for all GEMMs
      for (int j = 0; j < tb.n && ok; ++j) {
        const int nt = sel4(tb.nt, j), k0 = sel4(tb.k0, j), k1 = sel4(tb.k1, j), lt = sel4(tb.lt, j);
        for (int ti = lt >= 0 ? -1 : 0; ti < nt && ok; ++ti, ++i) {
          const int buf = i & 1;
          const int kb0 = ti < 0 ? sel4(tb.lk0, j) : k0, kb1 = ti < 0 ? sel4(tb.lk1, j) : k1;
          if (!mbar_wait(&sm.acce[buf], ((i >> 1) & 1) ^ 1)) { ok = false; break; }
          tc_fence_after();
          const uint32_t d = tmem + buf * p.npad;
          for (int k = kb0; k < kb1; ++k) {
            if (!mbar_wait(&sm.full[stage], ph) || *(volatile int *)&sm.abort) { ok = false; break; }
            tc_fence_after();
            const uint32_t a = smem_u32(ring + (size_t)stage * stage_bytes);
            const uint64_t ad = smem_desc(a), bd = smem_desc(a + A_BYTES);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) mma_bf16(d, ad + 2 * kk, bd + 2 * kk, idesc, (k > kb0 || kk > 0) ? 1u : 0u);
            mma_commit(&sm.empty[stage]);
            if (++stage == p.stages) {
              stage = 0;
              ph ^= 1;
            }
          }
          if (!ok) break;
          mma_commit(&sm.accf[buf]);
        }
      }
      if (!ok) {
        set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
        atomicExch(&sm.abort, 1);
      }
      mma_commit(&sm.drain);
      if (!mbar_wait(&sm.drain, 0)) set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
  } else {
    // ---------------- epilogue warps 2..5 ----------------
    const int sub = warp & 3;
    const int r = sub * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(sub * 32) << 16);
    const bool leader = threadIdx.x == 64;
    const SeqTab tb = *stab;
    bool ok = true;
    int i = 0;
    for (int j = 0; j < p.n && ok; ++j) {
      const SeqGemm &g = p.g[j];
      // every input of this GEMM's epilogue (norm partials, residual, positions) is
      // in place once the previous GEMM, or the previous launch, is finished
      if (leader) {
        if (j == 0)
          dep_wait(p.dep, p.status);
        else if (!p.independent && !counter_wait(p.g[j - 1].done, p.g[j - 1].done_n, p.status))
          set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
      }
      epi_bar();
      // positions and pool slots of the Q/K/V projection (the last GEMM, if any)
      // come from before this launch: set up while the first GEMM streams
      if (j == 0 && p.g[p.n - 1].mode == EP_QKV) {
        qkv_table(p.g[p.n - 1].ep.qkv, sm, p.M, r);
        epi_bar();
      }
      if (g.ep.in_ss) col_scales(g.ep, sm, p.M, r);
      const int nt = sel4(tb.nt, j), lt = sel4(tb.lt, j);
      unsigned int finished = 0;  // tiles whose columns of this CTA are written
      for (int ti = lt >= 0 ? -1 : 0; ti < nt && ok; ++ti, ++i) {
        const int t = ti < 0 ? g.Tf + lt : sel4(tb.t0, j) + ti * sel4(tb.dt, j);
        const int tl = ti < 0 ? lt : -1;
        const int fp = ti < 0 ? sel4(tb.lpart, j) : 0;  // the cluster's part of its leftover tile
        const uint32_t nb = seq_more(tb, j, ti) ? seq_recv_bytes(p.M, NPAD, rank) : 0u;
        switch (g.mode) {
          case EP_RESID:
            ok = seq_tile<EP_RESID, NPAD>(g, sm, rx, lane_addr, i, t, tl, fp, r, sub, lane, rank, leader, nb);
            break;
          case EP_SWIGLU:
            ok = seq_tile<EP_SWIGLU, NPAD>(g, sm, rx, lane_addr, i, t, tl, fp, r, sub, lane, rank, leader, nb);
            break;
          case EP_QKV:
            ok = seq_tile<EP_QKV, NPAD>(g, sm, rx, lane_addr, i, t, tl, fp, r, sub, lane, rank, leader, nb);
            break;
          case EP_SILU:
            ok = seq_tile<EP_SILU, NPAD>(g, sm, rx, lane_addr, i, t, tl, fp, r, sub, lane, rank, leader, nb);
            break;
          default:
            ok = seq_tile<EP_STORE_F32, NPAD>(g, sm, rx, lane_addr, i, t, tl, fp, r, sub, lane, rank, leader, nb);
            break;
        }
        // a leftover part counts for the owner that completed its columns
        if (leader) finished += ti >= 0 || sm.left_last ? 1u : 0u;
      }
      // this CTA's share of GEMM j is written (a barrier over the epilogue threads above)
      if (ok && leader && finished > 0) counter_add(g.done, finished);
    }
    if (!ok && leader) {
      set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
      atomicExch(&sm.abort, 1);
    }
  }

  __syncwarp();  // lanes that skipped a single-thread role wait for it here
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while a peer may still read its shared memory
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(p.tmem_cols) : "memory");
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
template <int EP>
cudaError_t ensure_smem_attr() {
  static bool done = false;
  if (done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<EP>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BUDGET + 2048);
  if (e == cudaSuccess) done = true;
  return e;
}

template <int EP>
cudaError_t launch_ep(const CUtensorMap &mw, const CUtensorMap &mx, const Params &p, size_t smem, cudaStream_t s) {
  cudaError_t e = ensure_smem_attr<EP>();
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.P * p.Q);
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  if (p.P > 1) {
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = p.P;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
  }
  return cudaLaunchKernelEx(&cfg, k_gemm_tc<EP>, mw, mx, p);
}

// clusters of P CTAs (with `smem` bytes each) that fit on the device at once
template <int EP>
int max_clusters(int P, size_t smem, bool use_cache) {
  static std::mutex mu;
  static std::map<std::pair<int, size_t>, int> cache;
  std::lock_guard<std::mutex> lock(mu);
  auto key = std::make_pair(P, smem);
  if (use_cache) {
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  int n = 0;
  if (ensure_smem_attr<EP>() == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(P);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = P;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, k_gemm_tc<EP>, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();
  if (use_cache) cache.emplace(key, n);
  return n;
}

struct Choice {
  int P = 0, Q = 0, stages = 0, rx_bytes = 0;
  size_t smem = 0;
};

// split and cluster count minimising the k-blocks each CTA streams (plus a
// small charge for the in-cluster reduction)
template <int EP>
Choice choose(int T, int kb, int npad, int sm_count, bool use_cache) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, int>, Choice> cache;
  if (use_cache) {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(std::make_tuple(T, kb, npad));
    if (it != cache.end()) return it->second;
  }
  const int stage_bytes = A_BYTES + npad * BK * 2;
  Choice best;
  long best_cost = -1;
  for (int P : {1, 2, 3, 4, 6, 8}) {
    if (P > kb || (P > 1 && npad > MAX_SPLIT_NPAD)) continue;
    // split-K receive area: P slots of [BM][w4] floats (w4 bounded with npad >= M)
    const size_t red_bytes = P > 1 ? (size_t)P * BM * (((npad + 4 * P - 1) / (4 * P)) * 4) * 4 : 0;
    int stages = (int)((SMEM_BUDGET - red_bytes - sizeof(Smem) - 1024) / stage_bytes);
    if (stages > 16) stages = 16;
    if (stages < 3) continue;
    const size_t smem = 1024 + (size_t)stages * stage_bytes + red_bytes + sizeof(Smem);
    int Q = P == 1 ? sm_count : max_clusters<EP>(P, smem, use_cache);
    if (Q <= 0) continue;
    if (Q > T) Q = T;
    const long rounds = (T + Q - 1) / Q;
    const long cost = rounds * ((kb + P - 1) / P) + (P > 1 ? 3 : 0);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best.P = P;
      best.Q = Q;
      best.stages = stages;
      best.rx_bytes = (int)red_bytes;
      best.smem = smem;
    }
  }
  if (use_cache) {
    std::lock_guard<std::mutex> lock(mu);
    cache.emplace(std::make_tuple(T, kb, npad), best);
  }
  return best;
}

template <int EP>
cudaError_t run(const CUtensorMap &mw, const CUtensorMap &mx, Params p, int sm_count, cudaStream_t s, bool use_cache,
                DepChain *chain) {
  const Choice c = choose<EP>(p.T, p.kb, p.npad, sm_count, use_cache);
  if (c.P == 0) return cudaErrorInvalidValue;
  p.P = c.P;
  p.Q = c.Q;
  p.stages = c.stages;
  p.rx_bytes = c.rx_bytes;
  p.dep = chain ? chain->take((unsigned)(c.P * c.Q)) : Dep{};
  return launch_ep<EP>(mw, mx, p, c.smem, s);
}

size_t seq_smem(int npad, int *stages_out, int *rx_bytes_out) {
  const int stage_bytes = A_BYTES + npad * BK * 2;
  // receive area of the 4-way split: a [BM][npad / 4] fp32 slot per rank
  const size_t red_bytes = (size_t)SEQ_P * BM * (npad / SEQ_P) * 4;
  const size_t tail = SEQ_SMEM_ATT_OFF + sizeof(t5::T5Bars<SEQ_ATT_KVS>);  // Smem, schedule, attention barriers
  int stages = (int)((SMEM_BUDGET - red_bytes - tail - 1024) / stage_bytes);
  if (stages > 16) stages = 16;
  *stages_out = stages;
  *rx_bytes_out = (int)red_bytes;
  return 1024 + (size_t)stages * stage_bytes + red_bytes + tail;
}

// clusters of SEQ_P persistent CTAs that are resident at once
using SeqKernel = void (*)(SeqMaps, SeqParams);
// the instantiation for npad token columns (seq_npad), or null
SeqKernel seq_kernel(int npad) {
  switch (npad) {
    case 16: return k_gemm_seq<16>;
    case 32: return k_gemm_seq<32>;
    case 48: return k_gemm_seq<48>;
    case 64: return k_gemm_seq<64>;
    case 80: return k_gemm_seq<80>;
    case 96: return k_gemm_seq<96>;
    case 128: return k_gemm_seq<128>;
    default: return nullptr;
  }
}

int seq_clusters(int npad, size_t smem) {
  static std::mutex mu;
  static std::map<std::pair<int, size_t>, int> cache;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find({npad, smem});
  if (it != cache.end()) return it->second;
  int n = 0;
  const SeqKernel kern = seq_kernel(npad);
  if (kern && cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BUDGET + 2048) ==
      cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(SEQ_P);
    cfg.blockDim = dim3(SEQ_THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = SEQ_P;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();
  cache.emplace(std::make_pair(npad, smem), n);
  return n;
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    cudaGetLastError();
  });
  return fn;
}

struct MapKey {
  const void *ptr;
  int rows, cols, ld, box_rows;
  bool operator==(const MapKey &o) const {
    return ptr == o.ptr && rows == o.rows && cols == o.cols && ld == o.ld && box_rows == o.box_rows;
  }
};
struct MapKeyHash {
  size_t operator()(const MapKey &k) const {
    size_t h = std::hash<const void *>()(k.ptr);
    h ^= (size_t)k.rows * 0x9E3779B97F4A7C15ull + ((size_t)k.cols << 20) + ((size_t)k.ld << 40) + k.box_rows;
    return h;
  }
};

// bf16 row-major [rows][ld] matrix, tile box = 64 columns x box_rows rows, 128-byte swizzle
bool tensor_map(CUtensorMap *out, const void *ptr, int rows, int cols, int ld, int box_rows, bool use_cache) {
  static std::mutex mu;
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  const MapKey key{ptr, rows, cols, ld, box_rows};
  std::lock_guard<std::mutex> lock(mu);
  if (use_cache) {
    auto it = cache.find(key);
    if (it != cache.end()) {
      *out = it->second;
      return true;
    }
  }
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  CUtensorMap m;
  if (enc(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, es,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  if (use_cache) {
    if (cache.size() > 4096) cache.clear();
    cache.emplace(key, m);
  }
  *out = m;
  return true;
}

bool tensor_map_3d(CUtensorMap *out, const void *ptr, int d0, int d1, int d2, int b1, int b2) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc || b1 < 1 || b2 < 1 || b1 > 256 || b2 > 256) return false;
  cuuint64_t dims[3] = {(cuuint64_t)d0, (cuuint64_t)d1, (cuuint64_t)d2};
  cuuint64_t strides[2] = {(cuuint64_t)d0 * 2, (cuuint64_t)d0 * d1 * 2};
  cuuint32_t box[3] = {(cuuint32_t)BK, (cuuint32_t)b1, (cuuint32_t)b2};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

void tc_layout(TcWorkspace &w, char *base, size_t &off, int sm_count, size_t rows_max, int max_tiles) {
  w.sm_count = sm_count;  // split-K partials of whole tiles stay in distributed shared memory
  // the persistent launch's leftover-tile sums and counts, per GEMM slot
  off = (off + 255) & ~(size_t)255;
  const size_t acc_bytes = (size_t)SEQ_MAX * SEQ_LEFT_MAX * BM * MAX_SPLIT_NPAD * sizeof(float);
  const size_t ctr_bytes = (size_t)SEQ_MAX * SEQ_LEFT_MAX * SEQ_P * sizeof(unsigned int);
  const size_t wctr_bytes = (size_t)WIDE_MAX_TILES * sizeof(unsigned int);
  w.lacc = base ? reinterpret_cast<float *>(base + off) : nullptr;
  w.lctr = base ? reinterpret_cast<unsigned int *>(base + off + acc_bytes) : nullptr;
  w.wctr = base ? reinterpret_cast<unsigned int *>(base + off + acc_bytes + ctr_bytes) : nullptr;
  w.left_bytes = acc_bytes + ctr_bytes + wctr_bytes;
  off += (w.left_bytes + 255) & ~(size_t)255;
  // the wide launch's split-K partials: at most WIDE_SLOT_BYTES, and never more
  // than every tile of the widest projection for rows_max rows in 4 parts
  const int max_cols = (int)(rows_max < (size_t)WIDE_MAX_NPAD ? (rows_max + 15) / 16 * 16 : WIDE_MAX_NPAD);
  size_t want = (size_t)max_tiles * 4 * BM * max_cols * sizeof(float);
  w.wslot_bytes = want < WIDE_SLOT_BYTES ? want : WIDE_SLOT_BYTES;
  w.wslots = base ? reinterpret_cast<float *>(base + off) : nullptr;
  off += (w.wslot_bytes + 255) & ~(size_t)255;
}

bool tc_supports(int N, int K, int M, int ldx, const EpArgs &ep) {
  (void)ep;
  return N > 0 && M > 0 && K > 0 && K % BK == 0 && ldx % 8 == 0 && encode_fn() != nullptr;
}

cudaError_t tc_init(const TcWorkspace &w, cudaStream_t s) {
  if (w.lacc == nullptr) return cudaSuccess;
  return cudaMemsetAsync(w.lacc, 0, w.left_bytes, s);
}

cudaError_t gemm_tc(const TcWorkspace &w, const void *W, int N, int K, const void *X, int M, int ldx,
                    const EpArgs &ep_in, int *status, cudaStream_t s, bool use_caches, DepChain *chain) {
  CUtensorMap mw;
  if (!tensor_map(&mw, W, N, K, K, BM, use_caches)) return cudaErrorInvalidValue;
  for (int m0 = 0; m0 < M; m0 += MAX_NPAD) {
    const int Mc = M - m0 < MAX_NPAD ? M - m0 : MAX_NPAD;
    Params p{};
    p.N = N;
    p.K = K;
    p.M = Mc;
    p.npad = (Mc + 15) / 16 * 16;
    p.T = (N + BM - 1) / BM;
    p.kb = K / BK;
    int cols = 32;
    while (cols < 2 * p.npad) cols <<= 1;
    p.tmem_cols = cols;
    p.idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(p.npad >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
    p.status = status;
    EpArgs ep = ep_in;
    if (ep.out_f32) ep.out_f32 += (size_t)m0 * ep.ldo;
    if (ep.out_t) ep.out_t = static_cast<bf16 *>(ep.out_t) + (size_t)m0 * ep.ldt;
    if (ep.part_val) {
      ep.part_val += (size_t)m0 * ep.n_tiles;
      ep.part_idx += (size_t)m0 * ep.n_tiles;
    }
    if (ep.in_ss) ep.in_ss += m0;
    if (ep.out_ss) ep.out_ss += m0;
    if (ep.out_xn) ep.out_xn = static_cast<bf16 *>(ep.out_xn) + (size_t)m0 * ep.ld_xn;
    if (ep.out_stash) ep.out_stash = static_cast<bf16 *>(ep.out_stash) + (size_t)m0 * ep.ld_stash;
    ep.qkv.row0 = m0;
    p.ep = ep;
    CUtensorMap mx;
    if (!tensor_map(&mx, static_cast<const bf16 *>(X) + (size_t)m0 * ldx, Mc, K, ldx, p.npad, use_caches))
      return cudaErrorInvalidValue;
    cudaError_t e;
    switch (ep.mode) {
      case EP_STORE_F32: e = run<EP_STORE_F32>(mw, mx, p, w.sm_count, s, use_caches, chain); break;
      case EP_RESID: e = run<EP_RESID>(mw, mx, p, w.sm_count, s, use_caches, chain); break;
      case EP_SWIGLU: e = run<EP_SWIGLU>(mw, mx, p, w.sm_count, s, use_caches, chain); break;
      case EP_SILU: e = run<EP_SILU>(mw, mx, p, w.sm_count, s, use_caches, chain); break;
      case EP_ARGMAX: e = run<EP_ARGMAX>(mw, mx, p, w.sm_count, s, use_caches, chain); break;
      case EP_QKV: e = run<EP_QKV>(mw, mx, p, w.sm_count, s, use_caches, chain); break;
      default: e = cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

namespace {

inline uint32_t mma_idesc(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
}

struct WideChoice {
  int P = 0, Q = 0, stages = 0;
  size_t smem = 0;
};

// k-splits and tile groups minimising the k-blocks each CTA streams, with a
// charge for writing a split tile's partial to L2 and reading partials back
// (in k-block equivalents at L2 speed); the charge was set when one CTA read all
// P partials back, and its choices still match the fastest measured P on the
// batch-16 projections (O 4, QKV 3, down 4)
WideChoice choose_wide(int T, int kb, int npad, int sms, size_t slot_bytes) {
  WideChoice best;
  const int stage_bytes = A_BYTES + npad * BK * 2;
  int stages = (int)((SMEM_BUDGET - sizeof(Smem) - 1024) / stage_bytes);
  if (stages > 16) stages = 16;
  if (stages < 2) return best;
  const int part_kb = (npad * BM * 4 / (3 * A_BYTES)) + 1;  // one partial tile, in k-blocks at about 3x
  long best_cost = -1;
  for (int P : {1, 2, 3, 4, 6, 8}) {
    if (P > 1 && (kb / P < 2 || (size_t)T * P * BM * npad * sizeof(float) > slot_bytes)) continue;
    int Q = sms / P;
    if (Q < 1) continue;
    if (Q > T) Q = T;
    const long rounds = (T + Q - 1) / Q;
    const long cost = rounds * ((kb + P - 1) / P) + (P > 1 ? (long)part_kb * (1 + P) : 0);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best.P = P;
      best.Q = Q;
    }
  }
  best.stages = stages;
  best.smem = 1024 + (size_t)stages * stage_bytes + sizeof(Smem);
  return best;
}

template <int EP>
cudaError_t launch_wide(const CUtensorMap &mw, const CUtensorMap &mx1, const CUtensorMap &mx2, const WideParams &p,
                        size_t smem, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_wide<EP>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BUDGET + 2048);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.P * p.Q);
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_gemm_wide<EP>, mw, mx1, mx2, p);
}

// The one-pass launch's schedule for Mc <= WIDE_MAX_NPAD rows: padded columns,
// accumulators, k-split and grid (choose_wide), and the leftover split; false when
// no schedule fits.  Evaluated by the launch and by the schedule test hook.
bool wide_plan(WideParams &p, int N, int K, int Mc, int sms, size_t slot_bytes) {
  p.N = N;
  p.K = K;
  p.M = Mc;
  p.npad = (Mc + 15) / 16 * 16;
  p.T = (N + BM - 1) / BM;
  p.kb = K / BK;
  // two accumulators side by side when they fit, else two that share the
  // columns [512 - npad, npad) (up to 384 token columns), else one
  p.nbuf = 2 * p.npad <= 512 ? 2 : p.npad <= 384 ? 3 : 1;
  int cols = 32;
  while (cols < (p.nbuf == 3 ? 512 : p.nbuf * p.npad)) cols <<= 1;
  p.tmem_cols = cols;
  const WideChoice c = choose_wide(p.T, p.kb, p.npad, sms, slot_bytes);
  if (c.P == 0) return false;
  p.P = c.P;
  p.Q = c.Q;
  p.stages = c.stages;
  // one tile per CTA leaves T mod Q tiles over: split each over ls = Q / (T mod Q)
  // CTAs in k (at least two k-blocks a part), so that every CTA streams about the
  // same share instead of some CTAs a whole second tile.  Measured on gate/up
  // (192 tiles on 152 CTAs): 79.9 against 87.1 us at 272 rows, but 88.8 against
  // 82.7 us at 200 rows, so only above 256 token columns.
  p.Tl = 0;
  p.ls = 1;
  if (p.P == 1 && p.T > p.Q && p.npad > 256) {
    const int tl = p.T % p.Q, ls = tl > 0 ? p.Q / tl : 0;
    if (ls >= 2 && p.kb / ls >= 2 && (size_t)tl * ls * BM * p.npad * sizeof(float) <= slot_bytes) {
      p.Tl = tl;
      p.ls = ls;
    }
  }
  return true;
}

}  // namespace

bool gemm_wide_suits(const TcWorkspace &w, int N, int K, int M) {
  if (K < BK || K % BK) return false;
  const int Mc = M < WIDE_MAX_NPAD ? M : WIDE_MAX_NPAD;
  const WideChoice c = choose_wide((N + BM - 1) / BM, K / BK, (Mc + 15) / 16 * 16, w.sm_count, w.wslot_bytes);
  return c.P >= 1;
}

cudaError_t gemm_wide(const TcWorkspace &w, const void *W, int N, int K, const void *X, int M, int ldx,
                      const EpArgs &ep_in, int *status, cudaStream_t s, DepChain *chain) {
  if (N < 1 || K < BK || K % BK || M < 1 || ldx % 8 || (N + BM - 1) / BM > WIDE_MAX_TILES || w.wctr == nullptr)
    return cudaErrorInvalidValue;
  CUtensorMap mw;
  if (!tensor_map(&mw, W, N, K, K, BM)) return cudaErrorInvalidValue;
  for (int m0 = 0; m0 < M; m0 += WIDE_MAX_NPAD) {
    const int Mc = M - m0 < WIDE_MAX_NPAD ? M - m0 : WIDE_MAX_NPAD;
    WideParams p{};
    if (!wide_plan(p, N, K, Mc, w.sm_count, w.wslot_bytes)) return cudaErrorInvalidValue;
    const int n1 = p.npad < 256 ? p.npad : 256;
    p.idesc1 = mma_idesc(n1);
    p.idesc2 = p.npad > 256 ? mma_idesc(p.npad - 256) : 0u;
    p.status = status;
    p.slots = w.wslots;
    p.ctr = w.wctr;
    EpArgs ep = ep_in;
    if (ep.out_f32) ep.out_f32 += (size_t)m0 * ep.ldo;
    if (ep.out_t) ep.out_t = static_cast<bf16 *>(ep.out_t) + (size_t)m0 * ep.ldt;
    if (ep.part_val) {
      ep.part_val += (size_t)m0 * ep.n_tiles;
      ep.part_idx += (size_t)m0 * ep.n_tiles;
    }
    if (ep.in_ss) ep.in_ss += m0;
    if (ep.out_ss) ep.out_ss += m0;
    if (ep.out_xn) ep.out_xn = static_cast<bf16 *>(ep.out_xn) + (size_t)m0 * ep.ld_xn;
    if (ep.out_stash) ep.out_stash = static_cast<bf16 *>(ep.out_stash) + (size_t)m0 * ep.ld_stash;
    ep.qkv.row0 = m0;
    p.ep = ep;
    const bf16 *xs = static_cast<const bf16 *>(X) + (size_t)m0 * ldx;
    CUtensorMap mx1, mx2;
    if (!tensor_map(&mx1, xs, Mc, K, ldx, n1)) return cudaErrorInvalidValue;
    if (p.npad > 256) {
      if (!tensor_map(&mx2, xs, Mc, K, ldx, p.npad - 256)) return cudaErrorInvalidValue;
    } else {
      mx2 = mx1;
    }
    p.dep = chain ? chain->take((unsigned)(p.P * p.Q)) : Dep{};
    const size_t smem = 1024 + (size_t)p.stages * (A_BYTES + p.npad * BK * 2) + sizeof(Smem);  // as choose_wide
    cudaError_t e;
    switch (ep.mode) {
      case EP_STORE_F32: e = launch_wide<EP_STORE_F32>(mw, mx1, mx2, p, smem, s); break;
      case EP_RESID: e = launch_wide<EP_RESID>(mw, mx1, mx2, p, smem, s); break;
      case EP_SWIGLU: e = launch_wide<EP_SWIGLU>(mw, mx1, mx2, p, smem, s); break;
      case EP_SILU: e = launch_wide<EP_SILU>(mw, mx1, mx2, p, smem, s); break;
      case EP_ARGMAX: e = launch_wide<EP_ARGMAX>(mw, mx1, mx2, p, smem, s); break;
      case EP_QKV: e = launch_wide<EP_QKV>(mw, mx1, mx2, p, smem, s); break;
      default: e = cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// The tile schedule of one GEMM of a persistent launch over Q clusters: T
// tiles, of which the T mod Q left over from the round robin are split over
// ls = Q / (T mod Q) clusters each, when that divides evenly, every part keeps a
// k-block and the part slots exist (32 to 64 columns: one epilogue chunk per
// owner); cluster q then has nt_a + (q < nt_b) full tiles.
static void seq_plan(SeqGemm &g, int N, int K, int M, int Q, int npad, bool have_slots, int q0 = 0) {
  g.q0 = q0;
  g.Qg = Q;
  g.N = N;
  g.K = K;
  g.M = M;
  g.T = (N + BM - 1) / BM;
  g.kb = K / BK;
  const int lo = g.T % Q;
  g.Tf = g.T;
  g.Tl = 0;
  g.ls = 1;
  if (lo > 0 && npad >= 32 && npad <= MAX_SPLIT_NPAD && Q <= SEQ_LEFT_MAX && Q % lo == 0 && g.kb >= SEQ_P * (Q / lo) && have_slots) {
    g.Tf = g.T - lo;
    g.Tl = lo;
    g.ls = Q / lo;
  }
  g.nt_a = g.Tf / Q;
  g.nt_b = g.Tf % Q;
  g.ls_mag = g.ls > 1 ? (unsigned)((((uint64_t)1 << 32) + g.ls - 1) / g.ls) : 0u;
  g.parts_mag = (unsigned)((((uint64_t)1 << 32) + SEQ_P * g.ls - 1) / (SEQ_P * g.ls));
}

// token columns of the persistent kernel for M rows: M rounded up to 16, and
// 112 up to 128 (one instantiation fewer; the extra columns are zero rows of X)
static int seq_npad(int M) {
  const int n = (M + 15) / 16 * 16;
  return n == 112 ? 128 : n;
}

// From 16 rows: with a single row (16 padded columns, three owners without
// columns) the launch faulted the GPU (gate/up 24576 x 4096 and O 4096 x 4096);
// fewer than 16 rows take the row-tiled kernel.
bool seq_supported(int M) {
  return M >= 16 && seq_npad(M) <= SEQ_MAX_NPAD && encode_fn() != nullptr;
}

// two Q/K/V epilogues build the same column table (positions and pool slots)
static bool same_qkv_table(const QkvOut &a, const QkvOut &b) {
  return a.pos == b.pos && a.wr == b.wr && a.page_table == b.page_table && a.R == b.R &&
         a.pages_per_seq == b.pages_per_seq && a.page_size == b.page_size && a.hkv == b.hkv &&
         (a.bk == nullptr) == (b.bk == nullptr);
}

bool seq_attn_supported(const Dims &D, int batch, int M) {
  return D.hd == 128 && D.page_size == 64 && D.R * (D.hq / D.hkv) <= t5::T5_ROWS && batch >= 1 &&
         seq_supported(M);
}

cudaError_t gemm_seq(const TcWorkspace &w, int n, const SeqSpec *sp, int M, int *status, cudaStream_t s,
                     DepChain *chain, bool independent, const SeqAttnSpec *att) {
  if (n < 1 || n > SEQ_MAX || !chain || !chain->dev || !seq_supported(M)) return cudaErrorInvalidValue;
  if (att && (independent || !seq_attn_supported(att->D, att->batch, M))) return cudaErrorInvalidValue;
  SeqParams p{};
  SeqMaps maps{};
  p.n = n;
  p.independent = independent ? 1 : 0;
  p.M = M;
  p.npad = seq_npad(M);
  p.status = status;
  int cols = 32;
  while (cols < 2 * p.npad) cols <<= 1;
  p.tmem_cols = cols;
  const size_t smem = seq_smem(p.npad, &p.stages, &p.rx_bytes);
  p.Q = seq_clusters(p.npad, smem);
  if (p.Q < 1 || p.stages < 3) return cudaErrorInvalidValue;
  int q0_first = 0, qn_first = p.Q;  // clusters of the first GEMM
  if (att) {
    // the attention phase: its region is the ring and the receive area
    if ((size_t)p.stages * (A_BYTES + p.npad * BK * 2) + p.rx_bytes < t5::t5_region_bytes<SEQ_ATT_KVS>())
      return cudaErrorInvalidValue;
    const Dims &D = att->D;
    const int G = D.hq / D.hkv;
    SeqAttnPhase &at = p.att;
    at.on = 1;
    at.block = att->a.causal ? 0 : 1;
    at.D = D;
    at.a = att->a;
    at.n_units = D.hkv * att->batch;
    at.n_clusters = at.n_units < p.Q ? at.n_units : p.Q;
    if (!tensor_map(&maps.akv, att->a.pool, D.num_pages * 2 * D.hkv * D.page_size, D.hd, D.hd, 64))
      return cudaErrorInvalidValue;
    at.q_tma = tensor_map_3d(&maps.aq, att->a.q, D.hd, D.hq, att->batch * D.R, G, D.R) ? 1 : 0;
    if (p.tmem_cols < t5::T5_TMEM_COLS) p.tmem_cols = t5::T5_TMEM_COLS;
    // the phase on the first clusters (placed first); the first GEMM (it reads the
    // phase's output) on the others when they are the majority
    if (2 * at.n_clusters <= p.Q) {
      q0_first = at.n_clusters;
      qn_first = p.Q - at.n_clusters;
    }
  }
  const uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(p.npad >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
  for (int j = 0; j < n; ++j) {
    const SeqSpec &q = sp[j];
    const int mode = q.ep.mode;
    if (q.K % BK || q.K / BK < SEQ_P || q.N < 1 || q.ldx % 8 ||
        (mode != EP_STORE_F32 && mode != EP_RESID && mode != EP_SWIGLU && mode != EP_QKV && mode != EP_SILU) ||
        // the Q/K/V column table is built once, from the last GEMM
        (mode == EP_QKV && j != n - 1 &&
         !(independent && sp[n - 1].ep.mode == EP_QKV && same_qkv_table(q.ep.qkv, sp[n - 1].ep.qkv))))
      return cudaErrorInvalidValue;
    SeqGemm &g = p.g[j];
    g.mode = mode;
    seq_plan(g, q.N, q.K, M, j == 0 ? qn_first : p.Q, p.npad, w.lacc != nullptr, j == 0 ? q0_first : 0);
    if (g.Tl > 0) {
      g.lacc = w.lacc + (size_t)j * SEQ_LEFT_MAX * BM * MAX_SPLIT_NPAD;
      g.lctr = w.lctr + (size_t)j * SEQ_LEFT_MAX * SEQ_P;
    }
    g.idesc = idesc;
    g.ep = q.ep;
    g.ep.qkv.row0 = 0;
    if (!tensor_map(&maps.w[j], q.W, q.N, q.K, q.K, BM) || !tensor_map(&maps.x[j], q.X, M, q.K, q.ldx, p.npad))
      return cudaErrorInvalidValue;
  }
  auto done_count = [&](const SeqGemm &g) { return (unsigned)(SEQ_P * g.T); };  // each owner once per tile
  if (att) p.att.done = chain->alloc((unsigned)(SEQ_P * p.att.n_units), &p.att.done_n);  // each CTA once per unit
  if (independent) {
    // no GEMM waits for another: every GEMM counts into the launch's counter
    unsigned total = 0;
    for (int j = 0; j < n; ++j) total += done_count(p.g[j]);
    const Dep d = chain->take(total);
    for (int j = 0; j < n; ++j) {
      p.g[j].done = d.signal;
      p.g[j].done_n = chain->shadow[chain->last];
    }
    p.dep = d;
    p.dep.signal = nullptr;
  } else {
    for (int j = 0; j + 1 < n; ++j) p.g[j].done = chain->alloc(done_count(p.g[j]), &p.g[j].done_n);
    const Dep d = chain->take(done_count(p.g[n - 1]));
    p.g[n - 1].done = d.signal;
    p.g[n - 1].done_n = chain->shadow[chain->last];
    p.dep = d;
    p.dep.signal = nullptr;
  }

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.Q * SEQ_P);
  cfg.blockDim = dim3(SEQ_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = SEQ_P;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, seq_kernel(p.npad), maps, p);
}

}  // namespace dflow

// Test hook (see include/dflow.h): the one-pass launch's schedule for M <= 512
// rows, computed by the functions the launch and the kernel evaluate.
extern "C" dflow_status dflow_debug_wide_schedule(int32_t N, int32_t K, int32_t M, int32_t sms, int64_t slot_bytes,
                                                  int32_t *plan, int32_t *items, int32_t max_items) {
  using namespace dflow;
  if (N < 1 || K < BK || K % BK || M < 1 || M > WIDE_MAX_NPAD || sms < 1 || sms > 1024 || slot_bytes < 0 || !plan ||
      !items || max_items < 1)
    return DFLOW_ERR_INVALID_ARG;
  WideParams p{};
  if (!wide_plan(p, N, K, M, sms, (size_t)slot_bytes)) return DFLOW_ERR_UNSUPPORTED;
  const int grid = p.P * p.Q;
  const int32_t pl[10] = {p.npad, p.T, p.kb, p.P, p.Q, p.Tl, p.ls, grid, p.nbuf, p.stages};
  for (int i = 0; i < 10; ++i) plan[i] = pl[i];
  const size_t row = 1 + 6 * (size_t)max_items;
  for (int c = 0; c < grid; ++c) {
    const int n = wide_n_items(p, c);
    if (n > max_items) return DFLOW_ERR_CAPACITY;
    int32_t *out = items + (size_t)c * row;
    out[0] = n;
    for (int i = 0; i < n; ++i) {
      const WideItem it = wide_item(p, c, i);
      const int32_t v[6] = {it.t, it.k0, it.k1, it.part, it.parts, it.slot};
      for (int j = 0; j < 6; ++j) out[1 + 6 * i + j] = v[j];
    }
  }
  return DFLOW_OK;
}

// Test hook (see include/dflow.h): the persistent launch's schedule of one GEMM
// over Q clusters, computed by the same functions the kernel runs.
extern "C" dflow_status dflow_debug_seq_schedule(int32_t N, int32_t K, int32_t M, int32_t Q, int32_t *plan,
                                                 int32_t *ctas) {
  using namespace dflow;
  if (N < 1 || K < BK || K % BK || M < 1 || Q < 1 || Q > 1024 || !plan || !ctas) return DFLOW_ERR_INVALID_ARG;
  const int npad = seq_npad(M);
  if (npad > SEQ_MAX_NPAD || K / BK < SEQ_P) return DFLOW_ERR_UNSUPPORTED;
  SeqParams p{};
  p.n = 1;
  p.M = M;
  p.npad = npad;
  p.Q = Q;
  seq_plan(p.g[0], N, K, M, Q, npad, true);
  const SeqGemm &g = p.g[0];
  const int32_t pl[8] = {npad, g.T, g.kb, g.Tf, g.Tl, g.ls, SEQ_P * g.T, SEQ_LEFT_MAX};
  for (int i = 0; i < 8; ++i) plan[i] = pl[i];
  for (int c = 0; c < Q * SEQ_P; ++c) {
    const SeqTab t = seq_tab(p, c);
    const int32_t row[10] = {t.nt[0], t.t0[0], t.dt[0], t.k0[0], t.k1[0], t.lt[0], t.lk0[0], t.lk1[0], t.lpart[0],
                             (int32_t)seq_recv_bytes(M, npad, c % SEQ_P)};
    for (int i = 0; i < 10; ++i) ctas[(size_t)c * 10 + i] = row[i];
  }
  return DFLOW_OK;
}
