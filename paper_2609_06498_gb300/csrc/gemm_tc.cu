// Weight-streaming GEMM on the 5th-generation tensor cores (tcgen05 + TMEM),
// fed by TMA, for the dense projections of the round (Qwen3 QKV / O / gate-up /
// down, the Eq. 1 feature projection, the Eq. 4 relay MLP, the drafter context
// K/V projection and the LM head).
//
// out[m][n] = sum_k X[m][k] W[n][k] with few rows m (the B+1 block rows of each
// sequence) and many output features n.  The kernel computes the transposed
// product D[n][m] = W[n][:] . X[m][:] so the weight tile is the 128-row A
// operand and the token rows are the MMA's N dimension (padded to 16):
//
//   * W is cut into 128-feature tiles x 64-wide k-blocks ("units").  The units
//     are split evenly over one CTA per SM (stream-K): a CTA walks a contiguous
//     run of units, possibly across tile boundaries.
//   * warp 0 streams W and X k-blocks with TMA (128-byte swizzle) into a ring
//     of shared-memory stages; warp 1 issues tcgen05.mma (128 x Npad x 16) into
//     a TMEM accumulator (two buffers, so the epilogue of one tile overlaps the
//     MMAs of the next); warps 2-5 read the accumulator with tcgen05.ld and run
//     the fused epilogue.
//   * A tile finished by one CTA goes straight to the epilogue.  A tile split
//     across CTAs leaves fp32 partials in the workspace; the last CTA to arrive
//     on the tile's counter sums them in a fixed order (deterministic) and runs
//     the epilogue, then resets the counter.  Nobody spins on another CTA.
//   * Every mbarrier wait is bounded (about 2 s of globaltimer); on expiry the
//     kernel records DFLOW_ERR_DEVICE_TIMEOUT, drains its own copies and MMAs,
//     frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>
#include <unordered_map>

#include "gemm_tc.cuh"
#include "ptx.cuh"

namespace dflow {

namespace {

using namespace ptx;

constexpr int BM = 128;           // weight rows per tile (MMA M)
constexpr int BK = 64;            // k elements per unit (128 bytes of bf16: one swizzle row)
constexpr int A_BYTES = BM * BK * 2;
constexpr int MAX_NPAD = 256;
constexpr int THREADS = 192;
constexpr int SMEM_BUDGET = 224 * 1024;

// ---------------------------------------------------------------------------
// stream-K schedule (identical on host and device)
// ---------------------------------------------------------------------------
__host__ __device__ __forceinline__ int cta_start(int c, int U, int C) { return (int)((long long)c * U / C); }
__host__ __device__ __forceinline__ int cta_of_unit(int u, int U, int C) {
  int c = (int)(((long long)(u + 1) * C - 1) / U);
  if (c > C - 1) c = C - 1;
  while (c + 1 < C && cta_start(c + 1, U, C) <= u) ++c;
  while (c > 0 && cta_start(c, U, C) > u) --c;
  return c;
}

struct Params {
  int N, K, M, npad, tiles, kb, U, C, stages, tmem_cols, ldx;
  uint32_t idesc;
  EpArgs ep;
  float *part;
  int *cnt;
  int *status;
};

struct Smem {
  uint64_t full[16], empty[16], accf[2], acce[2], drain;
  uint32_t tmem;
  int flag;
  int abort;
  float xch[16][64];
  float rv[4][16];
  int ri[4][16];
};

// epilogue on one 16-column chunk; v[j] = D[row r][col c0+j]
template <int EP>
__device__ __forceinline__ void epilogue_chunk(const Params &p, Smem &sm, int t, int r, int sub, int lane, int c0,
                                               const float *v) {
  const int n = t * BM + r;
  const EpArgs &ep = p.ep;
  if constexpr (EP == EP_STORE_F32 || EP == EP_RESID || EP == EP_SILU) {
    if (n < p.N) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int col = c0 + j;
        if (col < p.M) {
          if constexpr (EP == EP_STORE_F32) ep.out_f32[(size_t)col * ep.ldo + n] = v[j];
          if constexpr (EP == EP_RESID) ep.out_f32[(size_t)col * ep.ldo + n] += v[j];
          if constexpr (EP == EP_SILU) reinterpret_cast<bf16 *>(ep.out_t)[(size_t)col * ep.ldt + n] = __float2bfloat16_rn(silu_f(v[j]));
        }
      }
    }
  } else if constexpr (EP == EP_SWIGLU) {
    // rows 0..63 of the tile are gate features 64t.., rows 64..127 the matching up features
    if (r >= 64) {
#pragma unroll
      for (int j = 0; j < 16; ++j) sm.xch[j][r - 64] = v[j];
    }
    epi_bar();
    if (r < 64 && t * BM + 64 + r < p.N) {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int col = c0 + j;
        if (col < p.M)
          reinterpret_cast<bf16 *>(ep.out_t)[(size_t)col * ep.ldt + t * 64 + r] =
              __float2bfloat16_rn(silu_f(v[j]) * sm.xch[j][r]);
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
      if (col < p.M) {
        ep.part_val[(size_t)col * ep.n_tiles + t] = bv;
        ep.part_idx[(size_t)col * ep.n_tiles + t] = bi;
      }
    }
    epi_bar();
  }
}

template <int EP>
__global__ void __launch_bounds__(THREADS, 1)
k_gemm_tc(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, const Params p) {
  if (*p.status) return;
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(dsm) + 1023) & ~(uintptr_t)1023);
  const int stage_bytes = A_BYTES + p.npad * BK * 2;
  Smem &sm = *reinterpret_cast<Smem *>(ring + (size_t)p.stages * stage_bytes);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int c = blockIdx.x;
  const int u0 = cta_start(c, p.U, p.C), u1 = cta_start(c + 1, p.U, p.C);

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

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint64_t pw = policy_evict_first(), px = policy_evict_last();
      int stage = 0;
      uint32_t ph = 0;
      int issued_phase[16];
      for (int s = 0; s < 16; ++s) issued_phase[s] = -1;
      for (int u = u0; u < u1; ++u) {
        if (!mbar_wait(&sm.empty[stage], ph ^ 1)) {
          set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
          atomicExch(&sm.abort, 1);
          break;
        }
        if (*(volatile int *)&sm.abort) break;
        const int t = u / p.kb, k = u % p.kb;
        uint8_t *a = ring + (size_t)stage * stage_bytes;
        mbar_expect_tx(&sm.full[stage], stage_bytes);
        tma_load_2d(a, &tmW, k * BK, t * BM, &sm.full[stage], pw);
        tma_load_2d(a + A_BYTES, &tmX, k * BK, 0, &sm.full[stage], px);
        issued_phase[stage] = (int)ph;
        if (++stage == p.stages) {
          stage = 0;
          ph ^= 1;
        }
      }
      // every copy this thread started has landed before the CTA may exit
      for (int s = 0; s < p.stages; ++s)
        if (issued_phase[s] >= 0 && !mbar_wait(&sm.full[s], (uint32_t)issued_phase[s]))
          set_status(p.status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      int seg = 0;
      bool ok = true;
      for (int u = u0; u < u1 && ok;) {
        const int t = u / p.kb;
        const int ue = min(u1, (t + 1) * p.kb);
        const int buf = seg & 1;
        if (!mbar_wait(&sm.acce[buf], ((seg >> 1) & 1) ^ 1)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem + buf * p.npad;
        for (int uu = u; uu < ue; ++uu) {
          if (!mbar_wait(&sm.full[stage], ph) || *(volatile int *)&sm.abort) { ok = false; break; }
          tc_fence_after();
          const uint32_t a = smem_u32(ring + (size_t)stage * stage_bytes);
          const uint64_t ad = smem_desc(a), bd = smem_desc(a + A_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            mma_bf16(d, ad + 2 * kk, bd + 2 * kk, p.idesc, (uu > u || kk > 0) ? 1u : 0u);
          mma_commit(&sm.empty[stage]);
          if (++stage == p.stages) {
            stage = 0;
            ph ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(&sm.accf[buf]);
        ++seg;
        u = ue;
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
    int seg = 0;
    for (int u = u0; u < u1;) {
      const int t = u / p.kb;
      const int ue = min(u1, (t + 1) * p.kb);
      const int buf = seg & 1;
      if (leader) sm.flag = mbar_wait(&sm.accf[buf], (seg >> 1) & 1) ? 1 : 0;
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
      const bool whole = (u == t * p.kb) && (ue == (t + 1) * p.kb);
      float v[16];
      if (whole) {
        for (int c0 = 0; c0 < p.npad; c0 += 16) {
          tmem_ld16(acc_addr + c0, v);
          epilogue_chunk<EP>(p, sm, t, r, sub, lane, c0, v);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.acce[buf]);
      } else {
        // partial tile: park the fp32 partial, count arrivals, the last one finishes the tile
        const int cf = cta_of_unit(t * p.kb, p.U, p.C), cl = cta_of_unit((t + 1) * p.kb - 1, p.U, p.C);
        const int slot = 2 * c + (t == u0 / p.kb ? 0 : 1);
        float *mine = p.part + (size_t)slot * BM * MAX_NPAD;
        for (int c0 = 0; c0 < p.npad; c0 += 16) {
          tmem_ld16(acc_addr + c0, v);
#pragma unroll
          for (int j = 0; j < 16; ++j) mine[(size_t)(c0 + j) * BM + r] = v[j];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.acce[buf]);
        __threadfence();
        epi_bar();
        if (leader) sm.flag = (atomicAdd(&p.cnt[t], 1) == cl - cf) ? 1 : 0;
        epi_bar();
        if (sm.flag) {
          __threadfence();
          for (int c0 = 0; c0 < p.npad; c0 += 16) {
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] = 0.f;
            for (int cc = cf; cc <= cl; ++cc) {
              const int s = 2 * cc + (t == cta_start(cc, p.U, p.C) / p.kb ? 0 : 1);
              const float *src = p.part + (size_t)s * BM * MAX_NPAD;
#pragma unroll
              for (int j = 0; j < 16; ++j) v[j] += __ldcg(src + (size_t)(c0 + j) * BM + r);
            }
            epilogue_chunk<EP>(p, sm, t, r, sub, lane, c0, v);
          }
          if (leader) p.cnt[t] = 0;
        }
      }
      epi_bar();  // sm.flag is rewritten by the leader at the top of the next segment
      ++seg;
      u = ue;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(p.tmem_cols) : "memory");
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
template <int EP>
cudaError_t launch_ep(const CUtensorMap &mw, const CUtensorMap &mx, const Params &p, size_t smem, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<EP>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BUDGET + 2048);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  k_gemm_tc<EP><<<p.C, THREADS, smem, s>>>(mw, mx, p);
  return cudaGetLastError();
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
bool tensor_map(CUtensorMap *out, const void *ptr, int rows, int cols, int ld, int box_rows) {
  static std::mutex mu;
  static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  const MapKey key{ptr, rows, cols, ld, box_rows};
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *out = it->second;
    return true;
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
  if (cache.size() > 4096) cache.clear();
  cache.emplace(key, m);
  *out = m;
  return true;
}


void tc_layout(TcWorkspace &w, char *base, size_t &off, int sm_count, size_t rows_max, int max_tiles) {
  (void)rows_max;
  w.sm_count = sm_count;
  const size_t part_bytes = (size_t)2 * sm_count * BM * MAX_NPAD * 4;
  w.part = base ? reinterpret_cast<float *>(base + off) : nullptr;
  w.part_elems = part_bytes / 4;
  off += (part_bytes + 255) & ~(size_t)255;
  w.counters = base ? reinterpret_cast<int *>(base + off) : nullptr;
  w.n_counters = max_tiles;
  off += ((size_t)max_tiles * 4 + 255) & ~(size_t)255;
}

bool tc_supports(int N, int K, int M, int ldx, const EpArgs &ep) {
  (void)ep;
  return N > 0 && M > 0 && K > 0 && K % BK == 0 && ldx % 8 == 0 && encode_fn() != nullptr;
}

cudaError_t tc_init(const TcWorkspace &w, cudaStream_t s) {
  return cudaMemsetAsync(w.counters, 0, (size_t)w.n_counters * 4, s);
}

cudaError_t gemm_tc(const TcWorkspace &w, const void *W, int N, int K, const void *X, int M, int ldx,
                    const EpArgs &ep_in, int *status, cudaStream_t s) {
  const int tiles = (N + BM - 1) / BM;
  if (tiles > w.n_counters) return cudaErrorInvalidValue;
  CUtensorMap mw;
  if (!tensor_map(&mw, W, N, K, K, BM)) return cudaErrorInvalidValue;
  for (int m0 = 0; m0 < M; m0 += MAX_NPAD) {
    const int Mc = M - m0 < MAX_NPAD ? M - m0 : MAX_NPAD;
    Params p{};
    p.N = N;
    p.K = K;
    p.M = Mc;
    p.npad = (Mc + 15) / 16 * 16;
    p.tiles = tiles;
    p.kb = K / BK;
    p.U = tiles * p.kb;
    p.C = p.U < w.sm_count ? p.U : w.sm_count;
    const int stage_bytes = A_BYTES + p.npad * BK * 2;
    p.stages = (SMEM_BUDGET - (int)sizeof(Smem) - 1024) / stage_bytes;
    if (p.stages > 16) p.stages = 16;
    if (p.stages < 2) return cudaErrorInvalidValue;
    int cols = 32;
    while (cols < 2 * p.npad) cols <<= 1;
    p.tmem_cols = cols;
    p.ldx = ldx;
    p.idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(p.npad >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
    p.part = w.part;
    p.cnt = w.counters;
    p.status = status;
    EpArgs ep = ep_in;
    if (ep.out_f32) ep.out_f32 += (size_t)m0 * ep.ldo;
    if (ep.out_t) ep.out_t = static_cast<bf16 *>(ep.out_t) + (size_t)m0 * ep.ldt;
    if (ep.part_val) {
      ep.part_val += (size_t)m0 * ep.n_tiles;
      ep.part_idx += (size_t)m0 * ep.n_tiles;
    }
    p.ep = ep;
    CUtensorMap mx;
    if (!tensor_map(&mx, static_cast<const bf16 *>(X) + (size_t)m0 * ldx, Mc, K, ldx, p.npad)) return cudaErrorInvalidValue;
    const size_t smem = 1024 + (size_t)p.stages * stage_bytes + sizeof(Smem);
    cudaError_t e;
    switch (ep.mode) {
      case EP_STORE_F32: e = launch_ep<EP_STORE_F32>(mw, mx, p, smem, s); break;
      case EP_RESID: e = launch_ep<EP_RESID>(mw, mx, p, smem, s); break;
      case EP_SWIGLU: e = launch_ep<EP_SWIGLU>(mw, mx, p, smem, s); break;
      case EP_SILU: e = launch_ep<EP_SILU>(mw, mx, p, smem, s); break;
      case EP_ARGMAX: e = launch_ep<EP_ARGMAX>(mw, mx, p, smem, s); break;
      default: e = cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace dflow
