// Block-query attention on tensor cores for bf16 caches (Sec. 3: the target
// verifies the whole draft block in one pass; the drafter attends to its
// injected context and to the block).
//
// One CTA owns (kv head, sequence, key split, group of 80 query rows).  The
// query rows are the block rows x the G query heads that share the kv head.
//   * warp 0 streams the K and V tiles of the split with TMA: one tile is one
//     64-token page of one kv head (a 2D tensor map over the paged pool, 128-
//     byte swizzle), double buffered; in drafter mode the block's own K/V rows
//     form one more tile, gathered by the same warp with vector loads.
//   * warps 1-5 each own 16 query rows: S = Q K^T and O += P V with
//     mma.sync m16n8k16 (bf16 in, fp32 accumulate), online softmax in base 2,
//     causal mask inside the verify block, keys past the valid context masked
//     (and their V rows zeroed in registers, so stale pool bytes never reach
//     the accumulator).
//   * the key splits of one (kv head, sequence, query group) form a thread-
//     block cluster: each split leaves (o, m, l) in its shared memory and every
//     CTA merges a slice of the query rows over all splits through
//     distributed shared memory, writing the final bf16 rows.  One launch per
//     attention call, no global partials.
#include <cuda.h>

#include "dflow_internal.cuh"
#include "gemm_tc.cuh"
#include "ptx.cuh"

namespace dflow {

namespace {

using namespace ptx;

constexpr int QROWS = 80;  // 5 consumer warps x 16 rows
constexpr int THREADS = 192;
constexpr int STAGES = 2;
constexpr int MAX_SPLITS = 16;  // cluster size (non-portable; 2 CTAs fit per SM)

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float *c, const uint32_t *a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}
__device__ __forceinline__ void cons_bar() { asm volatile("bar.sync 1, 160;" ::: "memory"); }

// byte offset of (row, 16-byte chunk) inside a tile stored as 64-column boxes
// of [64 rows][128 bytes] with the 128-byte swizzle
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
  return (uint32_t)((chunk >> 3) * 8192 + row * 128 + (((chunk & 7) ^ (row & 7)) << 4));
}

template <int HD, bool BLOCK>
__global__ void __launch_bounds__(THREADS, 2)
k_attn_tc(const __grid_constant__ CUtensorMap tm, Dims D, AttnArgs a, int qgroups, int *status) {
  (void)qgroups;
  pdl_entry();
  if (*status) return;
  constexpr int TILE = 64 * HD * 2;  // bytes of one K (or V) tile
  constexpr int QS = HD + 8;         // padded Q row (elements)
  constexpr int NB = HD / 64;
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(dsm) + 1023) & ~(uintptr_t)1023);
  uint8_t *ring = base;                                            // [STAGES][K tile | V tile]
  bf16 *qs = reinterpret_cast<bf16 *>(ring + STAGES * 2 * TILE);   // [QROWS][QS]
  uint64_t *full = reinterpret_cast<uint64_t *>(qs + QROWS * QS);
  uint64_t *empty = full + STAGES;
  float *m_sm = reinterpret_cast<float *>(empty + STAGES);  // [QROWS] running max (base 2) of this split
  float *l_sm = m_sm + QROWS;                               // [QROWS] softmax denominator of this split
  float *coef = l_sm + QROWS;                               // [QROWS][MAX_SPLITS] merge weights
  float *o_sm = reinterpret_cast<float *>(ring);            // [QROWS][HD] after the key loop (reuses the ring)

  const int kvh = blockIdx.x, b = blockIdx.y;
  const int split = blockIdx.z % a.n_splits, qg = blockIdx.z / a.n_splits;  // split = rank in the cluster
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = D.hq / D.hkv, R = D.R, QR = R * G, row0 = qg * QROWS;

  const int n_keys = a.causal ? a.kvlen[b] : a.seq_len[b] - 1;
  const int n_tiles = (n_keys + 63) / 64;
  const int t_lo = (int)((long long)split * n_tiles / a.n_splits);
  const int t_hi = (int)((long long)(split + 1) * n_tiles / a.n_splits);
  const bool extra = BLOCK && split == a.n_splits - 1;
  const int T = (t_hi - t_lo) + (extra ? 1 : 0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 5);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == 0) {
    // ---------------- producer ----------------
    const int *pt = a.page_table + (size_t)b * D.pages_per_seq;
    const uint64_t pol = policy_evict_first();
    int stage = 0;
    uint32_t ph = 0;
    int issued[STAGES];
    for (int s = 0; s < STAGES; ++s) issued[s] = -1;
    for (int it = 0; it < T; ++it) {
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&empty[stage], ph ^ 1) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
        break;
      }
      uint8_t *kt = ring + (size_t)stage * 2 * TILE, *vt = kt + TILE;
      const int tile = t_lo + it;
      if (tile < t_hi) {
        if (lane == 0) {
          const int page = pt[tile];
          const int rk = ((page * 2 + 0) * D.hkv + kvh) * 64, rv = ((page * 2 + 1) * D.hkv + kvh) * 64;
          mbar_expect_tx(&full[stage], 2 * TILE);
#pragma unroll
          for (int bx = 0; bx < NB; ++bx) {
            tma_load_2d(kt + bx * 8192, &tm, bx * 64, rk, &full[stage], pol);
            tma_load_2d(vt + bx * 8192, &tm, bx * 64, rv, &full[stage], pol);
          }
          issued[stage] = (int)ph;
        }
      } else {
        // the block's own K/V rows (drafter mode), zero past row R
        const bf16 *bk = static_cast<const bf16 *>(a.bk), *bv = static_cast<const bf16 *>(a.bv);
        for (int e = lane; e < 64 * (HD / 8); e += 32) {
          const int j = e / (HD / 8), c = e % (HD / 8);
          uint4 kx = make_uint4(0, 0, 0, 0), vx = make_uint4(0, 0, 0, 0);
          if (j < R) {
            const size_t off = ((size_t)(b * R + j) * D.hkv + kvh) * HD + c * 8;
            kx = *reinterpret_cast<const uint4 *>(bk + off);
            vx = *reinterpret_cast<const uint4 *>(bv + off);
          }
          *reinterpret_cast<uint4 *>(kt + swz(j, c)) = kx;
          *reinterpret_cast<uint4 *>(vt + swz(j, c)) = vx;
        }
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&full[stage]);
          issued[stage] = (int)ph;  // the drain below waits on the latest fill of every stage
        }
      }
      if (++stage == STAGES) {
        stage = 0;
        ph ^= 1;
      }
    }
    if (lane == 0)
      for (int s = 0; s < STAGES; ++s)
        if (issued[s] >= 0 && !mbar_wait(&full[s], (uint32_t)issued[s])) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
    __syncwarp();
    __syncthreads();  // (A) every copy into the ring has landed
  } else {

  // ---------------- consumers ----------------
  const int cw = warp - 1;              // 0..4
  const int g = lane / 4, t4 = lane % 4;
  const bf16 *q = static_cast<const bf16 *>(a.q);
  {
    // all of this thread's query chunks are loaded before any is stored
    constexpr int PER = QROWS * (HD / 8) / 160;
    uint4 v[PER];
#pragma unroll
    for (int k = 0; k < PER; ++k) {
      const int e = threadIdx.x - 32 + k * 160, r = e / (HD / 8), c = e % (HD / 8), qr = row0 + r;
      v[k] = make_uint4(0, 0, 0, 0);
      if (qr < QR) {
        const int i = qr / G, h = kvh * G + qr % G;
        v[k] = __ldg(reinterpret_cast<const uint4 *>(q + ((size_t)(b * R + i) * D.hq + h) * HD + c * 8));
      }
    }
#pragma unroll
    for (int k = 0; k < PER; ++k) {
      const int e = threadIdx.x - 32 + k * 160, r = e / (HD / 8), c = e % (HD / 8);
      *reinterpret_cast<uint4 *>(qs + r * QS + c * 8) = v[k];
    }
  }
  cons_bar();
  uint32_t qf[HD / 16][4];
  {
    const int mi = lane / 8;
    const int r = cw * 16 + (mi & 1) * 8 + (lane & 7);
#pragma unroll
    for (int kc = 0; kc < HD / 16; ++kc)
      ldsm_x4(smem_u32(qs + r * QS + kc * 16 + (mi >> 1) * 8), qf[kc][0], qf[kc][1], qf[kc][2], qf[kc][3]);
  }
  int qpos[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int qr = row0 + cw * 16 + g + 8 * h;
    qpos[h] = qr < QR ? a.pos[b * R + qr / G] : -1;
  }
  const float sl2 = 1.4426950408889634f * rsqrtf((float)HD);  // log2(e) / sqrt(hd)
  float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
  float o[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;

  int stage = 0;
  uint32_t ph = 0;
  for (int it = 0; it < T; ++it) {
    const int tile = t_lo + it;
    const bool blk = tile >= t_hi;
    int ok = 1;
    if (lane == 0) ok = mbar_wait(&full[stage], ph) ? 1 : 0;
    if (!__shfl_sync(0xffffffffu, ok, 0)) {
      if (lane == 0) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
      break;
    }
    mbar_wait(&full[stage], ph);  // completes at once; gives every lane the acquire
    const uint32_t kt = smem_u32(ring + (size_t)stage * 2 * TILE), vt = kt + TILE;
    const int key0 = blk ? 0 : tile * 64;
    const int lim = blk ? R : n_keys;  // keys at or past lim hold no data
    // ---- S = Q K^T over 64 keys
    float s[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int kc = 0; kc < HD / 16; ++kc) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int mi = lane / 8;
        const int key = np * 16 + (mi >> 1) * 8 + (lane & 7);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kt + swz(key, kc * 2 + (mi & 1)), b0, b1, b2, b3);
        mma16816(s[2 * np], qf[kc], b0, b1);
        mma16816(s[2 * np + 1], qf[kc], b2, b3);
      }
    }
    // ---- mask, online softmax (base 2)
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int h = e >> 1;
        const int kk = key0 + j * 8 + 2 * t4 + (e & 1);
        bool ok = kk < lim;
        if (!blk && a.causal) ok = ok && kk <= qpos[h];
        if (!blk && !a.causal) ok = ok && qpos[h] >= 0;
        if (blk) ok = ok && qpos[h] >= 0;
        const float v = ok ? s[j][e] * sl2 : -INFINITY;
        s[j][e] = v;
        mx[h] = fmaxf(mx[h], v);
      }
    }
    float corr[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 1));
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 2));
      const float mn = fmaxf(m[h], mx[h]);
      corr[h] = (mn == -INFINITY) ? 1.f : exp2f(m[h] - mn);
      m[h] = mn;
    }
    float rs[2] = {0.f, 0.f};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int h = e >> 1;
        const float p = (m[h] == -INFINITY) ? 0.f : exp2f(s[j][e] - m[h]);
        s[j][e] = p;
        rs[h] += p;
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) l[h] = l[h] * corr[h] + rs[h];
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      o[j][0] *= corr[0];
      o[j][1] *= corr[0];
      o[j][2] *= corr[1];
      o[j][3] *= corr[1];
    }
    // ---- O += P V
    const bool partial = key0 + 64 > lim;
#pragma unroll
    for (int kc2 = 0; kc2 < 4; ++kc2) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kc2][0], s[2 * kc2][1]);
      pa[1] = pack_bf16(s[2 * kc2][2], s[2 * kc2][3]);
      pa[2] = pack_bf16(s[2 * kc2 + 1][0], s[2 * kc2 + 1][1]);
      pa[3] = pack_bf16(s[2 * kc2 + 1][2], s[2 * kc2 + 1][3]);
#pragma unroll
      for (int dp = 0; dp < HD / 16; ++dp) {
        const int mi = lane / 8;
        const int key = kc2 * 16 + (mi & 1) * 8 + (lane & 7);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vt + swz(key, dp * 2 + (mi >> 1)), b0, b1, b2, b3);
        if (partial) {
          // rows (keys) of each 8x8 matrix this thread holds: 2*t4 and 2*t4+1
          const int k0 = key0 + kc2 * 16 + 2 * t4, k1 = k0 + 8;
          const uint32_t m0 = (k0 < lim ? 0xFFFFu : 0u) | (k0 + 1 < lim ? 0xFFFF0000u : 0u);
          const uint32_t m1 = (k1 < lim ? 0xFFFFu : 0u) | (k1 + 1 < lim ? 0xFFFF0000u : 0u);
          b0 &= m0;
          b1 &= m1;
          b2 &= m0;
          b3 &= m1;
        }
        mma16816(o[2 * dp], pa, b0, b1);
        mma16816(o[2 * dp + 1], pa, b2, b3);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[stage]);
    if (++stage == STAGES) {
      stage = 0;
      ph ^= 1;
    }
  }

  // ---- this split's (l) summed over the quad; (m, l) per row to shared memory
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    l[h] += __shfl_xor_sync(0xffffffffu, l[h], 1);
    l[h] += __shfl_xor_sync(0xffffffffu, l[h], 2);
  }
  __syncthreads();  // (A) the ring is free: reuse it for this split's o
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int rr = cw * 16 + g + 8 * h;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j)
      *reinterpret_cast<float2 *>(o_sm + rr * HD + j * 8 + 2 * t4) = make_float2(o[j][2 * h], o[j][2 * h + 1]);
    if (t4 == 0) {
      m_sm[rr] = m[h];
      l_sm[rr] = l[h];
    }
  }
  }  // consumers

  // ---- merge the splits of this cluster: CTA `split` finishes rows [r_lo, r_hi)
  __syncthreads();
  cluster_sync();
  // (the cluster always has MAX_SPLITS CTAs, so every loop below unrolls and all
  // remote loads of a thread are in flight together)
  constexpr int S = MAX_SPLITS;
  constexpr int RPR = (QROWS + S - 1) / S;
  const int r_lo = min(QROWS, split * RPR), r_hi = min(QROWS, r_lo + RPR);
  if (threadIdx.x < r_hi - r_lo) {
    const int rr = r_lo + threadIdx.x;
    float ms[S], ls[S], M = -INFINITY;
#pragma unroll
    for (int sp = 0; sp < S; ++sp) {
      ms[sp] = ld_dsmem_f32(mapa(smem_u32(m_sm + rr), (uint32_t)sp));
      ls[sp] = ld_dsmem_f32(mapa(smem_u32(l_sm + rr), (uint32_t)sp));
    }
#pragma unroll
    for (int sp = 0; sp < S; ++sp) M = fmaxf(M, ms[sp]);
    float L = 0.f;
#pragma unroll
    for (int sp = 0; sp < S; ++sp) L += (ms[sp] == -INFINITY) ? 0.f : exp2f(ms[sp] - M) * ls[sp];
#pragma unroll
    for (int sp = 0; sp < S; ++sp)
      coef[threadIdx.x * MAX_SPLITS + sp] = (ms[sp] == -INFINITY || L <= 0.f) ? 0.f : exp2f(ms[sp] - M) / L;
  }
  __syncthreads();
  bf16 *out = static_cast<bf16 *>(a.out);
  for (int e = threadIdx.x; e < (r_hi - r_lo) * (HD / 4); e += THREADS) {
    const int rr = r_lo + e / (HD / 4), d4 = (e % (HD / 4)) * 4, qr = row0 + rr;
    if (qr >= QR) continue;
    float4 x[S];
#pragma unroll
    for (int sp = 0; sp < S; ++sp) x[sp] = ld_dsmem_f4(mapa(smem_u32(o_sm + rr * HD + d4), (uint32_t)sp));
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int sp = 0; sp < S; ++sp) {
      const float c = coef[(rr - r_lo) * MAX_SPLITS + sp];
      acc.x += c * x[sp].x;
      acc.y += c * x[sp].y;
      acc.z += c * x[sp].z;
      acc.w += c * x[sp].w;
    }
    const int i = qr / G, head = kvh * G + qr % G;
    bf16 *dst = out + ((size_t)(b * R + i) * D.hq + head) * HD + d4;
    *reinterpret_cast<__nv_bfloat162 *>(dst) = __floats2bfloat162_rn(acc.x, acc.y);
    *reinterpret_cast<__nv_bfloat162 *>(dst + 2) = __floats2bfloat162_rn(acc.z, acc.w);
  }
  cluster_sync();  // peers may still read this CTA's shared memory until here
}

template <int HD, bool BLOCK>
cudaError_t launch(const CUtensorMap &tm, const Dims &D, int batch, const AttnArgs &a, int *status,
                   cudaStream_t s) {
  constexpr int TILE = 64 * HD * 2;
  const size_t smem = 1024 + STAGES * 2 * TILE + QROWS * (HD + 8) * 2 + 4 * STAGES * 8 +
                      (2 * QROWS + QROWS * MAX_SPLITS) * 4;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_attn_tc<HD, BLOCK>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_attn_tc<HD, BLOCK>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int G = D.hq / D.hkv;
  const int qgroups = (D.R * G + QROWS - 1) / QROWS;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(D.hkv, batch, a.n_splits * qgroups);
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = 1;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = a.n_splits;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, k_attn_tc<HD, BLOCK>, tm, D, a, qgroups, status);
}

}  // namespace

bool attention_tc_supported(const Dims &D) {
  return D.page_size == 64 && (D.hd == 64 || D.hd == 128);
}

cudaError_t attention_tc(const Dims &D, int batch, const AttnArgs &a_in, int *status, cudaStream_t s) {
  AttnArgs a = a_in;
  a.n_splits = MAX_SPLITS;  // one cluster of MAX_SPLITS key splits per (kv head, sequence, query group)
  CUtensorMap tm;
  const int rows = D.num_pages * 2 * D.hkv * D.page_size;
  if (!tensor_map(&tm, a.pool, rows, D.hd, D.hd, 64)) return cudaErrorInvalidValue;
  const bool block = !a.causal;
  if (D.hd == 128) return block ? launch<128, true>(tm, D, batch, a, status, s) : launch<128, false>(tm, D, batch, a, status, s);
  return block ? launch<64, true>(tm, D, batch, a, status, s) : launch<64, false>(tm, D, batch, a, status, s);
}

}  // namespace dflow
