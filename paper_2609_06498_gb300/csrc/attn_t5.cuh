// One unit of the tcgen05 paged block attention (Sec. 3: the target verifies the
// whole draft block in one pass; the drafter attends to its injected context and
// to the block): query rows of one (kv head, sequence, query group), key split
// `split` of the S CTAs of a thread-block cluster (cluster rank = split), merged
// through distributed shared memory.  Shared by the attention launch and by the
// persistent layer launch, which runs it as a phase.
#pragma once
#include <cuda.h>

#include "dflow_internal.cuh"
#include "ptx.cuh"

namespace dflow {
namespace t5 {

using namespace ptx;

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// byte offset of (row, 16-byte chunk) inside a tile stored as 64-column boxes
// of [64 rows][128 bytes] with the 128-byte swizzle
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
  return (uint32_t)((chunk >> 3) * 8192 + row * 128 + (((chunk & 7) ^ (row & 7)) << 4));
}

constexpr int T5_ROWS = 128;     // query rows per CTA (MMA M)
// key splits = cluster size S (8 when every 8-CTA cluster is resident at once, else 4); split s
// takes pages s, s + S, ...
constexpr float T5_TAU = 8.0f;   // rescale threshold, log2 units
constexpr int T5_TMEM_COLS = 256;  // O: 128 columns, S: two buffers of 64

// the unit's barriers and per-row results (two P buffers, each with its own
// ready / consumed barrier: a buffer is rewritten only after its previous P V is
// done, so neither barrier can run two phases ahead of its waiter)
template <int KVS>
struct T5Bars {
  uint64_t kv_full[KVS], kv_empty[KVS], s_full[2], s_free[2], p_ready[2], pv_done[2], q_full, drain;
  int n_keys;
  uint32_t tmem;  // the launch's TMEM columns (attention launch)
  float m[T5_ROWS], l[T5_ROWS];
};
// bytes of the unit's shared-memory region: Q [2][128][128 B], KVS K/V stages, 2 P tiles
template <int KVS>
constexpr size_t t5_region_bytes() { return (size_t)2 * T5_ROWS * 128 + (size_t)KVS * 2 * (64 * 128 * 2) + (size_t)2 * T5_ROWS * 128; }

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float *v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
      "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float *v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
      "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
      "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
      "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
// the hardware base-2 exponential (approximate, flushes subnormals; 2^-inf = 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// MN-major operand (row = k index, 64 contiguous n per 128-byte row), 128-byte
// swizzle: 64-element n blocks `lbo` bytes apart, 8-row k groups 1024 bytes apart
__device__ __forceinline__ uint64_t smem_desc_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFF) >> 4);
  d |= (uint64_t)(lbo >> 4) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}
// pages of split s: s, s + S, ...; the ones below n_tiles hold keys
template <int S>
__device__ __forceinline__ int t5_pool_tiles(int n_tiles, int split) {
  return n_tiles > split ? (n_tiles - 1 - split) / S + 1 : 0;
}

// All threads of the CTA call it.  Warp 0 loads (K/V pages and Q with TMA),
// warp 1 issues the MMAs, warps 2-5 run the softmax (thread = query row), other
// warps only take part in the barriers.  `base`: a 1024-byte-aligned region of
// t5_region_bytes<KVS>() bytes; tmem: 256 allocated columns.  dep: the launch
// dependency of Q and the block's K/V rows, or null when already satisfied.
template <bool BLOCK, int S, int KVS, int NT>
__device__ __forceinline__ void t5_unit(const CUtensorMap *tm, const CUtensorMap *tq, const Dims &D, const AttnArgs &a,
                                        int q_tma, uint8_t *base, T5Bars<KVS> &sm, uint32_t tmem, int kvh, int b,
                                        int qg, int split, const Dep *dep, int *status) {
  constexpr int HD = 128, TILE = 64 * HD * 2;  // one K or V page tile: 16 KB
  constexpr int PBUF = T5_ROWS * 128;          // one P tile: [128 rows][64 keys] bf16
  uint8_t *qs = base;                          // [2 boxes][128 rows][128 B]
  uint8_t *ring = qs + 2 * T5_ROWS * 128;      // [stage][K | V]
  uint8_t *ps = ring + KVS * 2 * TILE;         // [2][P tile]
  float *o_sm = reinterpret_cast<float *>(ring);  // [128][128] fp32 after the key loop
  static_assert(KVS * 2 * TILE >= T5_ROWS * 128 * 4, "the K/V ring holds the split's O rows for the merge");

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = D.hq / D.hkv, R = D.R, QR = R * G, row0 = qg * T5_ROWS;
  const int *pt = a.page_table + (size_t)b * D.pages_per_seq;
  const uint64_t pol = policy_evict_first();

  // Before the dependency wait (so that a CTA started early does its set-up and
  // first copies while the previous launch finishes): the key count, and the
  // K/V pages that hold only keys from before this round's block.  Those were
  // written by kernels that finished before the small kernel that heads this
  // chain of launches began (each small kernel waits for its predecessor's
  // completion before its dependents may start), as were the key counts; the
  // page table is the caller's.  Q and the pages with the block's own rows,
  // written by the projection just before, are read after the wait.
  int pg = 0, n_pre = 0, n_early = 0;
  // keys of the sequence, never past its page-table row (a state that fails the
  // round's checks sets the status, but every CTA of a cluster still runs the unit)
  const int nk = min(a.causal ? a.kvlen[b] : a.seq_len[b] - 1, D.pages_per_seq * 64);
  auto issue_page = [&](int it, int page) {  // warp 0, lane 0: page tile `page` into stage it
    uint8_t *kt = ring + (size_t)it * 2 * TILE, *vt = kt + TILE;
    const int rk = ((page * 2 + 0) * D.hkv + kvh) * 64, rv = ((page * 2 + 1) * D.hkv + kvh) * 64;
    mbar_expect_tx(&sm.kv_full[it], 2 * TILE);
    tma_load_2d(kt, tm, 0, rk, &sm.kv_full[it], pol);
    tma_load_2d(kt + 8192, tm, 64, rk, &sm.kv_full[it], pol);
    tma_load_2d(vt, tm, 0, rv, &sm.kv_full[it], pol);
    tma_load_2d(vt + 8192, tm, 64, rv, &sm.kv_full[it], pol);
  };
  if (warp == 0) {
    // page ids of this split's first 32 pages
    const int t = split + S * lane;
    pg = t < D.pages_per_seq ? __ldg(pt + t) : 0;
    const int n_old = a.causal ? nk - R : nk;  // pool keys older than this round's block
    n_pre = min(t5_pool_tiles<S>((nk + 63) / 64, split), KVS);
    while (n_early < n_pre && (split + S * n_early + 1) * 64 <= n_old) ++n_early;
    if (lane == 0) {
      prefetch_tensormap(tm);
      if (q_tma) prefetch_tensormap(tq);
      for (int s = 0; s < KVS; ++s) {
        mbar_init(&sm.kv_full[s], 1);
        mbar_init(&sm.kv_empty[s], 1);
      }
      for (int i = 0; i < 2; ++i) {
        mbar_init(&sm.s_full[i], 1);
        mbar_init(&sm.s_free[i], 4);
        mbar_init(&sm.pv_done[i], 1);
        mbar_init(&sm.p_ready[i], 4);
      }
      mbar_init(&sm.q_full, q_tma ? 1 : 4);
      mbar_init(&sm.drain, 1);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      sm.n_keys = nk;
    }
    for (int it = 0; it < n_early; ++it) {
      const int page = __shfl_sync(0xffffffffu, pg, it);
      if (lane == 0) issue_page(it, page);
    }
  }
  // without the Q map every softmax thread loads its own query row: then every
  // thread is ordered after the wait by the barrier below
  if (!q_tma && threadIdx.x == 0 && dep) dep_wait(*dep, status);
  tc_fence_before();
  __syncthreads();  // barriers and the key count are in place
  tc_fence_after();
  const uint32_t t_o = tmem, t_s = tmem + 128;
  const int n_keys = sm.n_keys;
  const int n_tiles = (n_keys + 63) / 64;
  const int Tp = t5_pool_tiles<S>(n_tiles, split);
  const int T = Tp + ((BLOCK && split == S - 1) ? 1 : 0);

  if (warp == 0) {
    // the projection's outputs: Q, then the first pages that hold block rows
    if (lane == 0) {
      if (q_tma && dep) dep_wait(*dep, status);
      if (dep && dep->wait) fence_proxy_async_global();  // rows just written by the projection, read by TMA
      if (q_tma) {
        const uint32_t qbytes = (uint32_t)(R * G * 128);
        mbar_expect_tx(&sm.q_full, 2 * qbytes);
        tma_load_3d(qs, tq, 0, kvh * G, b * R, &sm.q_full);
        tma_load_3d(qs + T5_ROWS * 128, tq, 64, kvh * G, b * R, &sm.q_full);
      }
    }
    for (int it = n_early; it < n_pre; ++it) {
      const int page = __shfl_sync(0xffffffffu, pg, it);
      if (lane == 0) issue_page(it, page);
    }
    __syncwarp();  // the other lanes read the projection's outputs (block rows) after lane 0's wait
  }

  if (warp == 0) {
    // ---------------- producer: the remaining K/V pages ----------------
    int n_issued = n_pre;
    for (int it = n_pre; it < T; ++it) {
      const int stage = it % KVS;
      const uint32_t ph = (it / KVS) & 1;
      if ((it & 31) == 0) {
        const int t = split + S * (it + lane);
        pg = (it + lane < Tp) ? pt[t] : 0;
      }
      const int page = __shfl_sync(0xffffffffu, pg, it & 31);
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&sm.kv_empty[stage], ph ^ 1) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) {
        if (lane == 0) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
        break;
      }
      uint8_t *kt = ring + (size_t)stage * 2 * TILE, *vt = kt + TILE;
      if (it < Tp) {
        if (lane == 0) {
          const int rk = ((page * 2 + 0) * D.hkv + kvh) * 64, rv = ((page * 2 + 1) * D.hkv + kvh) * 64;
          mbar_expect_tx(&sm.kv_full[stage], 2 * TILE);
          tma_load_2d(kt, tm, 0, rk, &sm.kv_full[stage], pol);
          tma_load_2d(kt + 8192, tm, 64, rk, &sm.kv_full[stage], pol);
          tma_load_2d(vt, tm, 0, rv, &sm.kv_full[stage], pol);
          tma_load_2d(vt + 8192, tm, 64, rv, &sm.kv_full[stage], pol);
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
        fence_async_smem();  // generic-proxy writes read by the tensor cores
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.kv_full[stage]);
      }
      n_issued = it + 1;
    }
    // every fill of the last KVS has landed before the CTA may exit
    if (lane == 0) {
      for (int it = n_issued > KVS ? n_issued - KVS : 0; it < n_issued; ++it)
        if (!mbar_wait(&sm.kv_full[it % KVS], (uint32_t)((it / KVS) & 1)))
          set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
      if (q_tma && !mbar_wait(&sm.q_full, 0)) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t ID_S = (1u << 4) | (1u << 7) | (1u << 10) | ((64u >> 3) << 17) | ((128u >> 4) << 24);
      constexpr uint32_t ID_PV =
          (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((128u >> 3) << 17) | ((128u >> 4) << 24);
      bool ok = mbar_wait(&sm.q_full, 0);
      const uint32_t qa = smem_u32(qs), pa = smem_u32(ps);
      auto pv = [&](int j) -> bool {
        if (!mbar_wait(&sm.p_ready[j & 1], (uint32_t)((j >> 1) & 1))) return false;
        tc_fence_after();
        const uint32_t vt = smem_u32(ring + (size_t)(j % KVS) * 2 * TILE + TILE);
        const uint32_t pj = pa + (uint32_t)(j & 1) * PBUF;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_bf16(t_o, smem_desc(pj + kk * 32), smem_desc_mn(vt + kk * 2048, 8192), ID_PV, (j > 0 || kk > 0) ? 1u : 0u);
        mma_commit(&sm.kv_empty[j % KVS]);
        mma_commit(&sm.pv_done[j & 1]);
        return true;
      };
      for (int i = 0; i < T && ok; ++i) {
        const int stage = i % KVS, buf = i & 1;
        if (!mbar_wait(&sm.kv_full[stage], (uint32_t)((i / KVS) & 1)) ||
            !mbar_wait(&sm.s_free[buf], (uint32_t)(((i >> 1) & 1) ^ 1))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t kt = smem_u32(ring + (size_t)stage * 2 * TILE);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk >> 2) * 8192 + (kk & 3) * 32;
          mma_bf16(t_s + buf * 64, smem_desc(qa + (kk >> 2) * 16384 + (kk & 3) * 32), smem_desc(kt + off), ID_S,
                   kk > 0 ? 1u : 0u);
        }
        mma_commit(&sm.s_full[buf]);
        if (i > 0 && !pv(i - 1)) ok = false;
      }
      if (ok && T > 0) ok = pv(T - 1);
      if (!ok) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
      mma_commit(&sm.drain);
      if (!mbar_wait(&sm.drain, 0)) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
    }
    __syncwarp();
  } else if (warp < 6) {
    // ---------------- softmax warps: thread = query row ----------------
    const int sub = warp & 3, row = sub * 32 + lane;
    const uint32_t lane_off = (uint32_t)(sub * 32) << 16;
    const int qr = row0 + row;
    const bool valid = qr < QR;
    const int qpos = valid ? a.pos[b * R + qr / G] : -1;
    if (!q_tma) {
      // this row of Q into the two 64-dim boxes (128-byte swizzle)
      const bf16 *q = static_cast<const bf16 *>(a.q);
      uint4 v[16];
      if (valid) {
        const uint4 *src = reinterpret_cast<const uint4 *>(q + ((size_t)(b * R + qr / G) * D.hq + kvh * G + qr % G) * HD);
#pragma unroll
        for (int c = 0; c < 16; ++c) v[c] = __ldg(src + c);
      } else {
#pragma unroll
        for (int c = 0; c < 16; ++c) v[c] = make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int c = 0; c < 16; ++c)
        *reinterpret_cast<uint4 *>(qs + (c >> 3) * (T5_ROWS * 128) + row * 128 + (((c & 7) ^ (row & 7)) << 4)) = v[c];
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.q_full);
    }
    // keys this row may see: pool keys [0, vis_pool) (causal: up to its own
    // position), block rows [0, vis_blk); rows past the group see nothing
    const bool live = valid && qpos >= 0;
    const int vis_pool = !live ? 0 : (a.causal ? min(n_keys, qpos + 1) : n_keys);
    const int vis_blk = live ? R : 0;
    const float sl2 = 1.4426950408889634f * rsqrtf((float)HD);
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    auto wait_all = [&](uint64_t *bar, uint32_t parity) -> bool {
      int w_ok = 1;
      if (lane == 0) w_ok = mbar_wait(bar, parity) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w_ok, 0)) return false;
      mbar_wait(bar, parity);  // completed: every lane observes it
      return true;
    };
    for (int i = 0; i < T; ++i) {
      const int buf = i & 1, stage = i % KVS;
      const bool blk = i >= Tp;
      const int tile = split + S * i;
      if (!wait_all(&sm.s_full[buf], (uint32_t)((i >> 1) & 1))) { ok = false; break; }
      tc_fence_after();
      float s[64];
      tmem_ld32(t_s + lane_off + buf * 64, s);
      tmem_ld32(t_s + lane_off + buf * 64 + 32, s + 32);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.s_free[buf]);
      // raw scores; only a tile that crosses this row's limit is masked
      const int lim_t = blk ? vis_blk : vis_pool - tile * 64;
      if (lim_t < 64) {
#pragma unroll
        for (int j = 0; j < 64; ++j) s[j] = j < lim_t ? s[j] : -INFINITY;
      }
      // row max in four independent chains; the positive scale commutes with max
      float m4[4] = {s[0], s[1], s[2], s[3]};
#pragma unroll
      for (int j = 4; j < 64; j += 4) {
        m4[0] = fmaxf(m4[0], s[j]);
        m4[1] = fmaxf(m4[1], s[j + 1]);
        m4[2] = fmaxf(m4[2], s[j + 2]);
        m4[3] = fmaxf(m4[3], s[j + 3]);
      }
      const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * sl2;
      const bool need = mx > m_used + T5_TAU || (m_used == -INFINITY && mx > -INFINITY);
      const float m_new = need ? mx : m_used;
      if (i > 0 && __any_sync(0xffffffffu, need)) {
        // rescale O: it must hold tiles < i (the P V of tile i - 1 is done)
        if (!wait_all(&sm.pv_done[(i - 1) & 1], (uint32_t)(((i - 1) >> 1) & 1))) { ok = false; break; }
        tc_fence_after();
        const float corr = need ? (m_used == -INFINITY ? 0.f : exp2f(m_used - m_new)) : 1.f;
        float o[32];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          tmem_ld32(t_o + lane_off + c * 32, o);
#pragma unroll
          for (int j = 0; j < 32; ++j) o[j] *= corr;
          tmem_st32(t_o + lane_off + c * 32, o);
        }
        l *= corr;
      }
      m_used = m_new;
      // the P buffer of tile i - 2 is free once its P V is done
      if (i > 1 && !wait_all(&sm.pv_done[buf], (uint32_t)(((i - 2) >> 1) & 1))) { ok = false; break; }
      // P = 2^(s * scale - m) (bf16) into the 128-byte-swizzled operand tile;
      // masked scores are -inf and give 0 (a row with nothing visible yet has
      // only masked scores, so the offset does not matter there)
      const float nm = m_used == -INFINITY ? 0.f : -m_used;
      uint8_t *pb = ps + buf * PBUF;
      float l4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        float p[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          p[e] = ex2_approx(fmaf(s[c * 8 + e], sl2, nm));
          l4[e & 3] += p[e];
        }
        uint4 u;
        u.x = pack_bf16(p[0], p[1]);
        u.y = pack_bf16(p[2], p[3]);
        u.z = pack_bf16(p[4], p[5]);
        u.w = pack_bf16(p[6], p[7]);
        *reinterpret_cast<uint4 *>(pb + row * 128 + (((c) ^ (row & 7)) << 4)) = u;
      }
      l += (l4[0] + l4[1]) + (l4[2] + l4[3]);
      if (!blk && tile * 64 + 64 > n_keys) {
        // V rows past the context: zero them so stale bytes never meet P = 0
        uint8_t *vt = ring + (size_t)stage * 2 * TILE + TILE;
        const int z0 = max(n_keys - tile * 64, 0);
        for (int e = row; e < (64 - z0) * 16; e += T5_ROWS) {
          const int j = z0 + e / 16, c = e % 16;
          *reinterpret_cast<uint4 *>(vt + swz(j, c)) = make_uint4(0, 0, 0, 0);
        }
      }
      fence_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.p_ready[buf]);
    }
    if (!ok && lane == 0) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
    // ---- this split's unnormalised O row, max and sum
    float o[128];
    if (ok && T > 0) {
      if (wait_all(&sm.pv_done[(T - 1) & 1], (uint32_t)(((T - 1) >> 1) & 1))) {
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(t_o + lane_off + c * 32, o + c * 32);
      } else {
        if (lane == 0) set_status(status, DFLOW_ERR_DEVICE_TIMEOUT);
#pragma unroll
        for (int j = 0; j < 128; ++j) o[j] = 0.f;
        m_used = -INFINITY;
        l = 0.f;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 128; ++j) o[j] = 0.f;
      m_used = -INFINITY;
      l = 0.f;
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");  // (B) every softmax warp has drained TMEM
    // the ring is reused for O once every copy and MMA has finished: wait for (A)
    __syncthreads();  // (A)
    // 16-byte chunks of a row XOR-permuted by (row & 7): eight consecutive rows
    // hit distinct banks
#pragma unroll
    for (int j = 0; j < 32; ++j)
      *reinterpret_cast<float4 *>(o_sm + row * HD + ((j ^ (row & 7)) << 2)) =
          make_float4(o[4 * j], o[4 * j + 1], o[4 * j + 2], o[4 * j + 3]);
    sm.m[row] = m_used;
    sm.l[row] = l;
  }
  if (warp < 2 || warp >= 6) __syncthreads();  // (A) for the producer, MMA and other warps

  // ---- merge the splits of this cluster: CTA `split` finishes a slice of the valid rows
  __syncthreads();
  cluster_sync();
  const int n_valid = min(QR - row0, T5_ROWS);
  const int rpc = (n_valid + S - 1) / S;
  const int r_lo = split * rpc, nr = max(min(r_lo + rpc, n_valid) - r_lo, 0);
  const int units = nr * (HD / 4);
  // one round trip of remote loads: thread t < S nr takes (row t / S, split t % S)'s
  // max and sum; every thread takes the S split partials of up to two
  // (row, 4-dim chunk) units
  float mv = -INFINITY, lv = 0.f;
  if (threadIdx.x < nr * S) {
    const int rr = r_lo + threadIdx.x / S, sp = threadIdx.x % S;
    mv = ld_dsmem_f32(mapa(smem_u32(sm.m + rr), (uint32_t)sp));
    lv = ld_dsmem_f32(mapa(smem_u32(sm.l + rr), (uint32_t)sp));
  }
  float4 x[2][S];
  auto load_units = [&](int u0) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int u = u0 + h * NT;
      if (u < units) {
        const int rr = r_lo + u / (HD / 4), c4 = u % (HD / 4);
        const int off = rr * HD + ((c4 ^ (rr & 7)) << 2);
#pragma unroll
        for (int sp = 0; sp < S; ++sp) x[h][sp] = ld_dsmem_f4(mapa(smem_u32(o_sm + off), (uint32_t)sp));
      }
    }
  };
  load_units(threadIdx.x);
  // merge weight of (row, split): 2^(m - M) / sum_s 2^(m_s - M) l_s over the S
  // lanes of the row (the Q tile is free now and holds them)
  float *wsm = reinterpret_cast<float *>(qs);  // [rpc][S]
  {
    float M = mv;
#pragma unroll
    for (int o = 1; o < S; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    const float c = mv == -INFINITY ? 0.f : exp2f(mv - M);
    float L = c * lv;
#pragma unroll
    for (int o = 1; o < S; o <<= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
    if (threadIdx.x < nr * S) wsm[threadIdx.x] = L > 0.f ? c / L : 0.f;
  }
  __syncthreads();
  bf16 *out = static_cast<bf16 *>(a.out);
  for (int u0 = threadIdx.x; u0 < units; u0 += 2 * NT) {
    if (u0 != (int)threadIdx.x) load_units(u0);  // units past the first two per thread (a full 128-row group)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int u = u0 + h * NT;
      if (u >= units) continue;
      const int rl = u / (HD / 4), d4 = (u % (HD / 4)) * 4, q_r = row0 + r_lo + rl;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int sp = 0; sp < S; ++sp) {
        const float c = wsm[rl * S + sp];
        acc.x += c * x[h][sp].x;
        acc.y += c * x[h][sp].y;
        acc.z += c * x[h][sp].z;
        acc.w += c * x[h][sp].w;
      }
      const int i = q_r / G, head = kvh * G + q_r % G;
      bf16 *dst = out + ((size_t)(b * R + i) * D.hq + head) * HD + d4;
      *reinterpret_cast<__nv_bfloat162 *>(dst) = __floats2bfloat162_rn(acc.x, acc.y);
      *reinterpret_cast<__nv_bfloat162 *>(dst + 2) = __floats2bfloat162_rn(acc.z, acc.w);
    }
  }
  cluster_sync();  // peers may still read this CTA's shared memory until here
}

}  // namespace t5
}  // namespace dflow
