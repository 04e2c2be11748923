// Block-query attention on the 5th-generation tensor cores for bf16 caches with
// 128-dim heads and 64-token pages (Sec. 3: the target verifies the whole draft
// block in one pass; the drafter attends to its injected context and to the
// block).
#include <cuda.h>
#include <stdlib.h>

#include "dflow_internal.cuh"
#include "gemm_tc.cuh"
#include "ptx.cuh"
#include "attn_t5.cuh"

namespace dflow {

namespace {

using namespace ptx;
using namespace t5;

constexpr int THREADS = 192;  // warp 0 loads, warp 1 issues MMAs, warps 2-5 run the softmax
// K/V pages in flight: five with 8- and 4-CTA clusters (a split's pages at 2K keys
// and batch 1-4 are then all issued before the dependency wait), four with 2-CTA
// clusters (long contexts at batch 16 measured slightly faster so)
template <int S>
constexpr int t5_kvs() { return S >= 4 ? 5 : 4; }
template <int S>
constexpr size_t t5_smem() { return 1024 + t5_region_bytes<t5_kvs<S>()>() + sizeof(T5Bars<t5_kvs<S>()>); }

// ===========================================================================
// Queries are the MMA's M (padded to 128),
// 64-key pages its N.  Warp 0 streams K/V pages (TMA; split s of the cluster
// takes pages s, s + 8, ...) and the query rows (two 3D TMA boxes that land in
// MMA row order), issuing the first copies right after the dependency wait;
// warp 1 issues S = Q K^T and O += P V into TMEM; warps 2-5 own one query row
// per thread: softmax straight out of TMEM (no shuffles), P to one of two
// shared-memory tiles (so the next page's softmax overlaps this page's P V),
// lazy rescaling of the O row (only when the running max grows by more than
// 2^8), zeroing of V rows past the context in a partial page.  The splits
// merge their (O, max, sum) through distributed shared memory.
// ===========================================================================
// q_tma: the CTA's query rows arrive as two boxes of the 3D map tq over
// [rows][hq][128] (64 dims x G heads x R rows); else each softmax thread loads its row
template <bool BLOCK, int S>
__global__ void __launch_bounds__(THREADS, 1)
k_attn_t5(const __grid_constant__ CUtensorMap tm, const __grid_constant__ CUtensorMap tq, Dims D, AttnArgs a,
          int q_tma, int *status) {
  // runs even after an earlier error (every wait is bounded): the CTAs of a
  // cluster must not disagree on whether to take part in its barriers
  pdl_trigger();
  constexpr int KVS = t5_kvs<S>();
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(dsm) + 1023) & ~(uintptr_t)1023);
  T5Bars<KVS> &sm = *reinterpret_cast<T5Bars<KVS> *>(base + t5_region_bytes<KVS>());
  const int warp = threadIdx.x / 32;
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&sm.tmem)),
                 "r"(T5_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem;
  t5_unit<BLOCK, S, KVS, THREADS>(&tm, &tq, D, a, q_tma, base, sm, tmem, (int)blockIdx.x, (int)blockIdx.y,
                                  (int)blockIdx.z / S, (int)blockIdx.z % S, &a.dep, status);
  if (threadIdx.x == 0) dep_signal(a.dep);  // every global write of this CTA is done
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(T5_TMEM_COLS) : "memory");
  }
}

// resident clusters of S CTAs of k_attn_t5<BLOCK, S> (0 when the query fails)
template <bool BLOCK, int S>
int t5_resident_clusters() {
  constexpr size_t smem = t5_smem<S>();
  static int n = -1;
  if (n >= 0) return n;
  n = 0;
  if (cudaFuncSetAttribute(k_attn_t5<BLOCK, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) ==
      cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = S;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, k_attn_t5<BLOCK, S>, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();
  return n;
}

template <bool BLOCK, int S>
cudaError_t launch_t5(const CUtensorMap &tm, const Dims &D, int batch, AttnArgs a, int *status, cudaStream_t s,
                      DepChain *chain) {
  constexpr size_t smem = t5_smem<S>();
  const int G = D.hq / D.hkv;
  const int qgroups = (D.R * G + T5_ROWS - 1) / T5_ROWS;
  // one group of query rows: they arrive as two 3D boxes (64 dims x G heads x R rows)
  CUtensorMap tq{};
  const int q_tma = (qgroups == 1 && tensor_map_3d(&tq, a.q, D.hd, D.hq, batch * D.R, G, D.R)) ? 1 : 0;
  a.dep = chain ? chain->take((unsigned)(D.hkv * batch * S * qgroups)) : Dep{};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(D.hkv, batch, S * qgroups);
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = 1;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = S;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, k_attn_t5<BLOCK, S>, tm, tq, D, a, q_tma, status);
}

// eight key splits per (kv head, sequence, query group) when every eight-CTA
// cluster is resident at once, else four when those all are, else two: a CTA's
// fixed costs (set-up, first pages, the cluster merge) are paid by fewer CTAs, and
// smaller clusters leave fewer SMs of a GPC idle.  (One split per unit measured
// faster on equal contexts but slower on ragged ones: the longest sequence's
// CTA then sets the launch time.)
template <bool BLOCK>
cudaError_t launch_t5_any(const CUtensorMap &tm, const Dims &D, int batch, const AttnArgs &a, int *status,
                          cudaStream_t s, DepChain *chain) {
  const int G = D.hq / D.hkv;
  const long long units = (long long)D.hkv * batch * ((D.R * G + T5_ROWS - 1) / T5_ROWS);
  const int r8 = t5_resident_clusters<BLOCK, 8>(), r4 = t5_resident_clusters<BLOCK, 4>();
  if (r8 < 1) return cudaErrorInvalidValue;
  if (units <= r8) return launch_t5<BLOCK, 8>(tm, D, batch, a, status, s, chain);
  if (units <= r4) return launch_t5<BLOCK, 4>(tm, D, batch, a, status, s, chain);
  // (the query also sets the 2-split kernel's shared-memory limit)
  if (t5_resident_clusters<BLOCK, 2>() < 1) return cudaErrorInvalidValue;
  return launch_t5<BLOCK, 2>(tm, D, batch, a, status, s, chain);
}

}  // namespace

bool attention_tc_supported(const Dims &D) { return D.page_size == 64 && D.hd == 128; }

cudaError_t attention_tc(const Dims &D, int batch, const AttnArgs &a, int *status, cudaStream_t s,
                         DepChain *chain) {
  CUtensorMap tm;
  const int rows = D.num_pages * 2 * D.hkv * D.page_size;
  if (!attention_tc_supported(D) || !tensor_map(&tm, a.pool, rows, D.hd, D.hd, 64)) return cudaErrorInvalidValue;
  return a.causal ? launch_t5_any<false>(tm, D, batch, a, status, s, chain)
                  : launch_t5_any<true>(tm, D, batch, a, status, s, chain);
}

}  // namespace dflow
