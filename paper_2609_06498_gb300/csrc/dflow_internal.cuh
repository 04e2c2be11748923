// Internal declarations shared by the translation units of libdflow.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dflow.h"

namespace dflow {

typedef __nv_bfloat16 bf16;

// ---------------------------------------------------------------------------
// element conversions
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

__device__ __forceinline__ float silu_f(float x) { return x / (1.0f + expf(-x)); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
// (value, index) max with ties to the lowest index
__device__ __forceinline__ void argmax_merge(float &v, int &i, float v2, int i2) {
  if (v2 > v || (v2 == v && i2 < i)) { v = v2; i = i2; }
}
__device__ __forceinline__ void warp_argmax(float &v, int &i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float v2 = __shfl_xor_sync(0xffffffffu, v, o);
    int i2 = __shfl_xor_sync(0xffffffffu, i, o);
    argmax_merge(v, i, v2, i2);
  }
}

// Programmatic dependent launch: the next kernel of the stream may start as
// soon as every CTA of this one has begun; griddepcontrol.wait blocks until the
// previous kernel has finished and its writes are visible.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_entry() {
  pdl_wait();
  pdl_trigger();
}

// first device-detected error wins
__device__ __forceinline__ void set_status(int *status, int code) { atomicCAS(status, 0, code); }

// launch with programmatic stream serialisation (the kernel must begin with pdl_entry)
template <typename Kern, typename... Args>
inline cudaError_t klaunch(Kern kernel, dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Completion counters between consecutive launches of the tensor-core kernels
// (GEMM, attention).  Every CTA of a launch adds 1 to the launch's counter
// (release) once all its global writes are done; a launch that directly
// follows such a launch acquires that counter until it reaches the previous
// launch's CTA count, instead of waiting for the previous grid to be torn down.
// Counters are cumulative across launches that share a slot.
struct Dep {
  const unsigned int *wait;  // previous launch's counter, or null: griddepcontrol.wait
  unsigned int wait_n;       // its value once every CTA of the previous launch is done
  unsigned int *signal;      // this launch's counter, or null
};

// Host side of the counters of one handle (its calls are issued in order on one
// stream).  A launch that counts takes the next slot; it waits on the previous
// slot only when the launch right before it counted too (brk() after any other
// launch).  Slots are reused round robin, their expected values accumulating.
constexpr int kDepSlots = 64;
struct DepChain {
  unsigned int *dev = nullptr;          // [kDepSlots] counters in device memory
  unsigned int shadow[kDepSlots] = {};  // value of each counter once every launch so far is done
  int last = -1;                        // slot of the previous launch when it counted, else -1
  int next = 0;
  bool dirty = true;                    // counters and shadow disagree: zero both before use
  Dep take(unsigned int n_ctas) {
    Dep d{};
    if (dev == nullptr) return d;
    if (last >= 0) {
      d.wait = dev + last;
      d.wait_n = shadow[last];
    }
    last = next;
    next = (next + 1) % kDepSlots;
    shadow[last] += n_ctas;
    d.signal = dev + last;
    return d;
  }
  // a counter for completions inside one launch (the chain's last slot is unchanged)
  unsigned int *alloc(unsigned int n, unsigned int *target) {
    if (dev == nullptr) return nullptr;
    const int s = next;
    next = (next + 1) % kDepSlots;
    shadow[s] += n;
    *target = shadow[s];
    return dev + s;
  }
  void brk() { last = -1; }
};

// ---------------------------------------------------------------------------
// GEMM: out[m][n] = sum_k X[m][k] * W[n][k] with a fused epilogue
// ---------------------------------------------------------------------------
enum EpMode {
  EP_STORE_F32 = 0,  // out_f32[m*ldo + n] = acc
  EP_RESID = 1,      // out_f32[m*ldo + n] += acc            (residual stream)
  EP_SWIGLU = 2,     // 128-row groups [64 gate | 64 up] -> out_t[m*ldt + 64g + f] = silu(g) * u
  EP_SILU = 3,       // out_t[m*ldt + n] = silu(acc)
  EP_ARGMAX = 4,     // per 128-row tile: (max, argmax) -> part_val/part_idx[m*n_tiles + tile]
  EP_QKV = 5,        // per 128-row tile = one head: q/k RMSNorm + rotary, q to q_out, k/v to the cache
};

// Targets of the fused Q/K/V epilogue (tensor-core path, head_dim 128).  The
// output rows are nq query heads, then hkv key heads, then hkv value heads.
struct QkvOut {
  int nq, hkv, hq_row;       // q heads in this output; kv heads; q heads per q_out row
  float eps;                 // q/k RMSNorm epsilon
  const float *qn, *kn;      // q/k norm gains [128]
  const float2 *rope;        // [max_ctx][64] (cos, sin)
  const int *pos, *wr;       // per global row: position, cache write allowed
  int row0;                  // global row of output column 0
  int R;                     // rows per sequence
  void *q_out;               // [rows][hq_row][128]
  void *pool;                // one layer of a paged pool (when bk == null)
  const int *page_table;
  int pages_per_seq, page_size, num_pages;
  void *bk, *bv;             // block K/V [rows][hkv][128] (drafter) or null
};

struct EpArgs {
  int mode;
  float *out_f32;
  int ldo;
  void *out_t;
  int ldt;
  float *part_val;
  int *part_idx;
  int n_tiles;
  // input RMSNorm folded into the epilogue: column m is scaled by
  // rsqrt(sum_i in_ss[i*ld_ss + m] * inv_d + eps) (the gain is already in X)
  const float *in_ss;
  int in_ss_n, ld_ss;
  float in_inv_d, in_eps;
  // EP_RESID extras for the updated rows x: squared-norm partial of this
  // tile's 128 features (out_ss[tile*ld_ss + m]), bf16(x * out_gain) and bf16(x)
  float *out_ss;
  void *out_xn;
  int ld_xn;
  const float *out_gain;
  void *out_stash;
  int ld_stash;
  QkvOut qkv;
};

// ---------------------------------------------------------------------------
// decoder dimensions as the kernels see them
// ---------------------------------------------------------------------------
struct Dims {
  int d, hq, hkv, hd, inter, vocab, B, R, page_size, num_pages, max_ctx, pages_per_seq;
  int n_feat;
  float rms_eps, ln_eps;
};

__host__ __device__ __forceinline__ size_t pool_layer_elems(const Dims &D) {
  return (size_t)D.num_pages * 2 * D.hkv * D.page_size * D.hd;
}
// element offset of (page, k|v, kv head, in-page slot) inside one layer of a pool
__host__ __device__ __forceinline__ size_t pool_off(const Dims &D, int page, int kv, int h, int slot) {
  return ((((size_t)page * 2 + kv) * D.hkv + h) * D.page_size + slot) * D.hd;
}

// ---------------------------------------------------------------------------
// launchers (each returns cudaGetLastError())
// ---------------------------------------------------------------------------
cudaError_t gemm_simt(int dtype, const void *W, int N, int K, const void *X, int M, int ldx,
                      const EpArgs &ep, const int *status, cudaStream_t s);

struct AttnArgs {
  const void *q;          // [rows][hq][hd]
  const void *pool;       // one layer of a paged K/V pool
  const int *page_table;  // [batch][pages_per_seq]
  const void *bk, *bv;    // block K/V [rows][hkv][hd] (non-causal mode) or null
  const int *pos;         // [rows] compute position of each row
  const int *seq_len;     // [batch]
  const int *kvlen;       // [batch] causal mode: keys 0..kvlen-1 hold data
  int causal;             // 1: keys 0..pos (paged); 0: context 0..n-2 (paged) + block rows
  int n_splits;
  float *part;            // [rows][hq][n_splits][hd + 2]
  void *out;              // [rows][hq * hd]
  Dep dep;                // completion counters (tcgen05 kernel only)
};
// chain: completion counters of the caller's launch sequence, or null
cudaError_t attention(int dtype, const Dims &D, int batch, const AttnArgs &a, int *status, cudaStream_t s,
                      DepChain *chain = nullptr);
// tensor-core path for bf16 caches with 64-token pages (attn_tc.cu)
bool attention_tc_supported(const Dims &D);
cudaError_t attention_tc(const Dims &D, int batch, const AttnArgs &a, int *status, cudaStream_t s,
                         DepChain *chain = nullptr);

}  // namespace dflow
