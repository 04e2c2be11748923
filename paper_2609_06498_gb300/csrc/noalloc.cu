// Greedy-token entry point that allocates nothing.
//
// Some callers cannot allocate device memory at all: code that runs inside a
// caller-managed memory pool or arena with a fixed budget, a plugin whose host
// framework owns every allocation, or a process that must not grow its memory
// footprint after start-up.  For them dflow_greedy_tokens_noalloc runs the LM
// head with the fused argmax (the same tensor-core kernel chain the round uses)
// with its per-tile partial results in a scratch array compiled into this
// library instead of in a caller workspace.
//
// The scratch is a file-scope __device__ array of about 1 MiB.  It becomes
// device memory when the library's GPU code is loaded on a device and stays
// there until the process exits.  Under CUDA's default lazy module loading
// that happens at the first use on each device: for this entry point, its
// first call there, which looks the array's address up with
// cudaGetSymbolAddress (host code cannot use the array's name as a device
// address) and keeps it.  So the first call on each device is the one that
// grows the device footprint: make it at set-up, before any fixed-budget
// window and before any stream capture (or set CUDA_MODULE_LOADING=EAGER,
// which places the array when the library is loaded).  That lookup is done
// once per device under a lock, so concurrent first calls from several host
// threads are safe.  All calls share the one array and it keeps the last
// call's contents: the status word is cleared at every call, and calls whose
// work overlaps on the GPU race on the array.  The stream must belong to the
// current device.
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>

#include "dflow_internal.cuh"
#include "gemm_tc.cuh"

namespace {

using namespace dflow;

constexpr int NA_MAX_ROWS = 64;      // hidden rows per call
constexpr int NA_MAX_TILES = 2048;   // 128-token vocabulary tiles: vocab <= 262144
constexpr int NA_MAX_DEVICES = 64;

struct NaScratch {
  float val[NA_MAX_ROWS * NA_MAX_TILES];  // per (row, tile) best logit
  int idx[NA_MAX_ROWS * NA_MAX_TILES];    // per (row, tile) token of that logit
  int status[64];                          // device status word of the call
};

static __device__ __align__(256) NaScratch g_na_scratch;

// per device: the array's address and the SM count, published together (the
// address is stored last, with release order, after the lookup under g_na_mu)
struct NaDevice {
  std::atomic<NaScratch *> addr{nullptr};
  int sms = 0;
};
NaDevice g_na_dev[NA_MAX_DEVICES];
std::mutex g_na_mu;

// the array's address on device `dev` (current), looked up once; null on failure
// (*code says why)
NaScratch *na_scratch(int dev, dflow_status *code) {
  NaDevice &nd = g_na_dev[dev];
  NaScratch *p = nd.addr.load(std::memory_order_acquire);
  if (p != nullptr) return p;
  std::lock_guard<std::mutex> lock(g_na_mu);
  p = nd.addr.load(std::memory_order_relaxed);
  if (p != nullptr) return p;
  int major = 0, minor = 0, sms = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    *code = DFLOW_ERR_CUDA;
    return nullptr;
  }
  if (major != 10 || minor != 3) {
    *code = DFLOW_ERR_UNSUPPORTED;
    return nullptr;
  }
  void *a = nullptr;
  if (cudaGetSymbolAddress(&a, g_na_scratch) != cudaSuccess || a == nullptr) {
    *code = DFLOW_ERR_CUDA;
    return nullptr;
  }
  nd.sms = sms;
  p = static_cast<NaScratch *>(a);
  nd.addr.store(p, std::memory_order_release);
  return p;
}

__global__ void k_na_clear(int *status) { status[0] = 0; }

// token[r] = argmax over the per-tile partials (ties: lowest id)
__global__ void k_na_reduce(const float *__restrict__ pv, const int *__restrict__ pi, int n_tiles, int rows,
                            int *__restrict__ tokens, const int *__restrict__ status) {
  const int r = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32, lane = threadIdx.x % 32;
  if (r >= rows) return;
  float v = -INFINITY;
  int idx = 0x7fffffff;
  for (int t = lane; t < n_tiles; t += 32) argmax_merge(v, idx, pv[(size_t)r * n_tiles + t], pi[(size_t)r * n_tiles + t]);
  warp_argmax(v, idx);
  if (lane == 0) tokens[r] = *status ? -1 : idx;
}

}  // namespace

extern "C" dflow_status dflow_greedy_tokens_noalloc(const void *lm_head, int32_t vocab, int32_t d, const void *hidden,
                                                    int32_t rows, int32_t *tokens, void *stream) {
  if (!lm_head || !hidden || !tokens || vocab < 1 || d < 1 || rows < 1) return DFLOW_ERR_INVALID_ARG;
  if (rows > NA_MAX_ROWS || (vocab + 127) / 128 > NA_MAX_TILES) return DFLOW_ERR_INVALID_ARG;
  if (d % 64 != 0) return DFLOW_ERR_UNSUPPORTED;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= NA_MAX_DEVICES) return DFLOW_ERR_UNSUPPORTED;
  if (stream != nullptr) {
    int sdev = -1;
    if (cudaStreamGetDevice(static_cast<cudaStream_t>(stream), &sdev) != cudaSuccess) return DFLOW_ERR_CUDA;
    if (sdev != dev) return DFLOW_ERR_INVALID_ARG;
  }
  dflow_status code = DFLOW_OK;
  NaScratch *S = na_scratch(dev, &code);
  if (S == nullptr) return code;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int n_tiles = (vocab + 127) / 128;
  k_na_clear<<<1, 1, 0, s>>>(S->status);
  if (cudaGetLastError() != cudaSuccess) return DFLOW_ERR_CUDA;
  TcWorkspace w;
  w.sm_count = g_na_dev[dev].sms;
  EpArgs ep{};
  ep.mode = EP_ARGMAX;
  ep.part_val = S->val;
  ep.part_idx = S->idx;
  ep.n_tiles = n_tiles;
  if (gemm_tc(w, lm_head, vocab, d, hidden, rows, d, ep, S->status, s, false) != cudaSuccess) return DFLOW_ERR_CUDA;
  k_na_reduce<<<(rows + 7) / 8, 256, 0, s>>>(S->val, S->idx, n_tiles, rows, tokens, S->status);
  if (cudaGetLastError() != cudaSuccess) return DFLOW_ERR_CUDA;
  return DFLOW_OK;
}
