// CUDA-core GEMM with fused epilogues for the fp32 parity model (bf16 models
// run every projection on the tensor-core kernels).
//
// out[m][n] = sum_k X[m][k] * W[n][k]; W row-major [N][K] (the layout of every
// projection of the Qwen3 layer), X row-major [M][ldx].  A CTA computes a tile
// of 128 output features x 16 rows; K is walked in chunks of 32.
#include "dflow_internal.cuh"

namespace dflow {

namespace {

constexpr int TN = 128, TM = 16, TK = 32;

template <typename T, int EP>
__global__ void __launch_bounds__(256)
k_gemm_simt(const T *__restrict__ W, const T *__restrict__ X, int N, int K, int M, int ldx,
            EpArgs ep, const int *__restrict__ status) {
  pdl_entry();
  if (*status) return;
  __shared__ float Ws[TN][TK + 1];
  __shared__ float Xs[TM][TK + 1];
  __shared__ float Cs[TM][TN + 1];
  const int n0 = blockIdx.x * TN, m0 = blockIdx.y * TM;
  const int tid = threadIdx.x, tm = tid / 16, tn = tid % 16;
  float acc[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) acc[j] = 0.f;

  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int e = tid; e < TN * TK; e += 256) {
      const int r = e / TK, c = e % TK, n = n0 + r;
      Ws[r][c] = (n < N) ? to_f(W[(size_t)n * K + k0 + c]) : 0.f;
    }
    for (int e = tid; e < TM * TK; e += 256) {
      const int r = e / TK, c = e % TK, m = m0 + r;
      Xs[r][c] = (m < M) ? to_f(X[(size_t)m * ldx + k0 + c]) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int k = 0; k < TK; ++k) {
      const float xv = Xs[tm][k];
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = fmaf(xv, Ws[tn + 16 * j][k], acc[j]);
    }
    __syncthreads();
  }

  const int m = m0 + tm;
  if constexpr (EP == EP_STORE_F32 || EP == EP_RESID || EP == EP_SILU) {
    if (m >= M) return;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int n = n0 + tn + 16 * j;
      if (n >= N) continue;
      if constexpr (EP == EP_STORE_F32) ep.out_f32[(size_t)m * ep.ldo + n] = acc[j];
      if constexpr (EP == EP_RESID) ep.out_f32[(size_t)m * ep.ldo + n] += acc[j];
      if constexpr (EP == EP_SILU) reinterpret_cast<T *>(ep.out_t)[(size_t)m * ep.ldt + n] = from_f<T>(silu_f(acc[j]));
    }
  } else {
#pragma unroll
  for (int j = 0; j < 8; ++j) Cs[tm][tn + 16 * j] = acc[j];
  __syncthreads();
  if (EP == EP_SWIGLU) {
    for (int e = tid; e < TM * 64; e += 256) {
      const int r = e / 64, f = e % 64, mm = m0 + r;
      if (mm < M && n0 + 64 + f < N)
        reinterpret_cast<T *>(ep.out_t)[(size_t)mm * ep.ldt + blockIdx.x * 64 + f] =
            from_f<T>(silu_f(Cs[r][f]) * Cs[r][64 + f]);
    }
  } else if (EP == EP_ARGMAX) {
    const int warp = tid / 32, lane = tid % 32;
    for (int r = warp; r < TM; r += 8) {
      const int mm = m0 + r;
      float v = -INFINITY;
      int idx = 0x7fffffff;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int n = n0 + lane + 32 * c;
        if (n < N) argmax_merge(v, idx, Cs[r][lane + 32 * c], n);
      }
      warp_argmax(v, idx);
      if (lane == 0 && mm < M) {
        ep.part_val[(size_t)mm * ep.n_tiles + blockIdx.x] = v;
        ep.part_idx[(size_t)mm * ep.n_tiles + blockIdx.x] = idx;
      }
    }
  }
  }
}

template <typename T>
cudaError_t launch(const void *W, int N, int K, const void *X, int M, int ldx, const EpArgs &ep,
                   const int *status, cudaStream_t s) {
  dim3 grid((N + TN - 1) / TN, (M + TM - 1) / TM);
  const T *w = static_cast<const T *>(W);
  const T *x = static_cast<const T *>(X);
  switch (ep.mode) {
    case EP_STORE_F32: klaunch(k_gemm_simt<T, EP_STORE_F32>, grid, 256, 0, s, w, x, N, K, M, ldx, ep, status); break;
    case EP_RESID: klaunch(k_gemm_simt<T, EP_RESID>, grid, 256, 0, s, w, x, N, K, M, ldx, ep, status); break;
    case EP_SWIGLU: klaunch(k_gemm_simt<T, EP_SWIGLU>, grid, 256, 0, s, w, x, N, K, M, ldx, ep, status); break;
    case EP_SILU: klaunch(k_gemm_simt<T, EP_SILU>, grid, 256, 0, s, w, x, N, K, M, ldx, ep, status); break;
    case EP_ARGMAX: klaunch(k_gemm_simt<T, EP_ARGMAX>, grid, 256, 0, s, w, x, N, K, M, ldx, ep, status); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t gemm_simt(int dtype, const void *W, int N, int K, const void *X, int M, int ldx,
                      const EpArgs &ep, const int *status, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  if (K % TK != 0 || dtype != DFLOW_F32) return cudaErrorInvalidValue;
  return launch<float>(W, N, K, X, M, ldx, ep, status, s);
}

}  // namespace dflow
