// Block-query attention against a paged K/V pool (Sec. 3: verification runs
// the target over the whole draft block in one pass; the drafter attends to
// its injected context and to the block).
//
// One CTA owns one (kv head, sequence, key split).  Its queries are the R
// block rows x the G = Hq/Hkv query heads sharing that kv head.  Keys are
// either the paged positions 0..pos (causal, target verify and prefill) or the
// drafter's context positions 0..n-2 followed by the R block rows (no mask).
// Each split writes an unnormalised partial (o, running max m, sum l); a
// second kernel merges the splits.
#include "dflow_internal.cuh"

namespace dflow {

namespace {

constexpr int KT = 32;   // keys per tile
constexpr int QPW = 4;   // query rows per warp per pass
constexpr int QG = 4 * QPW;  // query rows per pass

template <typename T, int HD>
__global__ void __launch_bounds__(128)
k_attn_split(Dims D, AttnArgs a, const int *__restrict__ status) {
  pdl_entry();
  if (*status) return;
  constexpr int DPL = HD / 32;  // dims per lane
  __shared__ float Qs[QG][HD];
  __shared__ float Ks[KT][HD + 1];
  __shared__ float Vs[KT][HD + 1];
  __shared__ int kpos_s[KT];

  const int kvh = blockIdx.x, b = blockIdx.y, split = blockIdx.z;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int G = D.hq / D.hkv, R = D.R, QR = R * G;
  const T *q = static_cast<const T *>(a.q);
  const T *pool = static_cast<const T *>(a.pool);
  const T *bk = static_cast<const T *>(a.bk);
  const T *bv = static_cast<const T *>(a.bv);
  const int *pt = a.page_table + (size_t)b * D.pages_per_seq;
  const float scale = rsqrtf((float)HD);

  int n_paged, n_keys;
  if (a.causal) {
    int mx = 0;
    for (int i = 0; i < R; ++i) mx = max(mx, a.pos[b * R + i]);
    n_paged = mx + 1;
    n_keys = n_paged;
  } else {
    n_paged = a.seq_len[b] - 1;
    n_keys = n_paged + R;
  }
  const int chunk = (n_keys + a.n_splits - 1) / a.n_splits;
  const int k_lo = min(n_keys, split * chunk), k_hi = min(n_keys, k_lo + chunk);

  for (int qb = 0; qb < QR; qb += QG) {
    __syncthreads();
    for (int e = threadIdx.x; e < QG * HD; e += 128) {
      const int r = e / HD, c = e % HD, qr = qb + r;
      float v = 0.f;
      if (qr < QR) {
        const int i = qr / G, h = kvh * G + qr % G;
        v = to_f(q[((size_t)(b * R + i) * D.hq + h) * HD + c]);
      }
      Qs[r][c] = v;
    }
    float m[QPW], l[QPW], o[QPW][DPL];
    int qpos[QPW];
#pragma unroll
    for (int t = 0; t < QPW; ++t) {
      m[t] = -INFINITY;
      l[t] = 0.f;
#pragma unroll
      for (int c = 0; c < DPL; ++c) o[t][c] = 0.f;
      const int qr = qb + warp * QPW + t;
      qpos[t] = qr < QR ? a.pos[b * R + qr / G] : -1;
    }
    for (int kt = k_lo; kt < k_hi; kt += KT) {
      __syncthreads();
      for (int e = threadIdx.x; e < KT * HD; e += 128) {
        const int j = e / HD, c = e % HD, kidx = kt + j;
        float kv = 0.f, vv = 0.f;
        if (kidx < k_hi) {
          if (kidx < n_paged) {
            const int page = pt[kidx / D.page_size], slot = kidx % D.page_size;
            kv = to_f(pool[pool_off(D, page, 0, kvh, slot) + c]);
            vv = to_f(pool[pool_off(D, page, 1, kvh, slot) + c]);
          } else {
            const size_t off = ((size_t)(b * R + (kidx - n_paged)) * D.hkv + kvh) * HD + c;
            kv = to_f(bk[off]);
            vv = to_f(bv[off]);
          }
        }
        Ks[j][c] = kv;
        Vs[j][c] = vv;
      }
      if (threadIdx.x < KT) kpos_s[threadIdx.x] = kt + threadIdx.x;
      __syncthreads();
#pragma unroll
      for (int t = 0; t < QPW; ++t) {
        const int qr = qb + warp * QPW + t;
        if (qr >= QR) break;
        const int kidx = kt + lane;
        bool ok = kidx < k_hi;
        if (a.causal) ok = ok && kpos_s[lane] <= qpos[t];
        float sc = -INFINITY;
        if (ok) {
          float acc = 0.f;
          const float *qrow = Qs[warp * QPW + t];
#pragma unroll 16
          for (int c = 0; c < HD; ++c) acc = fmaf(qrow[c], Ks[lane][c], acc);
          sc = acc * scale;
        }
        const float mx = warp_max(sc);
        const float mn = fmaxf(m[t], mx);
        if (mn == -INFINITY) continue;
        const float p = ok ? expf(sc - mn) : 0.f;
        const float corr = expf(m[t] - mn);
        l[t] = l[t] * corr + warp_sum(p);
#pragma unroll
        for (int c = 0; c < DPL; ++c) o[t][c] *= corr;
        for (int j = 0; j < KT; ++j) {
          const float pj = __shfl_sync(0xffffffffu, p, j);
#pragma unroll
          for (int c = 0; c < DPL; ++c) o[t][c] = fmaf(pj, Vs[j][lane + 32 * c], o[t][c]);
        }
        m[t] = mn;
      }
    }
#pragma unroll
    for (int t = 0; t < QPW; ++t) {
      const int qr = qb + warp * QPW + t;
      if (qr >= QR) break;
      const int i = qr / G, h = kvh * G + qr % G;
      float *dst = a.part + (((size_t)(b * R + i) * D.hq + h) * a.n_splits + split) * (HD + 2);
#pragma unroll
      for (int c = 0; c < DPL; ++c) dst[lane + 32 * c] = o[t][c];
      if (lane == 0) {
        dst[HD] = m[t];
        dst[HD + 1] = l[t];
      }
    }
  }
}

template <typename T, int HD>
__global__ void k_attn_combine(Dims D, int rows, int n_splits, const float *__restrict__ part,
                               T *__restrict__ out, const int *__restrict__ status) {
  pdl_entry();
  if (*status) return;
  const int rh = blockIdx.x;  // row * hq + head
  const int c = threadIdx.x;  // dimension
  const float *p = part + (size_t)rh * n_splits * (HD + 2);
  float M = -INFINITY;
  for (int s = 0; s < n_splits; ++s) M = fmaxf(M, p[s * (HD + 2) + HD]);
  float L = 0.f, acc = 0.f;
  if (M != -INFINITY) {
    for (int s = 0; s < n_splits; ++s) {
      const float ms = p[s * (HD + 2) + HD];
      if (ms == -INFINITY) continue;
      const float w = expf(ms - M);
      L += w * p[s * (HD + 2) + HD + 1];
      acc += w * p[s * (HD + 2) + c];
    }
  }
  out[(size_t)rh * HD + c] = from_f<T>(L > 0.f ? acc / L : 0.f);
}

template <typename T, int HD>
cudaError_t launch(const Dims &D, int batch, const AttnArgs &a, const int *status, cudaStream_t s) {
  dim3 grid(D.hkv, batch, a.n_splits);
  klaunch(k_attn_split<T, HD>, grid, 128, 0, s, D, a, status);
  const int rows = batch * D.R;
  klaunch(k_attn_combine<T, HD>, rows * D.hq, HD, 0, s, D, rows, a.n_splits, a.part,
                                                   static_cast<T *>(a.out), status);
  return cudaGetLastError();
}

}  // namespace

cudaError_t attention(int dtype, const Dims &D, int batch, const AttnArgs &a, int *status, cudaStream_t s,
                      DepChain *chain) {
  // bf16 caches: the tensor-core kernel; fp32 (the parity model): this one
  if (dtype == DFLOW_BF16) return attention_tc(D, batch, a, status, s, chain);
  if (chain) chain->brk();
  if (D.hd == 128) return launch<float, 128>(D, batch, a, status, s);
  if (D.hd == 64) return launch<float, 64>(D, batch, a, status, s);
  return cudaErrorInvalidValue;
}

}  // namespace dflow
