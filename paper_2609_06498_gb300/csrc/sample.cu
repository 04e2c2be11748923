// T = 1 verification of a draft block by speculative sampling.
//
// The paper reports T = 1 results (Sec. 5.2, Table 1) without printing the
// sampling rule; the rule here is the standard one for proposals drawn from a
// known distribution, applied per block position:
//   * the drafter proposes y_i ~ q_i = softmax(drafter logits of row i), i = 1..B;
//   * proposal i is accepted while u_i < p_i(y_i) / q_i(y_i), with
//     p_i = softmax(target logits of verify row i - 1);
//   * at the first rejection (offset i) the committed token is drawn from
//     max(0, p_i - q_i) normalised; after B acceptances the bonus is drawn
//     from p_{B+1}.
// Every draw is a Gumbel-max sample, argmax_v (log w_v + g_v), with
// g_v = -log(-log u_v); the uniforms come from a counter-based SplitMix64
// stream per (seed, sequence, round, row, purpose) indexed by the token id,
// u = (2 k + 1) / 2^24 with k the top 23 bits of the hash (exact in fp32).
//
// Passes over the logits are chunked: one CTA per (4096-entry chunk, row)
// reduces its chunk to a (max, sum exp) pair and, where a draw is taken, to a
// (value, token) Gumbel-max pair; one thread per row or sequence then merges
// the chunks in chunk order (ties go to the lower token id).
#include <math.h>

#include "sample.cuh"

namespace dflow {
namespace {

// SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number generators", 2014)
__device__ __forceinline__ uint64_t splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t noise_key(uint64_t seed, int seq, int rnd, int row, int purpose) {
  return splitmix64(seed ^ splitmix64(((uint64_t)seq << 48) ^ ((uint64_t)rnd << 24) ^ ((uint64_t)row << 8) ^
                                      (uint64_t)purpose));
}

__device__ __forceinline__ float noise_uniform(uint64_t key, int v) {
  const uint32_t k = (uint32_t)(splitmix64(key ^ (uint64_t)v) >> 41);  // 23 bits
  return (float)(2u * k + 1u) * 0x1p-24f;
}

__device__ __forceinline__ float gumbel(uint64_t key, int v) { return -logf(-logf(noise_uniform(key, v))); }

// (max, sum exp(x - max)) merge
__device__ __forceinline__ void lse_merge(float &m, float &s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float mn = fmaxf(m, m2);
  s = s * expf(m - mn) + s2 * expf(m2 - mn);
  m = mn;
}

// block-wide merge of per-thread (max, sum) and (value, token) pairs; the
// result is valid in thread 0
template <bool ARG>
__device__ void block_reduce(float &m, float &s, float &gv, int &gi) {
  __shared__ float sm_m[SAMP_THREADS / 32], sm_s[SAMP_THREADS / 32], sm_v[SAMP_THREADS / 32];
  __shared__ int sm_i[SAMP_THREADS / 32];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    lse_merge(m, s, m2, s2);
  }
  if (ARG) warp_argmax(gv, gi);
  if (lane == 0) {
    sm_m[warp] = m;
    sm_s[warp] = s;
    sm_v[warp] = gv;
    sm_i[warp] = gi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < SAMP_THREADS / 32; ++w) {
      lse_merge(m, s, sm_m[w], sm_s[w]);
      if (ARG) argmax_merge(gv, gi, sm_v[w], sm_i[w]);
    }
  }
}

// One (chunk, row) of a logits array [batch][R][V]: the chunk's (max, sum
// exp); with draft set, also the Gumbel-max pair of rows 1..B (the proposal
// draw of row i uses the NOISE_DRAFT stream of (sequence, round, i)).
__global__ void __launch_bounds__(SAMP_THREADS) k_samp_stats(const float *__restrict__ lg, int V, int R, int draft,
                                                            SampRound sr, SampWs w, const int *__restrict__ active,
                                                            const int *status) {
  pdl_entry();
  if (*status) return;
  const int c = blockIdx.x, r = blockIdx.y, b = r / R, i = r % R;
  if (!active[b]) return;
  const int v0 = c * SAMP_CHUNK, v1 = min(V, v0 + SAMP_CHUNK);
  const float *x = lg + (size_t)r * V;
  const bool draw = draft && i > 0;
  const uint64_t key = draw ? noise_key(sr.seed, b, sr.rnd, i, NOISE_DRAFT) : 0;
  constexpr int PER = SAMP_CHUNK / SAMP_THREADS;
  float xs[PER];
  float m = -INFINITY, s = 0.f, gv = -INFINITY;
  int gi = 0x7fffffff;
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int v = v0 + j * SAMP_THREADS + threadIdx.x;
    xs[j] = v < v1 ? x[v] : -INFINITY;
    m = fmaxf(m, xs[j]);
  }
  if (m != -INFINITY) {
#pragma unroll
    for (int j = 0; j < PER; ++j) s += expf(xs[j] - m);
  }
  if (draw) {
#pragma unroll
    for (int j = 0; j < PER; ++j) {
      const int v = v0 + j * SAMP_THREADS + threadIdx.x;
      if (v < v1) argmax_merge(gv, gi, xs[j] + gumbel(key, v), v);
    }
  }
  if (draw) block_reduce<true>(m, s, gv, gi);
  else block_reduce<false>(m, s, gv, gi);
  if (threadIdx.x == 0) {
    const size_t o = (size_t)r * w.nch + c;
    w.part[o] = make_float2(m, s);
    if (draw) {
      w.gv[o] = gv;
      w.gi[o] = gi;
    }
  }
}

// merged log-normaliser of row r from its chunk pairs
__device__ __forceinline__ float row_lse(const SampWs &w, int r) {
  float m = -INFINITY, s = 0.f;
  for (int c = 0; c < w.nch; ++c) {
    const float2 p = w.part[(size_t)r * w.nch + c];
    lse_merge(m, s, p.x, p.y);
  }
  return m + logf(s);
}

// one thread per block row: the proposal token (row 0: the anchor) and lse_q
__global__ void k_samp_draft_out(int R, int batch, SampWs w, const int *__restrict__ tokens,
                                 const int *__restrict__ seq_len, const int *__restrict__ active, int max_ctx,
                                 int *__restrict__ blk, const int *status) {
  pdl_entry();
  if (*status) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= batch * R) return;
  const int b = r / R, i = r % R;
  if (!active[b]) {
    blk[r] = i == 0 ? tokens[(size_t)b * max_ctx + seq_len[b] - 1] : 0;
    return;
  }
  w.lse_q[r] = row_lse(w, r);
  if (i == 0) {
    blk[r] = tokens[(size_t)b * max_ctx + seq_len[b] - 1];
    return;
  }
  float v = -INFINITY;
  int t = 0x7fffffff;
  for (int c = 0; c < w.nch; ++c) argmax_merge(v, t, w.gv[(size_t)r * w.nch + c], w.gi[(size_t)r * w.nch + c]);
  blk[r] = t;
}

// one CTA per sequence: lse_p of the B + 1 verify rows (a warp per row), then
// the acceptance tests in block order (thread 0)
__global__ void __launch_bounds__(SAMP_THREADS) k_samp_decide(const float *__restrict__ plog,
                                                             const float *__restrict__ qlog, int V, int R,
                                                             SampRound sr, SampWs w, const int *__restrict__ blk,
                                                             const int *__restrict__ active, const int *status) {
  pdl_entry();
  if (*status) return;
  const int b = blockIdx.x, B = R - 1;
  if (!active[b]) {
    if (threadIdx.x == 0) w.a[b] = 0;
    return;
  }
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  for (int j = warp; j < R; j += SAMP_THREADS / 32) {
    const int r = b * R + j;
    float m = -INFINITY, s = 0.f;
    for (int c = lane; c < w.nch; c += 32) {
      const float2 p = w.part[(size_t)r * w.nch + c];
      lse_merge(m, s, p.x, p.y);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
      lse_merge(m, s, m2, s2);
    }
    if (lane == 0) w.lse_p[r] = m + logf(s);
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  int a = B;
  for (int i = 1; i <= B; ++i) {
    const int y = blk[b * R + i];
    const float lp = plog[(size_t)(b * R + i - 1) * V + y] - w.lse_p[b * R + i - 1];
    const float lq = qlog[(size_t)(b * R + i) * V + y] - w.lse_q[b * R + i];
    const float u = noise_uniform(noise_key(sr.seed, b, sr.rnd, i, NOISE_ACCEPT), 0);
    if (!(logf(u) < lp - lq)) {
      a = i - 1;
      break;
    }
  }
  w.a[b] = a;
}

// One (chunk, sequence): the Gumbel-max pair of the committed token's draw for
// offset i = a + 1 (NOISE_RESAMPLE stream of row i): from max(0, p_i - q_i)
// after a rejection (log(p - q) = lp + log1p(-exp(lq - lp)) where lp > lq),
// from p_{B+1} after B acceptances; and, for the case where rounding leaves
// the residual empty, the pair of a draw from p_i with the same noise.
__global__ void __launch_bounds__(SAMP_THREADS) k_samp_resample(const float *__restrict__ plog,
                                                               const float *__restrict__ qlog, int V, int R,
                                                               SampRound sr, SampWs w,
                                                               const int *__restrict__ active, const int *status) {
  pdl_entry();
  if (*status) return;
  const int c = blockIdx.x, b = blockIdx.y, B = R - 1;
  if (!active[b]) return;
  const int a = w.a[b], i = a + 1;
  const int rp = b * R + a, rq = b * R + a + 1;
  const float *xp = plog + (size_t)rp * V;
  const float *xq = a < B ? qlog + (size_t)rq * V : nullptr;
  const float lsp = w.lse_p[rp], lsq = a < B ? w.lse_q[rq] : 0.f;
  const uint64_t key = noise_key(sr.seed, b, sr.rnd, i, NOISE_RESAMPLE);
  const int v0 = c * SAMP_CHUNK, v1 = min(V, v0 + SAMP_CHUNK);
  float rv = -INFINITY, pv = -INFINITY;
  int ri = 0x7fffffff, pi = 0x7fffffff;
  for (int v = v0 + threadIdx.x; v < v1; v += SAMP_THREADS) {
    const float g = gumbel(key, v), lp = xp[v] - lsp;
    argmax_merge(pv, pi, lp + g, v);
    if (xq != nullptr) {
      const float lq = xq[v] - lsq;
      if (lp > lq) argmax_merge(rv, ri, lp + log1pf(-expf(lq - lp)) + g, v);
    }
  }
  float m = 0.f, s = 0.f;  // unused lse slots of the shared reduction
  block_reduce<true>(m, s, rv, ri);
  __syncthreads();
  float m2 = 0.f, s2 = 0.f;
  block_reduce<true>(m2, s2, pv, pi);
  if (threadIdx.x == 0) {
    const size_t o = ((size_t)b * R) * w.nch + c;  // row b R (the anchor row) holds the residual pair,
    w.gv[o] = rv;                                   // row b R + 1 the draw from p
    w.gi[o] = ri;
    w.gv[o + w.nch] = pv;
    w.gi[o + w.nch] = pi;
  }
}

// one thread per sequence: merge the chunks and place the token at g[b R + a]
__global__ void k_samp_pick(int R, int batch, SampWs w, const int *__restrict__ active, int *__restrict__ g,
                            const int *status) {
  pdl_entry();
  if (*status) return;
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch || !active[b]) return;
  const int a = w.a[b];
  const size_t o = ((size_t)b * R) * w.nch;
  float rv = -INFINITY, pv = -INFINITY;
  int ri = 0x7fffffff, pi = 0x7fffffff;
  for (int c = 0; c < w.nch; ++c) {
    argmax_merge(rv, ri, w.gv[o + c], w.gi[o + c]);
    argmax_merge(pv, pi, w.gv[o + w.nch + c], w.gi[o + w.nch + c]);
  }
  // after B acceptances the draw is the one from p_{B+1}; after a rejection the
  // residual's, unless rounding left it empty
  g[(size_t)b * R + a] = (a < R - 1 && rv != -INFINITY) ? ri : pi;
}

}  // namespace

cudaError_t samp_draft(const float *qlog, int V, int R, int batch, SampRound sr, const SampWs &w,
                       const int *tokens, const int *seq_len, const int *active, int max_ctx, int *blk,
                       const int *status, cudaStream_t s, int *n_launch) {
  cudaError_t e = klaunch(k_samp_stats, dim3(w.nch, batch * R), dim3(SAMP_THREADS), 0, s, qlog, V, R, 1, sr, w,
                          active, status);
  if (e != cudaSuccess) return e;
  e = klaunch(k_samp_draft_out, dim3((batch * R + 127) / 128), dim3(128), 0, s, R, batch, w, tokens, seq_len, active,
              max_ctx, blk, status);
  *n_launch += 2;
  return e;
}

cudaError_t samp_verify(const float *plog, const float *qlog, int V, int R, int batch, SampRound sr,
                        const SampWs &w, const int *blk, const int *active, int *g, const int *status,
                        cudaStream_t s, int *n_launch) {
  cudaError_t e = klaunch(k_samp_stats, dim3(w.nch, batch * R), dim3(SAMP_THREADS), 0, s, plog, V, R, 0, sr, w,
                          active, status);
  if (e != cudaSuccess) return e;
  if ((e = klaunch(k_samp_decide, dim3(batch), dim3(SAMP_THREADS), 0, s, plog, qlog, V, R, sr, w, blk, active,
                   status)))
    return e;
  if ((e = klaunch(k_samp_resample, dim3(w.nch, batch), dim3(SAMP_THREADS), 0, s, plog, qlog, V, R, sr, w, active,
                   status)))
    return e;
  e = klaunch(k_samp_pick, dim3((batch + 127) / 128), dim3(128), 0, s, R, batch, w, active, g, status);
  *n_launch += 4;
  return e;
}

}  // namespace dflow
