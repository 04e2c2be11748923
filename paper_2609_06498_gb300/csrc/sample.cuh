// T = 1 verification (speculative sampling over a draft block): the kernels'
// host entry points, called by the round in api.cu.
#pragma once

#include "dflow_internal.cuh"

namespace dflow {

constexpr int SAMP_CHUNK = 4096;  // vocabulary entries per CTA of the row passes
constexpr int SAMP_THREADS = 256;

// purposes of the counter-based draws (the same numbering as the Python side's generator)
constexpr int NOISE_DRAFT = 0, NOISE_ACCEPT = 1, NOISE_RESAMPLE = 2;

inline int samp_chunks(int vocab) { return (vocab + SAMP_CHUNK - 1) / SAMP_CHUNK; }

// workspace views of one round (rows = batch * R)
struct SampWs {
  float2 *part;  // [rows][nch] per-chunk (max, sum exp(x - max)) of a logits row
  float *gv;     // [rows][nch] per-chunk Gumbel-max value
  int *gi;       // [rows][nch] its token
  float *lse_q;  // [rows] drafter log-normaliser of each block row
  float *lse_p;  // [rows] target log-normaliser of each verify row
  int *a;        // [batch] acceptance length
  int nch;
};

struct SampRound {
  uint64_t seed;
  int rnd;  // round index of the draws
};

// drafter logits [batch][R][V] -> block tokens (row 0 the anchor, rows 1..B
// Gumbel-max samples of softmax(q_i)) and the rows' log-normalisers
cudaError_t samp_draft(const float *qlog, int V, int R, int batch, SampRound sr, const SampWs &w,
                       const int *tokens, const int *seq_len, const int *active, int max_ctx, int *blk,
                       const int *status, cudaStream_t s, int *n_launch);

// target logits [batch][R][V] + drafter logits + block -> acceptance length in
// w.a[b] and the token committed after the accepted proposals in g[b R + a]
cudaError_t samp_verify(const float *plog, const float *qlog, int V, int R, int batch, SampRound sr,
                        const SampWs &w, const int *blk, const int *active, int *g, const int *status,
                        cudaStream_t s, int *n_launch);

}  // namespace dflow
