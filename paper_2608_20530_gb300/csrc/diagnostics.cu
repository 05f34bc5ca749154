// Diagnostics of a selected block: the local next-candidate distributions of Eq.
// "localar", the decision gaps of Eq. "margin" along a path, and coverage / oracle prefix
// / prefix acceptance against ground-truth tokens (Sec. 3.3 "Oracle-prefix supervision";
// Sec. 3.1 prefix acceptance).
//
// local_softmax_kernel: one warp per score row (the anchor row of a sequence, or the row
//   of one predecessor at one slot pair); lane k holds sigma * score[k], warp max and sum.
// path_probs_kernel: one warp per sequence walks the path; per step the same warp softmax
//   over the row of the path's predecessor, the chosen candidate's probability and its
//   gap to the best other candidate.
// acceptance_kernel: one thread per sequence (L <= 64, K <= 32 integer compares).
#include "internal.cuh"

namespace lilicorr {

namespace {

constexpr int DG_THREADS = 256;

// softmax over the K (<= 32) values v of a warp's lanes (lanes >= K hold -inf): returns
// this lane's probability and the row maximum
__device__ __forceinline__ float warp_softmax(float z, int lane, int K, float& zmax) {
  const float m = warp_max(lane < K ? z : -INFINITY);
  const float e = lane < K ? expf(z - m) : 0.f;
  const float sum = warp_sum(e);
  zmax = m;
  return e / sum;
}

__global__ void __launch_bounds__(DG_THREADS)
local_softmax_kernel(int B, int L, int K, const float* __restrict__ A, const float* __restrict__ P,
                     float sigma, float* __restrict__ pa, float* __restrict__ pp) {
  pdl_wait();
  const int rows_per_seq = 1 + (L - 1) * K;
  const long long row = (long long)blockIdx.x * (DG_THREADS / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= (long long)B * rows_per_seq) return;
  const int b = (int)(row / rows_per_seq), r = (int)(row % rows_per_seq);
  const float* src = r == 0 ? A + (size_t)b * K : P + ((size_t)b * (L - 1) * K + (r - 1)) * K;
  float* dst = r == 0 ? pa + (size_t)b * K : pp + ((size_t)b * (L - 1) * K + (r - 1)) * K;
  const float z = lane < K ? sigma * src[lane] : -INFINITY;
  float m;
  const float p = warp_softmax(z, lane, K, m);
  if (lane < K && dst) dst[lane] = p;
}

__global__ void __launch_bounds__(DG_THREADS)
path_probs_kernel(int B, int L, int K, const float* __restrict__ A, const float* __restrict__ P,
                  const int32_t* __restrict__ choice, float sigma, float* __restrict__ prob,
                  float* __restrict__ gap, float* __restrict__ log_prob) {
  pdl_wait();
  const int b = blockIdx.x * (DG_THREADS / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (b >= B) return;
  float lp = 0.f;
  int prev = 0;
  for (int s = 0; s < L; ++s) {
    const int c = choice[(size_t)b * L + s];
    const bool valid = c >= 0 && c < K && prev >= 0 && prev < K;
    const float* row = s == 0 ? A + (size_t)b * K
                              : P + (((size_t)b * (L - 1) + (s - 1)) * K + (valid ? prev : 0)) * K;
    const float z = lane < K ? sigma * row[lane] : -INFINITY;
    float m;
    const float p = warp_softmax(z, lane, K, m);
    const float pc = __shfl_sync(0xffffffffu, p, valid ? c : 0);
    const float zc = __shfl_sync(0xffffffffu, z, valid ? c : 0);
    const float other = warp_max((lane < K && lane != c) ? z : -INFINITY);
    if (lane == 0) {
      const size_t o = (size_t)b * L + s;
      const float ps = valid ? pc : NAN;               // a choice outside [0, K) has no probability
      if (prob) prob[o] = ps;
      if (gap) gap[o] = valid ? (K > 1 ? zc - other : INFINITY) : NAN;
      lp += logf(ps);
    }
    prev = c;
  }
  if (lane == 0 && log_prob) log_prob[b] = lp;
}

__global__ void __launch_bounds__(DG_THREADS)
acceptance_kernel(int B, int L, int K, const int32_t* __restrict__ ids,
                  const int32_t* __restrict__ tokens, const int32_t* __restrict__ truth,
                  int32_t* __restrict__ covered, int32_t* __restrict__ oracle_prefix,
                  int32_t* __restrict__ accepted) {
  pdl_wait();
  const int b = blockIdx.x * DG_THREADS + threadIdx.x;
  if (b >= B) return;
  int prefix = 0, acc = 0;
  bool run_cov = true, run_acc = true;
  for (int s = 0; s < L; ++s) {
    const size_t o = (size_t)b * L + s;
    const int32_t g = truth[o];
    int cov = 0;
    for (int k = 0; k < K; ++k) cov |= ids[o * K + k] == g ? 1 : 0;
    if (covered) covered[o] = cov;
    run_cov = run_cov && cov;
    prefix += run_cov ? 1 : 0;
    run_acc = run_acc && tokens[o] == g;
    acc += run_acc ? 1 : 0;
  }
  if (oracle_prefix) oracle_prefix[b] = prefix;
  if (accepted) accepted[b] = acc;
}

bool shape_ok(int B, int L, int K) {
  return B >= 0 && L > 0 && L <= LILICORR_MAX_L && K > 0 && K <= LILICORR_MAX_K;
}

}  // namespace

}  // namespace lilicorr

using namespace lilicorr;

extern "C" lilicorr_status_t lilicorr_local_softmax(int B, int L, int K, const float* anchor_scores,
                                                    const float* pair_scores, float sigma,
                                                    float* anchor_probs, float* pair_probs,
                                                    cudaStream_t stream) {
  if (!shape_ok(B, L, K)) return LILICORR_ERR_SHAPE;
  if (!(sigma > 0.f) || !isfinite(sigma)) return LILICORR_ERR_ARG;
  if (B == 0) return LILICORR_OK;
  if (!anchor_scores || !anchor_probs || (L > 1 && (!pair_scores || !pair_probs)))
    return LILICORR_ERR_ARG;
  const long long rows = (long long)B * (1 + (L - 1) * K);
  const int grid = (int)((rows + DG_THREADS / 32 - 1) / (DG_THREADS / 32));
  LL_TRY(launch_k(local_softmax_kernel, grid, DG_THREADS, 0, stream, B, L, K, anchor_scores,
                  pair_scores, sigma, anchor_probs, pair_probs));
  return LILICORR_OK;
}

extern "C" lilicorr_status_t lilicorr_path_probs(int B, int L, int K, const float* anchor_scores,
                                                 const float* pair_scores, const int32_t* choice,
                                                 float sigma, float* prob, float* gap,
                                                 float* log_prob, cudaStream_t stream) {
  if (!shape_ok(B, L, K)) return LILICORR_ERR_SHAPE;
  if (!(sigma > 0.f) || !isfinite(sigma)) return LILICORR_ERR_ARG;
  if (B == 0) return LILICORR_OK;
  if (!anchor_scores || (L > 1 && !pair_scores) || !choice) return LILICORR_ERR_ARG;
  LL_TRY(launch_k(path_probs_kernel, ceil_div(B, DG_THREADS / 32), DG_THREADS, 0, stream, B, L, K,
                  anchor_scores, pair_scores, choice, sigma, prob, gap, log_prob));
  return LILICORR_OK;
}

extern "C" lilicorr_status_t lilicorr_block_acceptance(int B, int L, int K, const int32_t* ids,
                                                       const int32_t* tokens, const int32_t* truth,
                                                       int32_t* covered, int32_t* oracle_prefix,
                                                       int32_t* accepted, cudaStream_t stream) {
  if (!shape_ok(B, L, K)) return LILICORR_ERR_SHAPE;
  if (B == 0) return LILICORR_OK;
  if (!ids || !tokens || !truth) return LILICORR_ERR_ARG;
  LL_TRY(launch_k(acceptance_kernel, ceil_div(B, DG_THREADS), DG_THREADS, 0, stream, B, L, K, ids,
                  tokens, truth, covered, oracle_prefix, accepted));
  return LILICORR_OK;
}
