// Steps (3) and (4): pair scores and the greedy walk, one CTA per sequence.
//
// Eq. "pair": adjacent slots are coupled by the cosine between the earlier
// candidate's out vector and the later candidate's in vector; the anchor (the
// paper's slot 0) carries one out vector. Sec. 3.5: the (L-1) K^2 + K terms are
// one small matrix product per slot pair, and the walk commits left to right
// c_s = argmax_k phi(s-1, c_{s-1}, k), touching no weights.
//
// For each slot pair the CTA stages the later slot's K in vectors in shared
// memory (plus their norms), then every warp takes earlier-slot rows and forms
// K dot products by lane-strided loads and a shuffle reduction. All scores stay
// in shared memory; warp 0 then walks the L steps with a warp argmax (ties to the
// lower index) and also reports each step's best-minus-second margin.
#include "internal.cuh"

namespace lilicorr {

namespace {

constexpr int PW_THREADS = 256;
constexpr float UNIT_EPS = 1e-12f;

// warp argmax of (v, idx) with ties to the lower idx
__device__ __forceinline__ void warp_argmax(float& v, int& idx) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
    if (ov > v || (ov == v && oi < idx)) { v = ov; idx = oi; }
  }
}

__global__ void __launch_bounds__(PW_THREADS) pair_walk_kernel(PairWalkArgs a) {
  extern __shared__ float sm[];
  const int b = blockIdx.x;
  const int L = a.L, K = a.K, d = a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = PW_THREADS / 32;
  const int n_scores = K + (L - 1) * K * K;
  // scores live in shared memory when they fit, else the walk reads the global copy
  float* sc = a.scores_in_smem ? sm : nullptr;  // [K] anchor row, then [(L-1)][K][K]
  float* s_in = sm + (a.scores_in_smem ? ((n_scores + 3) & ~3) : 0);   // [K][d]
  float* s_inn = s_in + (size_t)K * d;          // [K]

  if (a.do_pairs) {
    for (int t = -1; t < L - 1; ++t) {          // t = -1: anchor row; else slots (t, t+1)
      __syncthreads();
      const float* inb = a.in + ((size_t)(b * L + t + 1) * K) * a.ld_vec;
      for (int i = threadIdx.x; i < K * d; i += PW_THREADS) {
        const int k = i / d, c = i % d;
        s_in[i] = inb[(size_t)k * a.ld_vec + c];
      }
      __syncthreads();
      for (int k = warp; k < K; k += nw) {
        float ss = 0.f;
        for (int c = lane; c < d; c += 32) ss += s_in[k * d + c] * s_in[k * d + c];
        ss = warp_sum(ss);
        if (lane == 0) s_inn[k] = fmaxf(sqrtf(ss), UNIT_EPS);
      }
      __syncthreads();
      const int nrows = t < 0 ? 1 : K;
      for (int r = warp; r < nrows; r += nw) {
        const float* o = t < 0 ? a.anchor + (size_t)b * d
                               : a.out + ((size_t)(b * L + t) * K + r) * a.ld_vec;
        float oo = 0.f;
        for (int c = lane; c < d; c += 32) oo += o[c] * o[c];
        const float on = fmaxf(sqrtf(warp_sum(oo)), UNIT_EPS);
        for (int k2 = 0; k2 < K; ++k2) {
          float dot = 0.f;
          for (int c = lane; c < d; c += 32) dot = fmaf(o[c], s_in[k2 * d + c], dot);
          dot = warp_sum(dot);
          if (lane == 0) {
            const float v = dot / (on * s_inn[k2]);
            if (t < 0) {
              if (sc) sc[k2] = v;
              a.A[(size_t)b * K + k2] = v;
            } else {
              const size_t off = ((size_t)t * K + r) * K + k2;
              if (sc) sc[K + off] = v;
              a.P[(size_t)b * (L - 1) * K * K + off] = v;
            }
          }
        }
      }
    }
  } else if (sc) {
    for (int i = threadIdx.x; i < K; i += PW_THREADS) sc[i] = a.A[(size_t)b * K + i];
    for (int i = threadIdx.x; i < (L - 1) * K * K; i += PW_THREADS)
      sc[K + i] = a.P[(size_t)b * (L - 1) * K * K + i];
  }
  __syncthreads();     // also makes this CTA's global score writes visible to warp 0
  if (!a.do_walk || warp != 0) return;

  const float* gA = a.A + (size_t)b * K;
  const float* gP = a.P + (size_t)b * (L - 1) * K * K;
  int prev = 0;
  for (int s = 0; s < L; ++s) {
    const float* row = sc ? (s == 0 ? sc : sc + K + ((size_t)(s - 1) * K + prev) * K)
                          : (s == 0 ? gA : gP + ((size_t)(s - 1) * K + prev) * K);
    float v = lane < K ? row[lane] : -INFINITY;
    int idx = lane < K ? lane : 0x7fffffff;
    float best = v;
    int bi = idx;
    warp_argmax(best, bi);
    bi = __shfl_sync(0xffffffffu, bi, 0);     // one choice for the whole warp, even on NaN rows
    best = __shfl_sync(0xffffffffu, best, 0);
    if (bi < 0 || bi >= K) bi = 0;
    float second = (lane < K && lane != bi) ? v : -INFINITY;
    second = warp_max(second);
    if (lane == 0) {
      const size_t o = (size_t)b * L + s;
      if (a.choice) a.choice[o] = bi;
      if (a.tokens) a.tokens[o] = a.ids[o * K + bi];
      if (a.margin) a.margin[o] = K > 1 ? best - second : INFINITY;
    }
    prev = bi;
  }
}

}  // namespace

constexpr size_t PW_SMEM_MAX = 227 * 1024;

size_t pair_walk_smem_bytes(int L, int K, int d, bool scores) {
  const size_t n_scores = scores ? (size_t)K + (size_t)(L - 1) * K * K : 0;
  return sizeof(float) * (align_up(n_scores, 4) + (size_t)K * d + K);
}

// Shared memory needed at least (the in vectors of one slot and their norms).
size_t pair_walk_smem_bytes(int L, int K, int d) { return pair_walk_smem_bytes(L, K, d, false); }

lilicorr_status_t launch_pair_walk(const PairWalkArgs& in, cudaStream_t st) {
  if (in.B == 0) return LILICORR_OK;
  PairWalkArgs a = in;
  const int dv = a.do_pairs ? a.d : 0;
  a.scores_in_smem = pair_walk_smem_bytes(a.L, a.K, dv, true) <= PW_SMEM_MAX;
  const size_t smem = pair_walk_smem_bytes(a.L, a.K, dv, a.scores_in_smem);
  if (smem > PW_SMEM_MAX) return LILICORR_ERR_SHAPE;
  static bool configured[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !configured[dev]) {
    LL_CUDA_TRY(cudaFuncSetAttribute(pair_walk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     227 * 1024));
    configured[dev] = true;
  }
  pair_walk_kernel<<<a.B, PW_THREADS, smem, st>>>(a);
  return last_launch();
}

}  // namespace lilicorr
