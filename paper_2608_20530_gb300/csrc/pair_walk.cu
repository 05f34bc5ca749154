// Steps (3) and (4): pair scores and the greedy walk.
//
// Eq. "pair": adjacent slots are coupled by the cosine between the earlier
// candidate's out vector and the later candidate's in vector; the anchor (the
// paper's slot 0) carries one out vector. Sec. 3.5: the (L-1) K^2 + K terms are
// one small matrix product per slot pair, and the walk commits left to right
// c_s = argmax_k phi(s-1, c_{s-1}, k), touching no weights.
//
// pair_block_kernel: grid (B, L). CTA (b, j) scores the anchor row (j = 0) or the slot
// pair (j-1, j): both slots' vectors are staged in shared memory and each thread forms
// whole dot products (one output at a time). pair_rows_kernel, the same grid for vectors
// too long to stage twice: it stages slot j's K in vectors and their norms, every warp
// takes rows of the earlier slot and forms K dot products by lane-strided loads and a
// shuffle reduction. With the walk fused, the last CTA
// of a sequence to finish (atomic ticket, nobody waits) loads the sequence's
// scores into shared memory and walks them.
// walk_kernel: grid B, the walk alone over given scores.
// The walk is one warp: per step one butterfly over the candidates' lanes carries the best
// (ties to the lower index) and the second-best score, for the choice and the
// best-minus-second margin; the tokens are gathered for all slots after the walk. In Viterbi mode (App. E) the same warp computes the exact
// maximiser of the path score g(c) = sigma (A[c_1] + sum_s P[s-1, c_{s-1}, c_s]) instead:
// lane k keeps the best score of a path ending at candidate k, one sweep over the slots
// records each lane's best predecessor (ties to the lower index) in shared memory, and
// lane 0 traces the path back from the best final candidate (ties to the lower index).
#include "internal.cuh"
#include "walk.cuh"

namespace lilicorr {

namespace {
using namespace walk;

constexpr int PW_THREADS = 256;

// Asynchronous global -> shared copies: every thread issues all of its copies before
// any wait, so a staging loop costs one memory latency rather than one per iteration.
__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;"
               ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;"
               ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_wait_all() {
  asm volatile("cp.async.commit_group;\n cp.async.wait_group 0;" ::: "memory");
}
// The sequence's scores A [K] then P [(L-1) K K] into shared memory (caller syncs).
__device__ __forceinline__ void stage_scores(float* sm, const float* gA, const float* gP, int K,
                                             int n_scores) {
  for (int i = threadIdx.x; i < n_scores; i += PW_THREADS) cp4(sm + i, i < K ? gA + i : gP + (i - K));
  cp_wait_all();
}
constexpr float UNIT_EPS = 1e-12f;
constexpr size_t PW_SMEM_MAX = 200 * 1024;     // dynamic shared memory the launcher may ask for

__device__ __forceinline__ void warp_argmax(float& v, int& idx) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
    if (ov > v || (ov == v && oi < idx)) { v = ov; idx = oi; }
  }
}

// Exact best path of one sequence (one full warp). back: [L * K] bytes of shared memory;
// the path goes to path[L] in shared memory.
__device__ void viterbi_sequence(const float* A, const float* P, int b, int L, int K, float sigma,
                                 float* score, uint8_t* back, uint8_t* path) {
  const int lane = threadIdx.x & 31;
  float best = lane < K ? sigma * A[lane] : -INFINITY;
  for (int s = 1; s < L; ++s) {
    const float* Ps = P + (size_t)(s - 1) * K * K;
    float bv = -INFINITY;
    int bk = 0;
    for (int k = 0; k < K; ++k) {
      const float pk = __shfl_sync(0xffffffffu, best, k);
      const float c = pk + sigma * (lane < K ? Ps[k * K + lane] : 0.f);
      if (c > bv) { bv = c; bk = k; }             // strict: the lower predecessor on ties
    }
    if (lane < K) back[s * K + lane] = (uint8_t)bk;
    best = lane < K ? bv : -INFINITY;
  }
  float v = best;
  int bi = lane < K ? lane : 0x7fffffff;
  warp_argmax(v, bi);
  bi = __shfl_sync(0xffffffffu, bi, 0);
  v = __shfl_sync(0xffffffffu, v, 0);
  if (bi < 0 || bi >= K) bi = 0;
  __syncwarp();
  if (lane == 0) {
    int c = bi;
    for (int s = L - 1; s >= 0; --s) {
      path[s] = (uint8_t)c;
      if (s > 0) c = back[s * K + c];
    }
    if (score) score[b] = v;
  }
}

__device__ __forceinline__ void run_walk(const PairWalkArgs& a, const float* A, const float* P,
                                         int b, uint8_t* back, uint8_t* path) {
  if (a.walk_mode == LILICORR_WALK_VITERBI)
    viterbi_sequence(A, P, b, a.L, a.K, a.sigma, a.path_score, back, path);
  else
    walk_sequence(A, P, b, a.L, a.K, a.margin, path);
  __syncwarp();
  const int lane = threadIdx.x & 31;
  for (int s = lane; s < a.L; s += 32) {        // choices and tokens, all slots at once
    const size_t o = (size_t)b * a.L + s;
    const int c = path[s];
    if (a.choice) a.choice[o] = c;
    if (a.tokens) a.tokens[o] = a.ids[o * a.K + c];
  }
}

// The walk after the pair scores: the last CTA of a sequence to finish (atomic ticket,
// nobody waits) stages the sequence's scores in shared memory and walks them.
__device__ __forceinline__ void walk_after_pairs(const PairWalkArgs& a, float* sm, int* s_last,
                                                 uint8_t* s_back, uint8_t* s_path) {
  const int b = blockIdx.x, L = a.L, K = a.K;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) *s_last = atomicAdd(&a.counters[b], 1u) == (uint32_t)(L - 1);
  __syncthreads();
  if (!*s_last) return;
  __threadfence();
  const int n_scores = K + (L - 1) * K * K;
  const float* gA = a.A + (size_t)b * K;
  const float* gP = a.P + (size_t)b * (L - 1) * K * K;
  const float* A = gA;
  const float* P = gP;
  if (a.scores_in_smem) {                       // reuse the staging buffer for the scores
    stage_scores(sm, gA, gP, K, n_scores);
    __syncthreads();
    A = sm;
    P = sm + K;
  }
  if ((threadIdx.x >> 5) == 0) {
    run_walk(a, A, P, b, s_back, s_path);
    if ((threadIdx.x & 31) == 0) a.counters[b] = 0u;   // leave the workspace reusable
  }
}

// Row stride (floats) of the staged vectors: 16-byte aligned rows whose 16-byte pieces
// start on different banks for consecutive rows.
__host__ __device__ __forceinline__ int pw_stride(int d) { return (d + 3) / 4 * 4 + 4; }

// CTA (b, j): the slot pair (j - 1, j), or the anchor row (j = 0). Both slots' vectors
// (K in vectors of slot j, K out vectors of slot j - 1 or the anchor's one) are staged in
// shared memory by asynchronous copies, all issued before one wait; each warp takes the
// norms of some rows; then thread t forms whole dot products, one output (k, k') at a time,
// reading both rows from shared memory (no cross-lane reductions) and storing the cosine.
__global__ void __launch_bounds__(PW_THREADS) pair_block_kernel(PairWalkArgs a) {
  pdl_wait();
  extern __shared__ float sm[];
  __shared__ int s_last;
  __shared__ float s_norm[2 * LILICORR_MAX_K];
  __shared__ uint8_t s_back[LILICORR_MAX_L * LILICORR_MAX_K];
  __shared__ uint8_t s_path[LILICORR_MAX_L];
  const int b = blockIdx.x, j = blockIdx.y;
  const int L = a.L, K = a.K, d = a.d, ds = pw_stride(d);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = PW_THREADS / 32;
  const int nrows = j == 0 ? 1 : K;                 // vectors of the earlier slot (or anchor)
  const float* inb = a.in + (size_t)(b * L + j) * K * a.ld_vec;
  const float* outb = j == 0 ? a.anchor + (size_t)b * d
                             : a.out + (size_t)(b * L + j - 1) * K * a.ld_vec;
  const int ldo = j == 0 ? d : a.ld_vec;
  const bool v4 = ((d | a.ld_vec) & 3) == 0 && (reinterpret_cast<uintptr_t>(a.in) & 15) == 0 &&
                  (reinterpret_cast<uintptr_t>(a.out) & 15) == 0 &&
                  (reinterpret_cast<uintptr_t>(a.anchor) & 15) == 0;
  // rows 0 .. K-1: in vectors of slot j; rows K .. K+nrows-1: out vectors (or the anchor)
  if (v4) {
    const int dv = d >> 2;
    for (int i = threadIdx.x; i < (K + nrows) * dv; i += PW_THREADS) {
      const int row = i / dv, c = 4 * (i - row * dv);
      const float* src = row < K ? inb + (size_t)row * a.ld_vec + c : outb + (size_t)(row - K) * ldo + c;
      cp16(sm + (size_t)row * ds + c, src);
    }
    cp_wait_all();
  } else {
    for (int i = threadIdx.x; i < (K + nrows) * d; i += PW_THREADS) {
      const int row = i / d, c = i - row * d;
      sm[(size_t)row * ds + c] = row < K ? inb[(size_t)row * a.ld_vec + c]
                                         : outb[(size_t)(row - K) * ldo + c];
    }
  }
  __syncthreads();
  for (int v = warp; v < K + nrows; v += nw) {
    float ss = 0.f;
    for (int c = lane; c < d; c += 32) ss = fmaf(sm[(size_t)v * ds + c], sm[(size_t)v * ds + c], ss);
    ss = warp_sum(ss);
    if (lane == 0) s_norm[v] = fmaxf(sqrtf(ss), UNIT_EPS);
  }
  __syncthreads();
  for (int o = threadIdx.x; o < nrows * K; o += PW_THREADS) {
    const int r = o / K, k2 = o - r * K;
    const float* x = sm + (size_t)(K + r) * ds;
    const float* y = sm + (size_t)k2 * ds;
    float acc0 = 0.f, acc1 = 0.f;
    int c = 0;
    if ((d & 3) == 0) {
      for (; c < d; c += 8) {
        const float4 x0 = *reinterpret_cast<const float4*>(x + c);
        const float4 y0 = *reinterpret_cast<const float4*>(y + c);
        acc0 = fmaf(x0.x, y0.x, fmaf(x0.y, y0.y, fmaf(x0.z, y0.z, fmaf(x0.w, y0.w, acc0))));
        if (c + 4 < d) {
          const float4 x1 = *reinterpret_cast<const float4*>(x + c + 4);
          const float4 y1 = *reinterpret_cast<const float4*>(y + c + 4);
          acc1 = fmaf(x1.x, y1.x, fmaf(x1.y, y1.y, fmaf(x1.z, y1.z, fmaf(x1.w, y1.w, acc1))));
        }
      }
    } else {
      for (; c < d; ++c) acc0 = fmaf(x[c], y[c], acc0);
    }
    const float v = (acc0 + acc1) / (s_norm[K + r] * s_norm[k2]);
    if (j == 0) a.A[(size_t)b * K + k2] = v;
    else a.P[((size_t)b * (L - 1) + (j - 1)) * K * K + (size_t)r * K + k2] = v;
  }
  if (!a.do_walk) return;
  walk_after_pairs(a, sm, &s_last, s_back, s_path);
}

__global__ void __launch_bounds__(PW_THREADS) pair_rows_kernel(PairWalkArgs a) {
  pdl_wait();
  extern __shared__ float sm[];
  __shared__ int s_last;
  __shared__ uint8_t s_back[LILICORR_MAX_L * LILICORR_MAX_K];
  __shared__ uint8_t s_path[LILICORR_MAX_L];
  const int b = blockIdx.x, j = blockIdx.y;          // j = 0: anchor row; j >= 1: pair (j-1, j)
  const int L = a.L, K = a.K, d = a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = PW_THREADS / 32;
  float* s_in = sm;                                  // [K][d]
  float* s_inn = s_in + (size_t)K * d;               // [K]

  const float* inb = a.in + (size_t)(b * L + j) * K * a.ld_vec;
  // 16-byte vectors when every row starts 16-byte aligned (d and the row stride multiples
  // of 4 floats)
  const bool v4 = ((d | a.ld_vec) & 3) == 0 && (reinterpret_cast<uintptr_t>(a.in) & 15) == 0 &&
                  (reinterpret_cast<uintptr_t>(a.out) & 15) == 0 &&
                  (reinterpret_cast<uintptr_t>(a.anchor) & 15) == 0;
  if (v4) {
    const int dv = d >> 2;
    for (int i = threadIdx.x; i < K * dv; i += PW_THREADS) {
      const int k = i / dv, c = i - k * dv;
      cp16(s_in + (size_t)k * d + 4 * c, inb + (size_t)k * a.ld_vec + 4 * c);
    }
    cp_wait_all();
  } else {
    for (int i = threadIdx.x; i < K * d; i += PW_THREADS) {
      const int k = i / d, c = i % d;
      s_in[i] = inb[(size_t)k * a.ld_vec + c];
    }
  }
  __syncthreads();
  for (int k = warp; k < K; k += nw) {
    float ss = 0.f;
    for (int c = lane; c < d; c += 32) ss += s_in[k * d + c] * s_in[k * d + c];
    ss = warp_sum(ss);
    if (lane == 0) s_inn[k] = fmaxf(sqrtf(ss), UNIT_EPS);
  }
  __syncthreads();
  const int nrows = j == 0 ? 1 : K;
  for (int r = warp; r < nrows; r += nw) {
    const float* o = j == 0 ? a.anchor + (size_t)b * d
                            : a.out + ((size_t)(b * L + j - 1) * K + r) * a.ld_vec;
    if (v4 && d <= 512) {
      // the row in registers (up to 4 vectors per lane), four dot products at a time
      float4 ov[4];
      float oo = 0.f;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = 4 * (lane + 32 * u);
        ov[u] = c < d ? __ldcg(reinterpret_cast<const float4*>(o + c)) : make_float4(0.f, 0.f, 0.f, 0.f);
        oo = fmaf(ov[u].x, ov[u].x, fmaf(ov[u].y, ov[u].y, fmaf(ov[u].z, ov[u].z, fmaf(ov[u].w, ov[u].w, oo))));
      }
      const float on = fmaxf(sqrtf(warp_sum(oo)), UNIT_EPS);
      for (int k0 = 0; k0 < K; k0 += 4) {
        float dot[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int c = 4 * (lane + 32 * u);
          if (c >= d) break;
#pragma unroll
          for (int qq = 0; qq < 4; ++qq)
            if (k0 + qq < K) {
              const float4 w = *reinterpret_cast<const float4*>(s_in + (size_t)(k0 + qq) * d + c);
              dot[qq] = fmaf(ov[u].x, w.x, fmaf(ov[u].y, w.y, fmaf(ov[u].z, w.z, fmaf(ov[u].w, w.w, dot[qq]))));
            }
        }
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) dot[qq] = warp_sum(dot[qq]);
        if (lane == 0) {
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) {
            const int k2 = k0 + qq;
            if (k2 >= K) break;
            const float v = dot[qq] / (on * s_inn[k2]);
            if (j == 0) a.A[(size_t)b * K + k2] = v;
            else a.P[((size_t)b * (L - 1) + (j - 1)) * K * K + (size_t)r * K + k2] = v;
          }
        }
      }
      continue;
    }
    float oo = 0.f;
    for (int c = lane; c < d; c += 32) oo = fmaf(o[c], o[c], oo);
    const float on = fmaxf(sqrtf(warp_sum(oo)), UNIT_EPS);
    for (int k0 = 0; k0 < K; k0 += 4) {          // four dot products at a time
      float dot[4] = {0.f, 0.f, 0.f, 0.f};
      for (int c = lane; c < d; c += 32) {
        const float x = o[c];
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (k0 + q < K) dot[q] = fmaf(x, s_in[(k0 + q) * d + c], dot[q]);
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) dot[q] = warp_sum(dot[q]);
      if (lane == 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int k2 = k0 + q;
          if (k2 >= K) break;
          const float v = dot[q] / (on * s_inn[k2]);
          if (j == 0) a.A[(size_t)b * K + k2] = v;
          else a.P[((size_t)b * (L - 1) + (j - 1)) * K * K + (size_t)r * K + k2] = v;
        }
      }
    }
  }
  if (!a.do_walk) return;
  walk_after_pairs(a, sm, &s_last, s_back, s_path);
}

__global__ void __launch_bounds__(PW_THREADS) walk_kernel(PairWalkArgs a) {
  pdl_wait();
  extern __shared__ float sm[];
  __shared__ uint8_t s_back[LILICORR_MAX_L * LILICORR_MAX_K];
  __shared__ uint8_t s_path[LILICORR_MAX_L];
  const int b = blockIdx.x, L = a.L, K = a.K;
  const int n_scores = K + (L - 1) * K * K;
  const float* A = a.A + (size_t)b * K;
  const float* P = a.P + (size_t)b * (L - 1) * K * K;
  if (a.scores_in_smem) {
    stage_scores(sm, A, P, K, n_scores);
    __syncthreads();
    A = sm;
    P = sm + K;
  }
  if ((threadIdx.x >> 5) == 0) run_walk(a, A, P, b, s_back, s_path);
}

}  // namespace

// Shared memory the pair kernel needs at least (one slot's in vectors and norms).
size_t pair_walk_smem_bytes(int L, int K, int d) {
  (void)L;
  return sizeof(float) * ((size_t)K * d + K);
}

lilicorr_status_t launch_pair_walk(const PairWalkArgs& in, cudaStream_t st) {
  if (in.B == 0) return LILICORR_OK;
  PairWalkArgs a = in;
  const size_t score_bytes = sizeof(float) * ((size_t)a.K + (size_t)(a.L - 1) * a.K * a.K);
  a.scores_in_smem = score_bytes <= PW_SMEM_MAX;
  static bool cfg_pair[64] = {false}, cfg_walk[64] = {false};
  if (a.do_pairs) {
    if (a.do_walk && !a.counters) return LILICORR_ERR_ARG;
    // both slots' vectors staged: when that stays within 100 KB (two CTAs per SM at least)
    const size_t block_smem = sizeof(float) * (size_t)2 * a.K * pw_stride(a.d);
    if (block_smem <= 100 * 1024) {
      static bool cfg_block[64] = {false};
      size_t smem = block_smem;
      if (a.do_walk && a.scores_in_smem && score_bytes > smem) smem = score_bytes;
      LL_TRY(allow_max_dynamic_smem(pair_block_kernel, cfg_block));
      LL_TRY(launch_k(pair_block_kernel, dim3(a.B, a.L), PW_THREADS, smem, st, a));
      return LILICORR_OK;
    }
    size_t smem = pair_walk_smem_bytes(a.L, a.K, a.d);
    if (smem > PW_SMEM_MAX) return LILICORR_ERR_SHAPE;
    if (a.do_walk && a.scores_in_smem && score_bytes > smem) smem = score_bytes;
    LL_TRY(allow_max_dynamic_smem(pair_rows_kernel, cfg_pair));
    dim3 grid(a.B, a.L);
    LL_TRY(launch_k(pair_rows_kernel, grid, PW_THREADS, smem, st, a));
    return LILICORR_OK;
  }
  LL_TRY(allow_max_dynamic_smem(walk_kernel, cfg_walk));
  LL_TRY(launch_k(walk_kernel, a.B, PW_THREADS, a.scores_in_smem ? score_bytes : 0, st, a));
  return LILICORR_OK;
}

}  // namespace lilicorr
