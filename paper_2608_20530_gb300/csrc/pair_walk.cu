// Steps (3) and (4): pair scores and the greedy walk.
//
// Eq. "pair": adjacent slots are coupled by the cosine between the earlier
// candidate's out vector and the later candidate's in vector; the anchor (the
// paper's slot 0) carries one out vector. Sec. 3.5: the (L-1) K^2 + K terms are
// one small matrix product per slot pair, and the walk commits left to right
// c_s = argmax_k phi(s-1, c_{s-1}, k), touching no weights.
//
// pair_block_kernel: grid (B, L). CTA (b, j) scores the anchor row (j = 0) or the slot
// pair (j-1, j): both slots' vectors are staged in shared memory and the outputs are
// formed in 4 x 4 blocks, 16 lanes per block. pair_rows_kernel, the same grid for vectors
// too long to stage twice (or rows off 16-byte boundaries): it stages slot j's K in
// vectors and their norms, every warp
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

// pair_block_kernel's staging: rows padded to a multiple of 4 per slot, row stride d + 4.
__host__ __device__ __forceinline__ int pb_rows(int K) { return (K + 3) / 4 * 4; }
__host__ __device__ __forceinline__ size_t pb_smem_bytes(int K, int d) {
  return sizeof(float) * (size_t)2 * pb_rows(K) * (d + 4);
}

__device__ __forceinline__ float dot4(const float4& x, const float4& y, float acc) {
  return fmaf(x.x, y.x, fmaf(x.y, y.y, fmaf(x.z, y.z, fmaf(x.w, y.w, acc))));
}

// Dot products of the 4 x 4 block of rows x (xr..xr+3, the earlier slot) and y (yr..yr+3,
// slot j) over the 16-byte columns f = split, split + 16, ... within [f0, f1); the thread's
// squared norms of those rows alongside when nx / ny are asked for.
__device__ __forceinline__ void block_dots(const float* sm, int ds, int xr, int yr, int f0, int f1,
                                           int split, bool want_nx, bool want_ny,
                                           float (&acc)[4][4], float (&nx)[4], float (&ny)[4]) {
  for (int f = f0 + split; f < f1; f += 16) {
    float4 xv[4], yv[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      xv[r] = *reinterpret_cast<const float4*>(sm + (size_t)(xr + r) * ds + 4 * f);
      yv[r] = *reinterpret_cast<const float4*>(sm + (size_t)(yr + r) * ds + 4 * f);
    }
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = dot4(xv[r], yv[c], acc[r][c]);
    if (want_nx)
#pragma unroll
      for (int r = 0; r < 4; ++r) nx[r] = dot4(xv[r], xv[r], nx[r]);
    if (want_ny)
#pragma unroll
      for (int c = 0; c < 4; ++c) ny[c] = dot4(yv[c], yv[c], ny[c]);
  }
}

// Sum over the 16 lanes that share a block (lanes 0-15 or 16-31 of the warp).
template <int N>
__device__ __forceinline__ void sum16(float (&v)[N]) {
#pragma unroll
  for (int o = 1; o < 16; o <<= 1)
#pragma unroll
    for (int i = 0; i < N; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], o);
}

// CTA (b, j): the slot pair (j - 1, j), or the anchor row (j = 0). The K in vectors of slot
// j (rows 0 .. K-1) and the earlier slot's out vectors or the anchor (rows R ..) are staged
// in shared memory by asynchronous copies in two column halves, so the products of the
// first half run while the second lands. The nrows x K outputs go in 4 x 4 blocks: thread t
// takes block t / 16 and the 16-byte columns t % 16, t % 16 + 16, ... of every row, so the
// 16 lanes of a block read 256 consecutive bytes of a row (no bank conflicts) and each
// loaded piece feeds four products; the 16 partial sums meet by shuffles. The row norms
// come out of the same pass (blocks of the first row / column group).
__global__ void __launch_bounds__(PW_THREADS) pair_block_kernel(PairWalkArgs a) {
  pdl_wait();
  extern __shared__ float sm[];
  __shared__ int s_last;
  __shared__ float s_nx[LILICORR_MAX_K], s_ny[LILICORR_MAX_K];
  __shared__ uint8_t s_back[LILICORR_MAX_L * LILICORR_MAX_K];
  __shared__ uint8_t s_path[LILICORR_MAX_L];
  const int b = blockIdx.x, j = blockIdx.y;
  const int L = a.L, K = a.K, d = a.d, ds = d + 4, d4 = d >> 2;
  const int R = pb_rows(K);                         // first row of the earlier slot
  const int nrows = j == 0 ? 1 : K;                 // vectors of the earlier slot (or anchor)
  const int nbx = (nrows + 3) >> 2, nby = R >> 2, nblk = nbx * nby;
  const float* inb = a.in + (size_t)(b * L + j) * K * a.ld_vec;
  const float* outb = j == 0 ? a.anchor + (size_t)b * d
                             : a.out + (size_t)(b * L + j - 1) * K * a.ld_vec;
  const int ldo = j == 0 ? d : a.ld_vec;
  const int h4 = (d4 + 1) >> 1;                     // 16-byte columns of the first half
  // stage both column halves (two commit groups), a warp per row and a lane per 16-byte
  // column; padding rows read as zero
  const int nr = R + 4 * nbx;
  const int wp = threadIdx.x >> 5, ln = threadIdx.x & 31;
  for (int h = 0; h < 2; ++h) {
    const int f0 = h ? h4 : 0, f1 = h ? d4 : h4;
    for (int row = wp; row < nr; row += PW_THREADS / 32) {
      const bool in_row = row < R;
      const int k = in_row ? row : row - R;
      float* dst = sm + (size_t)row * ds;
      if (k < (in_row ? K : nrows)) {
        const float* src = in_row ? inb + (size_t)k * a.ld_vec : outb + (size_t)k * ldo;
        for (int f = f0 + ln; f < f1; f += 32) cp16(dst + 4 * f, src + 4 * f);
      } else {
        for (int f = f0 + ln; f < f1; f += 32)
          *reinterpret_cast<float4*>(dst + 4 * f) = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  }

  const int split = threadIdx.x & 15;
  float* outp = j == 0 ? a.A + (size_t)b * K
                       : a.P + ((size_t)b * (L - 1) + (j - 1)) * K * K;
  // this lane's output of a reduced block: row 4 bx + split / 4, column 4 by + split % 4
  auto put = [&](int bx, int by, const float (&acc)[4][4]) {
    float v = 0.f;
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) v = split == 4 * r + c ? acc[r][c] : v;
    const int r = 4 * bx + (split >> 2), k2 = 4 * by + (split & 3);
    if (r < nrows && k2 < K) outp[(size_t)r * K + k2] = v / (s_nx[r] * s_ny[k2]);
  };
  auto put_norms = [&](int bx, int by, const float (&nx)[4], const float (&ny)[4]) {
    if (split != 0) return;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      if (by == 0 && 4 * bx + r < nrows) s_nx[4 * bx + r] = fmaxf(sqrtf(nx[r]), UNIT_EPS);
      if (bx == 0 && 4 * by + r < K) s_ny[4 * by + r] = fmaxf(sqrtf(ny[r]), UNIT_EPS);
    }
  };

  if (nblk <= PW_THREADS / 16) {
    // one block per thread (K <= 16): the first half's products while the second lands
    const int blk = threadIdx.x >> 4;
    const bool active = blk < nblk;
    const int bx = active ? blk / nby : 0, by = active ? blk % nby : 0;
    float acc[4][4] = {}, nx[4] = {}, ny[4] = {};
    asm volatile("cp.async.wait_group 1;" ::: "memory");
    __syncthreads();
    if (active) block_dots(sm, ds, R + 4 * bx, 4 * by, 0, h4, split, by == 0, bx == 0, acc, nx, ny);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    if (active) block_dots(sm, ds, R + 4 * bx, 4 * by, h4, d4, split, by == 0, bx == 0, acc, nx, ny);
    sum16(nx);
    sum16(ny);
    if (active) put_norms(bx, by, nx, ny);
    float flat[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) flat[i] = acc[i >> 2][i & 3];
    sum16(flat);
#pragma unroll
    for (int i = 0; i < 16; ++i) acc[i >> 2][i & 3] = flat[i];
    __syncthreads();                               // the norms
    if (active) put(bx, by, acc);
  } else {
    // more blocks than the CTA holds at once (K > 16): norms first, then block after block
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    for (int blk0 = 0; blk0 < nbx + nby; blk0 += PW_THREADS / 16) {
      // norms of row group blk (x rows for blk < nbx, else y rows), as blocks with bx or by 0
      // (the loop is warp-uniform: the sums below take every lane)
      const int blk = blk0 + (threadIdx.x >> 4);
      const bool act = blk < nbx + nby;
      float acc[4][4] = {}, nx[4] = {}, ny[4] = {};
      const bool xs = blk < nbx;
      const int bx = xs ? blk : 0, by = xs ? 0 : (act ? blk - nbx : 0);
      if (act) block_dots(sm, ds, R + 4 * bx, 4 * by, 0, d4, split, xs, !xs, acc, nx, ny);
      sum16(nx);
      sum16(ny);
      if (act && split == 0)
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          if (xs && 4 * bx + r < nrows) s_nx[4 * bx + r] = fmaxf(sqrtf(nx[r]), UNIT_EPS);
          if (!xs && 4 * by + r < K) s_ny[4 * by + r] = fmaxf(sqrtf(ny[r]), UNIT_EPS);
        }
    }
    __syncthreads();
    for (int blk0 = 0; blk0 < nblk; blk0 += PW_THREADS / 16) {
      const int blk = blk0 + (threadIdx.x >> 4);
      const bool active = blk < nblk;                // warp-uniform: 2 blocks per warp
      const int bx = active ? blk / nby : 0, by = active ? blk % nby : 0;
      float acc[4][4] = {}, nx[4], ny[4];
      if (active) block_dots(sm, ds, R + 4 * bx, 4 * by, 0, d4, split, false, false, acc, nx, ny);
      float flat[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) flat[i] = acc[i >> 2][i & 3];
      sum16(flat);
#pragma unroll
      for (int i = 0; i < 16; ++i) acc[i >> 2][i & 3] = flat[i];
      if (active) put(bx, by, acc);
    }
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
    // both slots' vectors staged, 16-byte pieces: when the rows are 16-byte aligned and the
    // staging stays within 100 KB (two CTAs per SM at least)
    const size_t block_smem = pb_smem_bytes(a.K, a.d);
    const bool v4 = ((a.d | a.ld_vec) & 3) == 0 && aligned16(a.in) && aligned16(a.out) &&
                    aligned16(a.anchor);
    if (v4 && block_smem <= 100 * 1024) {
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
