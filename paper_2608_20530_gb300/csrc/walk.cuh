// The greedy walk of step (4) over one sequence's scores, shared by the pair kernel and
// the cluster network kernel's fused tail (Sec. 3.5: c_s = argmax_k phi(s-1, c_{s-1}, k),
// left to right, ties to the lower index).
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace lilicorr {
namespace walk {

// Best value (ties to the lower index), its index and the second-best value over the
// first `width` lanes (a power of two): one butterfly that carries the top two.
__device__ __forceinline__ void group_top2(float& v1, int& i1, float& v2, int width) {
  for (int o = width >> 1; o > 0; o >>= 1) {
    const float ov1 = __shfl_xor_sync(0xffffffffu, v1, o);
    const int oi1 = __shfl_xor_sync(0xffffffffu, i1, o);
    const float ov2 = __shfl_xor_sync(0xffffffffu, v2, o);
    if (ov1 > v1 || (ov1 == v1 && oi1 < i1)) {
      v2 = fmaxf(v1, ov2);
      v1 = ov1;
      i1 = oi1;
    } else {
      v2 = fmaxf(v2, ov1);
    }
  }
}

// Walk one sequence (called by one full warp). A [K], P [(L-1)][K][K] in any memory; the
// choices go to path[L] in shared memory (the tokens are gathered after the walk, so no
// step waits on a global load).
__device__ __forceinline__ void walk_sequence(const float* A, const float* P, int b, int L, int K,
                                              float* margin, uint8_t* path) {
  const int lane = threadIdx.x & 31;
  int width = 1;                                 // lanes that hold candidates, rounded up
  while (width < K) width <<= 1;
  int prev = 0;
  for (int s = 0; s < L; ++s) {
    const float* row = s == 0 ? A : P + ((size_t)(s - 1) * K + prev) * K;
    float best = lane < K ? row[lane] : -INFINITY, second = -INFINITY;
    int bi = lane < K ? lane : 0x7fffffff;
    group_top2(best, bi, second, width);
    bi = __shfl_sync(0xffffffffu, bi, 0);      // one choice for the warp, even on NaN rows
    if (bi < 0 || bi >= K) bi = 0;
    if (lane == 0) {
      path[s] = (uint8_t)bi;
      if (margin) margin[(size_t)b * L + s] = K > 1 ? best - second : INFINITY;
    }
    prev = bi;
  }
}

}  // namespace walk
}  // namespace lilicorr
