// Step (2), attention core of the unfused chain (App. A: bidirectional attention over the
// L*K nodes with the signed slot-distance and same-slot biases) on the tcgen05 tensor
// cores, for 32- and 64-wide heads and up to 256 nodes per sequence.
//
// CTA = (sequence, head, 128 queries), 256 threads: two per query row (tensor-memory
// lane), each taking half of the keys. Q, K and V rows (zero-padded to 64 columns) are
// staged in shared memory as 128-byte-swizzled rows: for Q and K that is the K-major
// operand layout of S = Q K^T; for V it is the MN-major layout of the B operand of P V
// (the 64 head columns of a key contiguous, keys 128 bytes apart, 8-key groups 1024 bytes
// apart), so V needs no transpose. One thread issues
//   S = Q K^T      (M 128, N = keys padded to 64, K 64)           into tensor memory,
// the threads turn their rows of S into probabilities (scale and biases in log2 units,
// padded keys masked, two passes: maximum, then 2^(s - max) as bf16 into shared memory
// over the dead Q and K tiles, with the row sums), and one thread issues
//   O = P V        (M 128, N 64, K = keys)                         over S's columns;
// the threads scale their rows of O by 1 / sum and store them. Waits are bounded.
#include "internal.cuh"
#include "tc_ptx.cuh"

namespace lilicorr {

namespace {
using namespace tc;

constexpr int UA_THREADS = 256;               // two threads per query row
constexpr int UA_MAX_KEYS = 256;
constexpr uint32_t UA_TMEM = 256;
constexpr uint32_t UA_CHUNK = 128 * 128;       // 128 rows x 128 bytes
constexpr long long UA_WAIT = 4000000000ll;
constexpr float UA_LOG2E = 1.4426950408889634f;

__device__ __forceinline__ float ex2u(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// Packed fp32 pairs: one instruction for both halves.
__device__ __forceinline__ uint64_t pk2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void upk2(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.ftz.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.ftz.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src)
               : "memory");
}

// Shared-memory bytes of one CTA (beyond the 1024-byte alignment slack): region A holds Q
// and K, later P; region B the V rows; then the distance biases, the key slots and two
// mbarriers.
__host__ __device__ constexpr size_t ua_region_a(int LKp) {
  return (size_t)(LKp / 64) * UA_CHUNK > UA_CHUNK + (size_t)LKp * 128
             ? (size_t)(LKp / 64) * UA_CHUNK
             : UA_CHUNK + (size_t)LKp * 128;
}
__host__ __device__ constexpr size_t ua_smem(int LKp, int HD, int L) {
  return 1024 + ua_region_a(LKp) + (size_t)LKp * 128 +
         ((sizeof(float) * (2 * L - 1) + LKp + 15) / 16) * 16 + 32;
}

template <int HD>
__global__ void __launch_bounds__(UA_THREADS, 2)
attention_umma_kernel(const __grid_constant__ CUtensorMap map_qkv, int use_tma,
                      const __nv_bfloat16* __restrict__ qkv, int L, int K, int D, int n_heads,
                      const float* __restrict__ dist, const float* __restrict__ same,
                      __nv_bfloat16* __restrict__ out, uint32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint32_t s_tmem;
  __shared__ float s_red[2][128];
  const int LK = L * K, LKp = (LK + 63) / 64 * 64, nkc = LKp / 64;
  uint8_t* sQ = sm;                                   // [128][64] bf16, swizzled
  uint8_t* sK = sm + UA_CHUNK;                        // [LKp][64] bf16, swizzled
  uint8_t* sP = sm;                                   // nkc chunks of [128][64 keys] bf16
  uint8_t* sV = sm + ua_region_a(LKp);                // [LKp][64] bf16, swizzled rows
  float* s_dist = reinterpret_cast<float*>(sV + (size_t)LKp * 128);
  uint8_t* s_slot = reinterpret_cast<uint8_t*>(s_dist + 2 * L - 1);
  uint64_t* bars = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(s_slot + LKp) + 7) & ~static_cast<uintptr_t>(7));
  uint64_t* bar_s = bars;
  uint64_t* bar_o = bars + 1;
  uint64_t* bar_qk = bars + 2;                        // TMA staging: Q and K, then V
  uint64_t* bar_v = bars + 3;

  const int tid = threadIdx.x, warp = tid >> 5;
  // the query tiles of one (sequence, head) are neighbours in the grid, so the second
  // tile's K and V rows come from L2
  const int b = blockIdx.y / n_heads, h = blockIdx.y % n_heads;
  const int q0 = blockIdx.x * 128;
  const size_t ld = 3 * (size_t)D;
  const __nv_bfloat16* base = qkv + (size_t)b * LK * ld + (size_t)h * HD;

  if (warp == 0) tmem_alloc(&s_tmem, UA_TMEM);
  if (tid == 0) {
    mbar_init(bar_s, 1);
    mbar_init(bar_o, 1);
    mbar_init(bar_qk, 1);
    mbar_init(bar_v, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  pdl_wait();

  if (use_tma) {
    // 64-wide heads of 256-node sequences (no padding anywhere): Q, K and V as five
    // 128-row TMA boxes of the q|k|v buffer, issued by one thread, in the same swizzled
    // rows as the copies below
    if (tid == 0) {
      const int row0 = b * LK, col = h * HD;
      mbar_expect_tx(bar_qk, 3 * UA_CHUNK);
      tma_load_2d(sQ, &map_qkv, bar_qk, col, row0 + q0);
      tma_load_2d(sK, &map_qkv, bar_qk, D + col, row0);
      tma_load_2d(sK + UA_CHUNK, &map_qkv, bar_qk, D + col, row0 + 128);
      mbar_expect_tx(bar_v, 2 * UA_CHUNK);
      tma_load_2d(sV, &map_qkv, bar_v, 2 * D + col, row0);
      tma_load_2d(sV + UA_CHUNK, &map_qkv, bar_v, 2 * D + col, row0 + 128);
    }
  } else {
    // ---- staging: Q, K and V rows by asynchronous copies (zeros past the head width and
    // past the nodes) in two groups, Q and K first (S needs them), V second (it lands while
    // the probabilities are formed); the biases and the key slots
    const uint4 zero = make_uint4(0, 0, 0, 0);
    for (int i = tid; i < 128 * 8; i += UA_THREADS) {
      const int r = i >> 3, p = i & 7;
      uint8_t* dst = sQ + swz(r, p);
      if (p < HD / 8 && q0 + r < LK) cp16(dst, base + (size_t)(q0 + r) * ld + 8 * p);
      else *reinterpret_cast<uint4*>(dst) = zero;
    }
    for (int i = tid; i < LKp * 8; i += UA_THREADS) {
      const int j = i >> 3, p = i & 7;
      uint8_t* dk = sK + swz(j, p);
      if (p < HD / 8 && j < LK) cp16(dk, base + (size_t)j * ld + D + 8 * p);
      else *reinterpret_cast<uint4*>(dk) = zero;
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    for (int i = tid; i < LKp * 8; i += UA_THREADS) {
      const int j = i >> 3, p = i & 7;
      uint8_t* dv = sV + swz(j, p);
      if (p < HD / 8 && j < LK) cp16(dv, base + (size_t)j * ld + 2 * D + 8 * p);
      else *reinterpret_cast<uint4*>(dv) = zero;
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
  for (int i = tid; i < 2 * L - 1; i += UA_THREADS) s_dist[i] = dist[(size_t)h * (2 * L - 1) + i] * UA_LOG2E;
  for (int i = tid; i < LKp; i += UA_THREADS) s_slot[i] = (uint8_t)min(i / K, L - 1);
  asm volatile("cp.async.wait_group 1;" ::: "memory");       // Q and K
  fence_async_shared();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  bool ok = true;

  // ---- S = Q K^T
  if (tid == 0) {
    if (use_tma && !mbar_wait(bar_qk, 0, UA_WAIT)) ok = false;
    const uint64_t qd = smem_desc(sQ), kd = smem_desc(sK);
#pragma unroll
    for (int k = 0; k < 4; ++k) mma_bf16(tmem, qd + 2ull * k, kd + 2ull * k, instr_desc(128, LKp), k > 0);
    mma_commit(bar_s);
  }
  if (!mbar_wait(bar_s, 0, UA_WAIT)) ok = false;
  tc_fence_after();

  // ---- probabilities of this thread's query row, over its half of the keys
  const int row = tid & 127, half = tid >> 7;
  const int q = q0 + row;
  const int si = s_slot[min(q, LK - 1)];
  const float qscale = rsqrtf((float)HD) * UA_LOG2E;
  const float same_l2 = same[h] * UA_LOG2E;
  const uint32_t trow = tmem + ((uint32_t)((warp & 3) * 32) << 16);
  const int kh = LKp / 2, kbeg = half * kh, kend = kbeg + kh;
  const bool k8 = (K & 7) == 0;
  // the key's logit in log2 units (bias from the slot distance and same-slot term)
  auto logit = [&](float sv, int j) {
    const int sj = s_slot[j];
    return j < LK ? fmaf(sv, qscale, s_dist[sj - si + L - 1] + (sj == si ? same_l2 : 0.f))
                  : -INFINITY;
  };
  float mx = -INFINITY;
  float sum = 0.f;
  if (k8 && LK == UA_MAX_KEYS) {
    // Every key real and 8-key groups sharing a slot: the 16 group biases of this half row
    // in registers; the maximum over the raw scores of a group first (the scale is positive,
    // so the largest logit of the group is that score mapped once), then the probabilities
    // on fp32 pairs.
    float bg[UA_MAX_KEYS / 16];
#pragma unroll
    for (int gi = 0; gi < UA_MAX_KEYS / 16; ++gi) {
      const int sj = s_slot[kbeg + 8 * gi];
      bg[gi] = s_dist[sj - si + L - 1] + (sj == si ? same_l2 : 0.f);
    }
#pragma unroll
    for (int ch = 0; ch < UA_MAX_KEYS / 64; ++ch) {
      uint32_t r[32];
      tmem_ld32(trow + kbeg + 32 * ch, r);
#pragma unroll
      for (int g8 = 0; g8 < 4; ++g8) {
        float m8 = __uint_as_float(r[8 * g8]);
#pragma unroll
        for (int e = 1; e < 8; ++e) m8 = fmaxf(m8, __uint_as_float(r[8 * g8 + e]));
        mx = fmaxf(mx, fmaf(m8, qscale, bg[4 * ch + g8]));
      }
    }
    s_red[half][row] = mx;
    __syncthreads();
    mx = fmaxf(s_red[0][row], s_red[1][row]);
    const uint64_t qs2 = pk2(qscale, qscale);
    uint64_t acc = pk2(0.f, 0.f);
#pragma unroll
    for (int ch = 0; ch < UA_MAX_KEYS / 64; ++ch) {
      uint32_t r[32];
      tmem_ld32(trow + kbeg + 32 * ch, r);
      uint32_t pk[16];
#pragma unroll
      for (int g8 = 0; g8 < 4; ++g8) {
        const float bm = bg[4 * ch + g8] - mx;
        const uint64_t bm2 = pk2(bm, bm);
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
          float t0, t1;
          upk2(ffma2(pk2(__uint_as_float(r[8 * g8 + e]), __uint_as_float(r[8 * g8 + e + 1])), qs2,
                     bm2),
               t0, t1);
          const float p0 = ex2u(t0), p1 = ex2u(t1);
          acc = fadd2(acc, pk2(p0, p1));
          pk[(8 * g8 + e) >> 1] = pack_bf16x2(p0, p1);
        }
      }
      const int c0 = kbeg + 32 * ch;
      uint8_t* chunk = sP + (size_t)(c0 >> 6) * UA_CHUNK;
      const int piece0 = (c0 & 63) >> 3;
#pragma unroll
      for (int u = 0; u < 4; ++u)
        *reinterpret_cast<uint4*>(chunk + swz(row, piece0 + u)) =
            make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
    }
    float a0, a1;
    upk2(acc, a0, a1);
    sum = a0 + a1;
  } else {
  for (int c0 = kbeg; c0 < kend; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(trow + c0, r);
    if (k8) {
#pragma unroll
      for (int g8 = 0; g8 < 4; ++g8) {
        const int j0 = c0 + 8 * g8, sj = s_slot[j0];
        const float bias = s_dist[sj - si + L - 1] + (sj == si ? same_l2 : 0.f);
#pragma unroll
        for (int e = 0; e < 8; ++e)
          mx = fmaxf(mx, j0 + e < LK ? fmaf(__uint_as_float(r[8 * g8 + e]), qscale, bias) : -INFINITY);
      }
    } else {
#pragma unroll
      for (int e = 0; e < 32; ++e) mx = fmaxf(mx, logit(__uint_as_float(r[e]), c0 + e));
    }
  }
  s_red[half][row] = mx;
  __syncthreads();
  mx = fmaxf(s_red[0][row], s_red[1][row]);
  for (int c0 = kbeg; c0 < kend; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(trow + c0, r);
    float pv[32];
    if (k8) {
#pragma unroll
      for (int g8 = 0; g8 < 4; ++g8) {
        const int j0 = c0 + 8 * g8, sj = s_slot[j0];
        const float bias = s_dist[sj - si + L - 1] + (sj == si ? same_l2 : 0.f);
#pragma unroll
        for (int e = 0; e < 8; ++e)
          pv[8 * g8 + e] = j0 + e < LK ? ex2u(fmaf(__uint_as_float(r[8 * g8 + e]), qscale, bias) - mx)
                                       : 0.f;
      }
    } else {
#pragma unroll
      for (int e = 0; e < 32; ++e) pv[e] = ex2u(logit(__uint_as_float(r[e]), c0 + e) - mx);
    }
    uint32_t pk[16];
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
      sum += pv[e] + pv[e + 1];
      pk[e >> 1] = pack_bf16x2(pv[e], pv[e + 1]);
    }
    uint8_t* chunk = sP + (size_t)(c0 >> 6) * UA_CHUNK;
    const int piece0 = (c0 & 63) >> 3;
#pragma unroll
    for (int u = 0; u < 4; ++u)
      *reinterpret_cast<uint4*>(chunk + swz(row, piece0 + u)) =
          make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
  }
  }
  __syncthreads();                                   // both halves' maxima read
  s_red[half][row] = sum;
  asm volatile("cp.async.wait_group 0;" ::: "memory");       // V
  fence_async_shared();
  tc_fence_before();
  __syncthreads();                                   // every row of P written, S read
  tc_fence_after();
  const float inv = 1.0f / (s_red[0][row] + s_red[1][row]);

  // ---- O = P V over S's first 64 columns; V is the MN-major B operand (instruction
  // descriptor bit 16), each K step of 16 keys starting 16 rows (2048 bytes) further on
  if (tid == 0) {
    if (use_tma && !mbar_wait(bar_v, 0, UA_WAIT)) ok = false;
    constexpr uint32_t idesc_pv = instr_desc(128, 64) | (1u << 16);
    for (int kc = 0; kc < nkc; ++kc) {
      const uint64_t pd = smem_desc(sP + (size_t)kc * UA_CHUNK);
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_bf16(tmem, pd + 2ull * k, smem_desc(sV + (size_t)(64 * kc + 16 * k) * 128), idesc_pv,
                 (kc | k) > 0);
    }
    mma_commit(bar_o);
  }
  if (!mbar_wait(bar_o, 0, UA_WAIT)) ok = false;
  tc_fence_after();

  // ---- this row of O, normalised, as bf16 (32 columns per thread)
  for (int c0 = 32 * half; c0 < HD; c0 += 64) {
    uint32_t r[32];
    tmem_ld32(trow + c0, r);
    if (q < LK && ok) {
      __nv_bfloat16* dst = out + ((size_t)b * LK + q) * D + (size_t)h * HD + c0;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        uint4 w;
        w.x = pack_bf16x2(__uint_as_float(r[8 * u]) * inv, __uint_as_float(r[8 * u + 1]) * inv);
        w.y = pack_bf16x2(__uint_as_float(r[8 * u + 2]) * inv, __uint_as_float(r[8 * u + 3]) * inv);
        w.z = pack_bf16x2(__uint_as_float(r[8 * u + 4]) * inv, __uint_as_float(r[8 * u + 5]) * inv);
        w.w = pack_bf16x2(__uint_as_float(r[8 * u + 6]) * inv, __uint_as_float(r[8 * u + 7]) * inv);
        *reinterpret_cast<uint4*>(dst + 8 * u) = w;
      }
    }
  }
  if (!ok && status && tid == 0) set_status(status, LILICORR_ERR_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, UA_TMEM);
  }
}

template <int HD>
lilicorr_status_t launch_umma_hd(const __nv_bfloat16* qkv, int B, int L, int K, int D,
                                 int n_heads, const float* dist, const float* same,
                                 __nv_bfloat16* out, uint32_t* status, cudaStream_t st) {
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(attention_umma_kernel<HD>, configured));
  const int LK = L * K, LKp = (LK + 63) / 64 * 64;
  dim3 grid(ceil_div(LK, 128), B * n_heads);
  // TMA staging where no row or column is padded: 64-wide heads, 256-node sequences
  CUtensorMap map;
  memset(&map, 0, sizeof(map));
  const int use_tma = HD == 64 && LK == UA_MAX_KEYS;
  if (use_tma && !make_map(&map, qkv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, B * LK, 3 * D, 3 * D,
                           128, 64))
    return LILICORR_ERR_CUDA;
  LL_TRY(launch_k(attention_umma_kernel<HD>, grid, UA_THREADS, ua_smem(LKp, HD, L), st, map,
                  use_tma, qkv, L, K, D, n_heads, dist, same, out, status));
  return LILICORR_OK;
}

}  // namespace

bool attention_umma_supported(int L, int K, int D, int n_heads) {
  const int hd = D / n_heads;
  return (hd == 32 || hd == 64) && hd * n_heads == D && L * K >= 1 && L * K <= UA_MAX_KEYS &&
         L <= 128 && D % 8 == 0;
}

lilicorr_status_t launch_attention_umma(const void* qkv, int B, int L, int K, int D, int n_heads,
                                        const float* dist, const float* same, void* out,
                                        uint32_t* status, cudaStream_t st) {
  if (B == 0) return LILICORR_OK;
  if (!attention_umma_supported(L, K, D, n_heads)) return LILICORR_ERR_SHAPE;
  const auto* q = static_cast<const __nv_bfloat16*>(qkv);
  auto* o = static_cast<__nv_bfloat16*>(out);
  if (D / n_heads == 32) return launch_umma_hd<32>(q, B, L, K, D, n_heads, dist, same, o, status, st);
  return launch_umma_hd<64>(q, B, L, K, D, n_heads, dist, same, o, status, st);
}

}  // namespace lilicorr
