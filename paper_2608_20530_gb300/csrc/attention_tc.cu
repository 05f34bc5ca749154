// Step (2), the scoring Transformer's attention core on the bf16 head, with warp-level
// tensor-core instructions (mma.sync m16n8k16, bf16 operands, fp32 accumulation).
//
// App. A: every node attends to all L*K nodes of its sequence (no mask); the logits
// carry two learned per-head biases, dist[h, s_j - s_i + L - 1] and same[h] when the
// two nodes share a slot. One CTA takes (sequence b, head h, 64 queries); its K and V
// rows (bf16) and its queries are staged in shared memory (rows padded by 16 bytes so
// ldmatrix is conflict-free). Each warp owns 16 queries and sweeps the keys in blocks
// of 64 with an online softmax: S = Q K^T (ldmatrix + mma), scale, add the biases,
// running max / rescale, P = exp(S - max) packed to bf16 straight from the accumulator
// registers, O += P V (V fragments by ldmatrix.trans). O / rowsum is stored as bf16.
#include "internal.cuh"

namespace lilicorr {

namespace {

constexpr int AT_KBLK = 64;                  // keys per softmax block
constexpr float LOG2E = 1.4426950408889634f;

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void cp_async_16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;"
               ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// WARPS warps (16 queries each) share one staging of K and V: 4 when CTAs are scarce,
// 8 when there are plenty (twice the queries per staged key, and at 64-wide heads the
// shared memory of two CTAs then fills the register file's 16 warps per SM).
template <int HD, int WARPS>
__global__ void __launch_bounds__(WARPS * 32, HD <= 64 ? 16 / WARPS : 1)   // 16 warps per SM
attention_mma_kernel(const __nv_bfloat16* __restrict__ qkv, int L, int K, int D, int n_heads,
                     const float* __restrict__ dist, const float* __restrict__ same,
                     __nv_bfloat16* __restrict__ out) {
  pdl_wait();
  constexpr int AT_WARPS = WARPS;
  constexpr int AT_QROWS = 16 * WARPS;       // queries per CTA
  constexpr int HP = HD + 8;                 // padded row, elements
  constexpr int KS = HD / 16;                // k-steps of Q K^T
  constexpr int NB = HD / 8;                 // 8-wide dim blocks of O
  extern __shared__ __align__(16) uint8_t sm_raw[];
  const int LK = L * K;
  const int LKp = (LK + AT_KBLK - 1) / AT_KBLK * AT_KBLK;
  __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(sm_raw);
  __nv_bfloat16* Vs = Ks + (size_t)LKp * HP;
  __nv_bfloat16* Qs = Vs + (size_t)LKp * HP;
  float* s_dist = reinterpret_cast<float*>(Qs + (size_t)AT_QROWS * HP);
  uint8_t* s_slot = reinterpret_cast<uint8_t*>(s_dist + 2 * L - 1);   // slot of each key

  const int b = blockIdx.x / n_heads, h = blockIdx.x % n_heads;
  const int q0 = blockIdx.y * AT_QROWS;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t ld = 3 * (size_t)D;
  const __nv_bfloat16* base = qkv + (size_t)b * LK * ld + (size_t)h * HD;

  // ---- stage K, V (all keys, zero rows past LK) and this CTA's queries: asynchronous
  // copies, all issued before one wait
  constexpr int RV = HD / 8;                 // 16-byte vectors per row
  const uint4 zero = make_uint4(0, 0, 0, 0);
  for (int i = threadIdx.x; i < LKp * RV; i += AT_WARPS * 32) {
    const int j = i / RV, c = (i % RV) * 8;
    if (j < LK) {
      cp_async_16(Ks + (size_t)j * HP + c, base + (size_t)j * ld + D + c);
      cp_async_16(Vs + (size_t)j * HP + c, base + (size_t)j * ld + 2 * D + c);
    } else {
      *reinterpret_cast<uint4*>(Ks + (size_t)j * HP + c) = zero;
      *reinterpret_cast<uint4*>(Vs + (size_t)j * HP + c) = zero;
    }
  }
  for (int i = threadIdx.x; i < AT_QROWS * RV; i += AT_WARPS * 32) {
    const int j = i / RV, c = (i % RV) * 8;
    if (q0 + j < LK) cp_async_16(Qs + (size_t)j * HP + c, base + (size_t)(q0 + j) * ld + c);
    else *reinterpret_cast<uint4*>(Qs + (size_t)j * HP + c) = zero;
  }
  asm volatile("cp.async.commit_group;\n cp.async.wait_group 0;" ::: "memory");
  for (int i = threadIdx.x; i < 2 * L - 1; i += AT_WARPS * 32)
    s_dist[i] = dist[(size_t)h * (2 * L - 1) + i] * LOG2E;
  const bool k8 = (K & 7) == 0;
  if (!k8)
    for (int i = threadIdx.x; i < LK; i += AT_WARPS * 32) s_slot[i] = (uint8_t)(i / K);
  __syncthreads();

  const int g = lane >> 2, t = lane & 3;
  const int qrow = warp * 16;                // this warp's first query within the CTA
  // Q fragments for every k-step
  uint32_t qa[KS][4];
#pragma unroll
  for (int ks = 0; ks < KS; ++ks) {
    const int r = qrow + (lane & 15), c = ks * 16 + (lane >> 4) * 8;
    ldsm_x4(smem_addr(Qs + (size_t)r * HP + c), qa[ks]);
  }
  const int i0 = q0 + qrow + g, i1 = i0 + 8;  // the two query rows this thread holds
  const int si0 = min(i0 / K, L - 1), si1 = min(i1 / K, L - 1);   // padded rows: any slot
  const float same_l2 = same[h] * LOG2E;
  const float qscale = rsqrtf((float)HD) * LOG2E;

  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[NB][4];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb) o[nb][0] = o[nb][1] = o[nb][2] = o[nb][3] = 0.f;

  for (int kb = 0; kb < LKp; kb += AT_KBLK) {
    float s[8][4];
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) s[nb][0] = s[nb][1] = s[nb][2] = s[nb][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks)
#pragma unroll
      for (int nb = 0; nb < 8; nb += 2) {
        uint32_t bf[4];
        const int key = kb + nb * 8 + (lane & 7) + ((lane >> 4) << 3);
        const int col = ks * 16 + ((lane >> 3) & 1) * 8;
        ldsm_x4(smem_addr(Ks + (size_t)key * HP + col), bf);
        mma16816(s[nb], qa[ks], bf[0], bf[1]);
        mma16816(s[nb + 1], qa[ks], bf[2], bf[3]);
      }
    // scale, biases (log2 units), mask padded keys; block row maxima
    float bm0 = -INFINITY, bm1 = -INFINITY;
    if (k8) {
      // K % 8 == 0: the 8 keys of a tile share one slot, so one bias per query row
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
        const int jt = kb + nb * 8;
        const bool in = jt < LK;
        const int sj = jt / K;
        const float b0 = s_dist[sj - si0 + L - 1] + (si0 == sj ? same_l2 : 0.f);
        const float b1 = s_dist[sj - si1 + L - 1] + (si1 == sj ? same_l2 : 0.f);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float v = in ? fmaf(s[nb][e], qscale, e < 2 ? b0 : b1) : -INFINITY;
          s[nb][e] = v;
          if (e < 2) bm0 = fmaxf(bm0, v); else bm1 = fmaxf(bm1, v);
        }
      }
    } else {
#pragma unroll
      for (int nb = 0; nb < 8; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int j = kb + nb * 8 + 2 * t + (e & 1);
          const int si = e < 2 ? si0 : si1;
          float v;
          if (j < LK) {
            const int sj = s_slot[j];
            v = s[nb][e] * qscale + s_dist[sj - si + L - 1] + (si == sj ? same_l2 : 0.f);
          } else {
            v = -INFINITY;
          }
          s[nb][e] = v;
          if (e < 2) bm0 = fmaxf(bm0, v); else bm1 = fmaxf(bm1, v);
        }
    }
    bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 1));
    bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 2));
    bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 1));
    bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 2));
    const float mn0 = fmaxf(m0, bm0), mn1 = fmaxf(m1, bm1);
    const float c0 = ex2f(m0 - mn0), c1 = ex2f(m1 - mn1);   // 0 on the first block
    m0 = mn0;
    m1 = mn1;
    l0 *= c0;
    l1 *= c1;
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
      o[nb][0] *= c0; o[nb][1] *= c0;
      o[nb][2] *= c1; o[nb][3] *= c1;
    }
    // P = exp2(S - max), packed into bf16 A fragments of the next product
    uint32_t pa[4][4];
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
      const float p0 = ex2f(s[nb][0] - mn0), p1 = ex2f(s[nb][1] - mn0);
      const float p2 = ex2f(s[nb][2] - mn1), p3 = ex2f(s[nb][3] - mn1);
      l0 += p0 + p1;
      l1 += p2 + p3;
      const int kk = nb >> 1;
      if ((nb & 1) == 0) {
        pa[kk][0] = pack_bf16(p0, p1);
        pa[kk][1] = pack_bf16(p2, p3);
      } else {
        pa[kk][2] = pack_bf16(p0, p1);
        pa[kk][3] = pack_bf16(p2, p3);
      }
    }
    // O += P V over the 64 keys (4 k-steps of 16)
#pragma unroll
    for (int kk = 0; kk < 4; ++kk)
#pragma unroll
      for (int nb = 0; nb < NB; nb += 2) {
        uint32_t vf[4];
        const int key = kb + kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int col = nb * 8 + (lane >> 4) * 8;
        ldsm_x4_t(smem_addr(Vs + (size_t)key * HP + col), vf);
        mma16816(o[nb], pa[kk], vf[0], vf[1]);
        if (nb + 1 < NB) mma16816(o[nb + 1], pa[kk], vf[2], vf[3]);
      }
  }
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = 1.0f / l0, inv1 = 1.0f / l1;
#pragma unroll
  for (int nb = 0; nb < NB; ++nb) {
    const int c = h * HD + nb * 8 + 2 * t;
    if (i0 < LK)
      *reinterpret_cast<__nv_bfloat162*>(out + ((size_t)b * LK + i0) * D + c) =
          __floats2bfloat162_rn(o[nb][0] * inv0, o[nb][1] * inv0);
    if (i1 < LK)
      *reinterpret_cast<__nv_bfloat162*>(out + ((size_t)b * LK + i1) * D + c) =
          __floats2bfloat162_rn(o[nb][2] * inv1, o[nb][3] * inv1);
  }
}

template <int HD, int WARPS>
lilicorr_status_t launch_hdw(const __nv_bfloat16* qkv, int B, int L, int K, int D, int n_heads,
                             const float* dist, const float* same, __nv_bfloat16* out,
                             cudaStream_t st) {
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(attention_mma_kernel<HD, WARPS>, configured));
  const int LK = L * K;
  const int LKp = (LK + AT_KBLK - 1) / AT_KBLK * AT_KBLK;
  const size_t smem = sizeof(__nv_bfloat16) * (size_t)(2 * LKp + 16 * WARPS) * (HD + 8) +
                      sizeof(float) * (2 * L - 1) + LKp;
  dim3 grid(B * n_heads, ceil_div(LK, 16 * WARPS));
  LL_TRY(launch_k(attention_mma_kernel<HD, WARPS>, grid, WARPS * 32, smem, st, qkv, L, K, D,
                  n_heads, dist, same, out));
  return LILICORR_OK;
}

template <int HD>
lilicorr_status_t launch_hd(const __nv_bfloat16* qkv, int B, int L, int K, int D, int n_heads,
                            const float* dist, const float* same, __nv_bfloat16* out,
                            cudaStream_t st) {
  const long long ctas8 = (long long)B * n_heads * ceil_div(L * K, 128);
  if (L * K > 64 && ctas8 >= 2LL * num_sms())
    return launch_hdw<HD, 8>(qkv, B, L, K, D, n_heads, dist, same, out, st);
  return launch_hdw<HD, 4>(qkv, B, L, K, D, n_heads, dist, same, out, st);
}

}  // namespace

size_t attention_tc_smem_bytes(int LK, int hd, int L) {     // the larger (8-warp) layout
  const int LKp = (LK + AT_KBLK - 1) / AT_KBLK * AT_KBLK;
  return sizeof(__nv_bfloat16) * (size_t)(2 * LKp + 128) * (hd + 8) + sizeof(float) * (2 * L - 1) +
         LKp;
}

bool attention_tc_supported(int hd) { return hd == 16 || hd == 32 || hd == 64 || hd == 128; }

lilicorr_status_t launch_attention_tc(const void* qkv, int B, int L, int K, int D, int n_heads,
                                      const float* dist, const float* same, void* out,
                                      cudaStream_t st) {
  if (B == 0) return LILICORR_OK;
  const auto* q = static_cast<const __nv_bfloat16*>(qkv);
  auto* o = static_cast<__nv_bfloat16*>(out);
  switch (D / n_heads) {
    case 16: return launch_hd<16>(q, B, L, K, D, n_heads, dist, same, o, st);
    case 32: return launch_hd<32>(q, B, L, K, D, n_heads, dist, same, o, st);
    case 64: return launch_hd<64>(q, B, L, K, D, n_heads, dist, same, o, st);
    case 128: return launch_hd<128>(q, B, L, K, D, n_heads, dist, same, o, st);
  }
  return LILICORR_ERR_SHAPE;
}

}  // namespace lilicorr
