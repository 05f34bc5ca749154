// Step (2): the scoring network's fp32 CUDA-core kernels (Sec. 3.2; App. A "Architecture").
//
// Node construction, RMSNorm, target state, bidirectional attention with the two
// learned bias tables, the fusion input and row normalisation, plus a tiled
// fp32 linear layer with fused bias / per-sequence bias / SiLU / residual
// epilogue. The fp32 head runs every matrix product here; the bf16 head runs its
// large products on the tensor cores (gemm_tc.cu) and the rest here.
#include "internal.cuh"

namespace lilicorr {

namespace {

constexpr float RMS_EPS = 1e-6f;
constexpr float UNIT_EPS = 1e-12f;

// ----------------------------------------------------------------------------- linear
constexpr int GB_M = 64, GB_N = 64, GB_K = 16, G_THREADS = 256;

template <typename TA, typename TW, typename TC>
__global__ void __launch_bounds__(G_THREADS) gemm_simt_kernel(GemmArgs g) {
  pdl_wait();
  __shared__ float As[GB_K][GB_M + 4];
  __shared__ __align__(16) float Ws[GB_K][GB_N + 4];
  const TA* A = static_cast<const TA*>(g.A);
  const TW* W = static_cast<const TW*>(g.W);
  const int tid = threadIdx.x;
  const int m0 = blockIdx.y * GB_M, n0 = blockIdx.x * GB_N;
  const int tx = tid & 15, ty = tid >> 4;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < g.Kd; k0 += GB_K) {
#pragma unroll
    for (int i = tid; i < GB_M * GB_K; i += G_THREADS) {
      const int r = i / GB_K, c = i % GB_K;
      const int gm = m0 + r, gk = k0 + c;
      As[c][r] = (gm < g.M && gk < g.Kd) ? ld_elem(A, (size_t)gm * g.lda + gk) : 0.f;
      const int gn = n0 + r;
      Ws[c][r] = (gn < g.N && gk < g.Kd) ? ld_elem(W, (size_t)gn * g.ldw + gk) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GB_K; ++kk) {
      float a[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
      const float4 b = *reinterpret_cast<const float4*>(&Ws[kk][tx * 4]);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        acc[i][0] = fmaf(a[i], b.x, acc[i][0]);
        acc[i][1] = fmaf(a[i], b.y, acc[i][1]);
        acc[i][2] = fmaf(a[i], b.z, acc[i][2]);
        acc[i][3] = fmaf(a[i], b.w, acc[i][3]);
      }
    }
    __syncthreads();
  }
  TC* C = static_cast<TC*>(g.C);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= g.N) continue;
      float v = acc[i][j];
      if (g.bias) v += g.bias[n];
      if (g.bias_rows) v += g.bias_rows[(size_t)(m / g.rows_per_bias) * g.N + n];
      if (g.act == ACT_SILU) v = silu_f(v);
      if (g.residual) v += g.residual[(size_t)m * g.ldr + n];
      st_elem(C, (size_t)m * g.ldc + n, v);
    }
  }
}

template <typename TA, typename TW>
lilicorr_status_t gemm_dispatch_c(const GemmArgs& g, dim3 grid, cudaStream_t st) {
  if (g.c_dt == LILICORR_F32) LL_TRY(launch_k(gemm_simt_kernel<TA, TW, float>, grid, G_THREADS, 0, st, g));
  else LL_TRY(launch_k(gemm_simt_kernel<TA, TW, __nv_bfloat16>, grid, G_THREADS, 0, st, g));
  return LILICORR_OK;
}
template <typename TA>
lilicorr_status_t gemm_dispatch_w(const GemmArgs& g, dim3 grid, cudaStream_t st) {
  if (g.w_dt == LILICORR_F32) return gemm_dispatch_c<TA, float>(g, grid, st);
  return gemm_dispatch_c<TA, __nv_bfloat16>(g, grid, st);
}

// ----------------------------------------------------------------------------- skinny linear
// Few rows (M <= 64: one row per slot or per sequence) against long rows (Kd up to H).
// CTA (column block of SK_NB, row block of SK_MB): its 256 threads split Kd in
// 8-element vectors, each accumulating SK_MB x SK_NB partial dot products, reduced by
// warp shuffles and shared memory. Many CTAs stream disjoint weight rows.
constexpr int SK_NB = 4, SK_MB = 16, SK_THREADS = 256;

__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 a = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[2 * i] = __uint_as_float(w[i] << 16);
    v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

template <typename TA, typename TW, typename TC, int MB>
__global__ void __launch_bounds__(SK_THREADS) gemm_skinny_kernel(GemmArgs g) {
  pdl_wait();
  __shared__ float red[SK_THREADS / 32][MB * SK_NB];
  const TA* A = static_cast<const TA*>(g.A);
  const TW* W = static_cast<const TW*>(g.W);
  const int n0 = blockIdx.x * SK_NB, m0 = blockIdx.y * MB;
  const int nb = min(SK_NB, g.N - n0), mb = min(MB, g.M - m0);
  float acc[MB][SK_NB];
#pragma unroll
  for (int i = 0; i < MB; ++i)
#pragma unroll
    for (int j = 0; j < SK_NB; ++j) acc[i][j] = 0.f;
  for (int k = threadIdx.x * 8; k < g.Kd; k += SK_THREADS * 8) {
    float w[SK_NB][8];
#pragma unroll
    for (int j = 0; j < SK_NB; ++j) {
      if (j < nb) load8(W + (size_t)(n0 + j) * g.ldw + k, w[j]);
      else
#pragma unroll
        for (int e = 0; e < 8; ++e) w[j][e] = 0.f;
    }
    // all row loads first (predicated, no early exit) so they are in flight together
    float a[MB][8];
#pragma unroll
    for (int i = 0; i < MB; ++i) {
      if (i < mb) load8(A + (size_t)(m0 + i) * g.lda + k, a[i]);
      else
#pragma unroll
        for (int e = 0; e < 8; ++e) a[i][e] = 0.f;
    }
#pragma unroll
    for (int i = 0; i < MB; ++i)
#pragma unroll
      for (int j = 0; j < SK_NB; ++j)
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[i][j] = fmaf(a[i][e], w[j][e], acc[i][j]);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < MB; ++i) {
    if (i >= mb) break;                            // rows past M: nothing to reduce
#pragma unroll
    for (int j = 0; j < SK_NB; ++j) {
      const float v = warp_sum(acc[i][j]);
      if (lane == 0) red[warp][i * SK_NB + j] = v;
    }
  }
  __syncthreads();
  if (threadIdx.x < MB * SK_NB) {
    const int i = threadIdx.x / SK_NB, j = threadIdx.x % SK_NB;
    if (i < mb && j < nb) {
      float v = 0.f;
#pragma unroll
      for (int w = 0; w < SK_THREADS / 32; ++w) v += red[w][threadIdx.x];
      const int m = m0 + i, n = n0 + j;
      if (g.bias) v += g.bias[n];
      if (g.bias_rows) v += g.bias_rows[(size_t)(m / g.rows_per_bias) * g.N + n];
      if (g.act == ACT_SILU) v = silu_f(v);
      if (g.residual) v += g.residual[(size_t)m * g.ldr + n];
      st_elem(static_cast<TC*>(g.C), (size_t)m * g.ldc + n, v);
    }
  }
}

// ----------------------------------------------------------------------------- row-block linear
// Per-sequence products with fp32 activations and more rows than the few-row kernel takes
// (the target state t of a batch against W_a and the fusion layer's t block: M = B up to
// 1024, Kd = D). CTA = 16 rows x 32 columns: lane = output column, warp = two rows. Per
// chunk of Kd, the 16 activation rows and the 32 weight rows are staged in shared memory by
// one round of asynchronous 16-byte copies (all in flight at once, coalesced); each lane
// then reads its weight row and the warp's two activation rows (broadcasts). No
// cross-lane reduction.
constexpr int GR_M = 16, GR_N = 32, GR_THREADS = 256;
__device__ __forceinline__ void cp16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;"
               ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src) : "memory");
}
template <typename TW>
struct GrCfg {
  static constexpr int KC = sizeof(TW) == 2 ? 256 : 128;      // Kd chunk staged at a time
  static constexpr int AS = KC + 4;                           // row strides (elements), padded
  static constexpr int WS = KC + 16 / (int)sizeof(TW);        // so 8 lanes' 16-byte reads differ in bank
};
template <typename TW, typename TC>
__global__ void __launch_bounds__(GR_THREADS) gemm_rows_kernel(GemmArgs g) {
  pdl_wait();
  using Cfg = GrCfg<TW>;
  constexpr int KC = Cfg::KC, AS = Cfg::AS, WS = Cfg::WS;
  constexpr int WV = 16 / (int)sizeof(TW);                    // weights per 16-byte piece
  __shared__ __align__(16) float As[GR_M * AS];
  __shared__ __align__(16) TW Ws[GR_N * WS];
  const float* A = static_cast<const float*>(g.A);
  const TW* W = static_cast<const TW*>(g.W);
  const int m0 = blockIdx.y * GR_M, n0 = blockIdx.x * GR_N;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int n = n0 + lane, r0 = 2 * warp;
  float acc0 = 0.f, acc1 = 0.f;
  for (int k0 = 0; k0 < g.Kd; k0 += KC) {
    const int kc = min(KC, g.Kd - k0);                          // a multiple of 8
    __syncthreads();                                            // the previous chunk is consumed
    for (int i = threadIdx.x; i < GR_M * (kc / 4); i += GR_THREADS) {
      const int r = i / (kc / 4), c = 4 * (i % (kc / 4));
      float* dst = &As[r * AS + c];
      if (m0 + r < g.M) cp16(dst, A + (size_t)(m0 + r) * g.lda + k0 + c);
      else *reinterpret_cast<float4*>(dst) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    for (int i = threadIdx.x; i < GR_N * (kc / WV); i += GR_THREADS) {
      const int r = i / (kc / WV), c = WV * (i % (kc / WV));
      TW* dst = &Ws[r * WS + c];
      if (n0 + r < g.N) cp16(dst, W + (size_t)(n0 + r) * g.ldw + k0 + c);
      else *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    const TW* wr = &Ws[lane * WS];
    const float* a0p = &As[r0 * AS];
    const float* a1p = a0p + AS;
#pragma unroll 4
    for (int k = 0; k < kc; k += 8) {
      float w[8];
      load8(wr + k, w);
      const float4 a0 = *reinterpret_cast<const float4*>(a0p + k);
      const float4 a1 = *reinterpret_cast<const float4*>(a0p + k + 4);
      const float4 b0 = *reinterpret_cast<const float4*>(a1p + k);
      const float4 b1 = *reinterpret_cast<const float4*>(a1p + k + 4);
      acc0 = fmaf(a0.x, w[0], fmaf(a0.y, w[1], fmaf(a0.z, w[2], fmaf(a0.w, w[3], acc0))));
      acc0 = fmaf(a1.x, w[4], fmaf(a1.y, w[5], fmaf(a1.z, w[6], fmaf(a1.w, w[7], acc0))));
      acc1 = fmaf(b0.x, w[0], fmaf(b0.y, w[1], fmaf(b0.z, w[2], fmaf(b0.w, w[3], acc1))));
      acc1 = fmaf(b1.x, w[4], fmaf(b1.y, w[5], fmaf(b1.z, w[6], fmaf(b1.w, w[7], acc1))));
    }
  }
  if (n >= g.N) return;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int m = m0 + r0 + i;
    if (m >= g.M) continue;
    float v = i ? acc1 : acc0;
    if (g.bias) v += g.bias[n];
    if (g.bias_rows) v += g.bias_rows[(size_t)(m / g.rows_per_bias) * g.N + n];
    if (g.act == ACT_SILU) v = silu_f(v);
    if (g.residual) v += g.residual[(size_t)m * g.ldr + n];
    st_elem(static_cast<TC*>(g.C), (size_t)m * g.ldc + n, v);
  }
}

template <typename TA, typename TW, int MB>
lilicorr_status_t skinny_dispatch_m(const GemmArgs& g, cudaStream_t st) {
  dim3 grid(ceil_div(g.N, SK_NB), ceil_div(g.M, MB));
  if (g.c_dt == LILICORR_F32) LL_TRY(launch_k(gemm_skinny_kernel<TA, TW, float, MB>, grid, SK_THREADS, 0, st, g));
  else LL_TRY(launch_k(gemm_skinny_kernel<TA, TW, __nv_bfloat16, MB>, grid, SK_THREADS, 0, st, g));
  return LILICORR_OK;
}
// rows per CTA: one per sequence-level row (M = 1), four for a few, else sixteen
template <typename TA, typename TW>
lilicorr_status_t skinny_dispatch_c(const GemmArgs& g, dim3 grid, cudaStream_t st) {
  (void)grid;
  if (g.M == 1) return skinny_dispatch_m<TA, TW, 1>(g, st);
  if (g.M <= 4) return skinny_dispatch_m<TA, TW, 4>(g, st);
  return skinny_dispatch_m<TA, TW, SK_MB>(g, st);
}
template <typename TA>
lilicorr_status_t skinny_dispatch_w(const GemmArgs& g, dim3 grid, cudaStream_t st) {
  if (g.w_dt == LILICORR_F32) return skinny_dispatch_c<TA, float>(g, grid, st);
  return skinny_dispatch_c<TA, __nv_bfloat16>(g, grid, st);
}

// ----------------------------------------------------------------------------- target state
// tn[b] = RMSNorm_H(mean over the n_tgt captured layers of T[b]) * gain (App. A).
// One CTA per sequence; each thread owns 8-element vectors of the row (H % 8 == 0),
// keeps its means in registers between the two passes (up to TN_VPT vectors).
constexpr int TN_THREADS = 512, TN_VPT = 4;

template <typename T, typename TO>
__global__ void __launch_bounds__(TN_THREADS)
target_norm_kernel(const T* __restrict__ Tin, int n_tgt, int H, const float* __restrict__ gain,
                   TO* __restrict__ tn) {
  pdl_wait();
  __shared__ float red[TN_THREADS / 32];
  __shared__ float s_total;
  const int b = blockIdx.x;
  const T* tb = Tin + (size_t)b * n_tgt * H;
  const int nv = H / 8;
  float mean[TN_VPT][8];
  float ss = 0.f;
  const float inv_p = 1.0f / (float)n_tgt;
#pragma unroll
  for (int q = 0; q < TN_VPT; ++q) {
    const int v = threadIdx.x + q * TN_THREADS;
#pragma unroll
    for (int e = 0; e < 8; ++e) mean[q][e] = 0.f;
    if (v >= nv) continue;
    for (int l = 0; l < n_tgt; ++l) {
      float x[8];
      load8(tb + (size_t)l * H + v * 8, x);
#pragma unroll
      for (int e = 0; e < 8; ++e) mean[q][e] += x[e];
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      mean[q][e] *= inv_p;
      ss += mean[q][e] * mean[q][e];
    }
  }
  // rows longer than TN_VPT * TN_THREADS * 8 are handled by a second strided pass
  for (int v = threadIdx.x + TN_VPT * TN_THREADS; v < nv; v += TN_THREADS) {
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int l = 0; l < n_tgt; ++l) {
      float x[8];
      load8(tb + (size_t)l * H + v * 8, x);
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] += x[e];
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      acc[e] *= inv_p;
      ss += acc[e] * acc[e];
      st_elem(tn, (size_t)b * H + v * 8 + e, acc[e]);
    }
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < TN_THREADS / 32 ? red[threadIdx.x] : 0.f;
    v = warp_sum(v);
    if (threadIdx.x == 0) s_total = v;
  }
  __syncthreads();
  const float r = rsqrtf(s_total / (float)H + RMS_EPS);
#pragma unroll
  for (int q = 0; q < TN_VPT; ++q) {
    const int v = threadIdx.x + q * TN_THREADS;
    if (v >= nv) continue;
#pragma unroll
    for (int e = 0; e < 8; ++e)
      st_elem(tn, (size_t)b * H + v * 8 + e, mean[q][e] * r * gain[v * 8 + e]);
  }
  for (int v = threadIdx.x + TN_VPT * TN_THREADS; v < nv; v += TN_THREADS)
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const size_t o = (size_t)b * H + v * 8 + e;
      st_elem(tn, o, ld_elem(tn, o) * r * gain[v * 8 + e]);
    }
}

// ----------------------------------------------------------------------------- nodes
// One CTA per slot row r = b*L + s. For candidate k (Sec. 3.2; App. A):
//   c1 = SiLU(W_c1 f_k + b_c1)   (first layer of the confidence network; the second
//                                 layer is a linear launch that adds into x)
//   x  = fold[id_k] + hproj[r] + slot[s] + rank[k]
// with f_k = [logp_k, exp(logp_k), logp_0 - logp_k, k / (K-1), 1{k = 0}].
template <typename TC1>
__global__ void node_build_kernel(int L, int K, int D, int V, const int32_t* __restrict__ ids,
                                  const float* __restrict__ logp, const float* __restrict__ fold,
                                  const float* __restrict__ hproj, const float* __restrict__ slot,
                                  const float* __restrict__ rank, const float* __restrict__ w1,
                                  const float* __restrict__ b1, TC1* __restrict__ c1,
                                  float* __restrict__ x, uint32_t* status) {
  pdl_wait();
  __shared__ float f[LILICORR_MAX_K][LILICORR_N_CONF];
  __shared__ int sid[LILICORR_MAX_K];
  extern __shared__ __align__(16) float s_w[];     // [N_CONF][D] = W_c1^T, then b_c1 [D]
  const int r = blockIdx.x;
  const int s = r % L;
  for (int i = threadIdx.x; i < D; i += blockDim.x) {
#pragma unroll
    for (int j = 0; j < LILICORR_N_CONF; ++j) s_w[j * D + i] = w1[i * LILICORR_N_CONF + j];
    s_w[LILICORR_N_CONF * D + i] = b1[i];
  }
  if (threadIdx.x < K) {
    const int k = threadIdx.x;
    const float lp = logp[(size_t)r * K + k];
    const float lp0 = logp[(size_t)r * K];
    f[k][0] = lp;
    f[k][1] = expf(lp);
    f[k][2] = lp0 - lp;
    f[k][3] = K > 1 ? (float)k / (float)(K - 1) : 0.f;
    f[k][4] = k == 0 ? 1.f : 0.f;
    int id = ids[(size_t)r * K + k];
    if (id < 0 || id >= V) {          // an id outside the vocabulary: flag it, read row 0
      set_status(status, LILICORR_ERR_ARG);
      id = 0;
    }
    sid[k] = id;
  }
  __syncthreads();
  const int D4 = D / 4;
#pragma unroll 2
  for (int i = threadIdx.x; i < K * D4; i += blockDim.x) {
    const int k = i / D4, n = (i % D4) * 4;
    const size_t node = (size_t)r * K + k;
    const float4 fo = *reinterpret_cast<const float4*>(fold + (size_t)sid[k] * D + n);
    const float4 hp = *reinterpret_cast<const float4*>(hproj + (size_t)r * D + n);
    const float4 sl = *reinterpret_cast<const float4*>(slot + (size_t)s * D + n);
    const float4 rk = *reinterpret_cast<const float4*>(rank + (size_t)k * D + n);
    float4 o;
    o.x = fo.x + hp.x + sl.x + rk.x;
    o.y = fo.y + hp.y + sl.y + rk.y;
    o.z = fo.z + hp.z + sl.z + rk.z;
    o.w = fo.w + hp.w + sl.w + rk.w;
    *reinterpret_cast<float4*>(x + node * D + n) = o;
    float4 z = *reinterpret_cast<const float4*>(s_w + LILICORR_N_CONF * D + n);
#pragma unroll
    for (int j = 0; j < LILICORR_N_CONF; ++j) {
      const float4 w = *reinterpret_cast<const float4*>(s_w + j * D + n);
      const float fj = f[k][j];
      z.x = fmaf(w.x, fj, z.x);
      z.y = fmaf(w.y, fj, z.y);
      z.z = fmaf(w.z, fj, z.z);
      z.w = fmaf(w.w, fj, z.w);
    }
    if constexpr (sizeof(TC1) == 2) {          // bf16 operand: tanh-based SiLU, 8-byte store
      uint2 u;
      u.x = bf16_pack2(silu_tanh(z.x), silu_tanh(z.y));
      u.y = bf16_pack2(silu_tanh(z.z), silu_tanh(z.w));
      *reinterpret_cast<uint2*>(c1 + node * D + n) = u;
    } else {
      *reinterpret_cast<float4*>(c1 + node * D + n) =
          make_float4(silu_f(z.x), silu_f(z.y), silu_f(z.z), silu_f(z.w));
    }
  }
}

// ----------------------------------------------------------------------------- RMSNorm
template <typename TY>
__global__ void rmsnorm_kernel(const float* __restrict__ x, int M, int D,
                               const float* __restrict__ gain, TY* __restrict__ y) {
  pdl_wait();
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const float* xr = x + (size_t)row * D;
  float ss = 0.f;
  for (int i = lane; i < D; i += 32) ss += xr[i] * xr[i];
  ss = warp_sum(ss);
  const float r = rsqrtf(ss / (float)D + RMS_EPS);
  for (int i = lane; i < D; i += 32) st_elem(y, (size_t)row * D + i, xr[i] * r * gain[i]);
}

// fin[row] = [xf, xf * t_b] with xf = RMSNorm(x[row]) * gain: the x and x*t blocks of
// the fusion layer's input [x; t; x*t] (App. A); the t block is a per-sequence bias.
template <typename TY>
__global__ void fusion_input_kernel(const float* __restrict__ x, int M, int LK, int D,
                                    const float* __restrict__ gain, const float* __restrict__ t,
                                    TY* __restrict__ fin) {
  pdl_wait();
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const float* xr = x + (size_t)row * D;
  const float* tb = t + (size_t)(row / LK) * D;
  float ss = 0.f;
  for (int i = lane; i < D; i += 32) ss += xr[i] * xr[i];
  ss = warp_sum(ss);
  const float r = rsqrtf(ss / (float)D + RMS_EPS);
  for (int i = lane; i < D; i += 32) {
    const float xf = xr[i] * r * gain[i];
    st_elem(fin, (size_t)row * 2 * D + i, xf);
    st_elem(fin, (size_t)row * 2 * D + D + i, xf * tb[i]);
  }
}

// dst[row] = src[row] / max(||src[row]||, 1e-12), rows of n floats.
__global__ void unit_rows_kernel(const float* __restrict__ src, int rows, int n, int ld_src,
                                 float* __restrict__ dst, int ld_dst) {
  pdl_wait();
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const float* s = src + (size_t)row * ld_src;
  float ss = 0.f;
  for (int i = lane; i < n; i += 32) ss += s[i] * s[i];
  ss = warp_sum(ss);
  const float inv = 1.0f / fmaxf(sqrtf(ss), UNIT_EPS);
  for (int i = lane; i < n; i += 32) dst[(size_t)row * ld_dst + i] = s[i] * inv;
}

// ----------------------------------------------------------------------------- attention
// One CTA per (sequence, head): all L*K nodes attend to all L*K nodes (no mask),
// logits q.k / sqrt(hd) + dist[h, s_j - s_i + L - 1] + same[h] * 1{s_i == s_j}.
// qkv rows hold [q | k | v], each D wide, head h in columns [h*hd, (h+1)*hd).
template <typename TO>
__global__ void attention_kernel(const float* __restrict__ qkv, int L, int K, int D, int n_heads,
                                 int q_per_cta, const float* __restrict__ dist,
                                 const float* __restrict__ same, TO* __restrict__ out) {
  pdl_wait();
  extern __shared__ float sm[];
  const int LK = L * K, hd = D / n_heads;
  const int b = blockIdx.x / n_heads, h = blockIdx.x % n_heads;
  const int q0 = blockIdx.y * q_per_cta, q1 = min(LK, q0 + q_per_cta);
  const int nw = blockDim.x >> 5, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* Ks = sm;                       // [LK][hd + 1]
  float* Vs = Ks + (size_t)LK * (hd + 1);   // [LK][hd]
  float* Qw = Vs + (size_t)LK * hd;     // [nw][hd]
  float* Pw = Qw + (size_t)nw * hd;     // [nw][LK]
  const size_t ld = 3 * (size_t)D;
  const float* base = qkv + (size_t)b * LK * ld;
  const int hv = hd / 4;                       // 16-byte vectors per head row
#pragma unroll 4
  for (int i = threadIdx.x; i < LK * hv; i += blockDim.x) {
    const int j = i / hv, c = (i % hv) * 4;
    const float4 kv = *reinterpret_cast<const float4*>(base + j * ld + D + h * hd + c);
    const float4 vv = *reinterpret_cast<const float4*>(base + j * ld + 2 * D + h * hd + c);
    float* kd = Ks + j * (hd + 1) + c;
    kd[0] = kv.x; kd[1] = kv.y; kd[2] = kv.z; kd[3] = kv.w;
    *reinterpret_cast<float4*>(Vs + j * hd + c) = vv;
  }
  __syncthreads();
  const float scale = rsqrtf((float)hd);
  const float* dh = dist + (size_t)h * (2 * L - 1);
  const float sh = same[h];
  float* q = Qw + warp * hd;
  float* p = Pw + (size_t)warp * LK;
  for (int i = q0 + warp; i < q1; i += nw) {
    for (int c = lane; c < hd; c += 32) q[c] = base[(size_t)i * ld + h * hd + c];
    __syncwarp();
    const int si = i / K;
    float mx = -INFINITY;
    for (int j = lane; j < LK; j += 32) {
      const float* kj = Ks + j * (hd + 1);
      float acc = 0.f;
      for (int c = 0; c < hd; ++c) acc = fmaf(q[c], kj[c], acc);
      const int sj = j / K;
      const float v = acc * scale + dh[sj - si + L - 1] + (si == sj ? sh : 0.f);
      p[j] = v;
      mx = fmaxf(mx, v);
    }
    mx = warp_max(mx);
    float sum = 0.f;
    for (int j = lane; j < LK; j += 32) {
      const float e = __expf(p[j] - mx);
      p[j] = e;
      sum += e;
    }
    sum = warp_sum(sum);
    __syncwarp();
    const float inv = 1.0f / sum;
    for (int c = lane; c < hd; c += 32) {
      float acc = 0.f;
      for (int j = 0; j < LK; ++j) acc = fmaf(p[j], Vs[j * hd + c], acc);
      st_elem(out, ((size_t)b * LK + i) * D + h * hd + c, acc * inv);
    }
    __syncwarp();
  }
}

}  // namespace

size_t attention_smem_bytes(int LK, int hd, int warps) {
  return sizeof(float) * ((size_t)LK * (hd + 1) + (size_t)LK * hd + (size_t)warps * hd +
                          (size_t)warps * LK);
}

bool gemm_rows_supported(const GemmArgs& g) {
  return g.a_dt == LILICORR_F32 && g.M > 0 && g.N > 0 && g.Kd % 8 == 0 && g.lda % 4 == 0 &&
         g.ldw % 8 == 0 && (reinterpret_cast<uintptr_t>(g.A) & 15) == 0 &&
         (reinterpret_cast<uintptr_t>(g.W) & 15) == 0;
}

lilicorr_status_t launch_gemm_rows(const GemmArgs& g, cudaStream_t st) {
  if (!gemm_rows_supported(g)) return LILICORR_ERR_SHAPE;
  const dim3 grid(ceil_div(g.N, GR_N), ceil_div(g.M, GR_M));
  if (g.w_dt == LILICORR_F32) {
    if (g.c_dt == LILICORR_F32) return launch_k(gemm_rows_kernel<float, float>, grid, GR_THREADS, 0, st, g);
    return launch_k(gemm_rows_kernel<float, __nv_bfloat16>, grid, GR_THREADS, 0, st, g);
  }
  if (g.c_dt == LILICORR_F32)
    return launch_k(gemm_rows_kernel<__nv_bfloat16, float>, grid, GR_THREADS, 0, st, g);
  return launch_k(gemm_rows_kernel<__nv_bfloat16, __nv_bfloat16>, grid, GR_THREADS, 0, st, g);
}

lilicorr_status_t launch_gemm_skinny(const GemmArgs& g, cudaStream_t st) {
  if (g.M == 0 || g.N == 0) return LILICORR_OK;
  if ((g.Kd % 8) || (g.lda % 8) || (g.ldw % 8)) return launch_gemm_simt(g, st);
  dim3 grid(ceil_div(g.N, SK_NB), ceil_div(g.M, SK_MB));
  if (g.a_dt == LILICORR_F32) return skinny_dispatch_w<float>(g, grid, st);
  return skinny_dispatch_w<__nv_bfloat16>(g, grid, st);
}

lilicorr_status_t launch_gemm_simt(const GemmArgs& g, cudaStream_t st) {
  if (g.M == 0 || g.N == 0) return LILICORR_OK;
  dim3 grid(ceil_div(g.N, GB_N), ceil_div(g.M, GB_M));
  if (g.a_dt == LILICORR_F32) return gemm_dispatch_w<float>(g, grid, st);
  return gemm_dispatch_w<__nv_bfloat16>(g, grid, st);
}

lilicorr_status_t launch_target_norm(const void* T, lilicorr_dtype_t dt, int B, int n_tgt, int H,
                                     const float* gain, void* tn, lilicorr_dtype_t tn_dt,
                                     cudaStream_t st) {
  if (B == 0) return LILICORR_OK;
  if (dt == LILICORR_F32 && tn_dt == LILICORR_F32)
    LL_TRY(launch_k(target_norm_kernel<float, float>, B, TN_THREADS, 0, st, 
        static_cast<const float*>(T), n_tgt, H, gain, static_cast<float*>(tn)));
  else if (dt == LILICORR_BF16 && tn_dt == LILICORR_F32)
    LL_TRY(launch_k(target_norm_kernel<__nv_bfloat16, float>, B, TN_THREADS, 0, st, 
        static_cast<const __nv_bfloat16*>(T), n_tgt, H, gain, static_cast<float*>(tn)));
  else if (dt == LILICORR_BF16)
    LL_TRY(launch_k(target_norm_kernel<__nv_bfloat16, __nv_bfloat16>, B, TN_THREADS, 0, st, 
        static_cast<const __nv_bfloat16*>(T), n_tgt, H, gain, static_cast<__nv_bfloat16*>(tn)));
  else
    return LILICORR_ERR_DTYPE;
  return LILICORR_OK;
}

lilicorr_status_t launch_node_build(const lilicorr_head* h, int B, const int32_t* ids,
                                    const float* logp, const float* hproj, void* c1,
                                    lilicorr_dtype_t c1_dt, float* x, uint32_t* status,
                                    cudaStream_t st) {
  const lilicorr_head_desc& d = h->desc;
  if (B == 0) return LILICORR_OK;
  const float* fold = static_cast<const float*>(h->fold);
  if (c1_dt == LILICORR_F32)
    LL_TRY(launch_k(node_build_kernel<float>, B * d.L, 256, sizeof(float) * (LILICORR_N_CONF + 1) * d.D, st, d.L, d.K, d.D, d.V, ids, logp, fold, hproj,
                                                      h->slot, h->rank, h->conf1_w, h->conf1_b,
                                                      static_cast<float*>(c1), x, status));
  else
    LL_TRY(launch_k(node_build_kernel<__nv_bfloat16>, B * d.L, 256, sizeof(float) * (LILICORR_N_CONF + 1) * d.D, st, 
        d.L, d.K, d.D, d.V, ids, logp, fold, hproj, h->slot, h->rank, h->conf1_w, h->conf1_b,
        static_cast<__nv_bfloat16*>(c1), x, status));
  return LILICORR_OK;
}

lilicorr_status_t launch_rmsnorm(const float* x, int M, int D, const float* gain, void* y,
                                 lilicorr_dtype_t y_dt, cudaStream_t st) {
  if (M == 0) return LILICORR_OK;
  const int grid = ceil_div(M, 8);
  if (y_dt == LILICORR_F32)
    LL_TRY(launch_k(rmsnorm_kernel<float>, grid, 256, 0, st, x, M, D, gain, static_cast<float*>(y)));
  else
    LL_TRY(launch_k(rmsnorm_kernel<__nv_bfloat16>, grid, 256, 0, st, x, M, D, gain,
                                                        static_cast<__nv_bfloat16*>(y)));
  return LILICORR_OK;
}

lilicorr_status_t launch_fusion_input(const float* x, int B, int LK, int D, const float* gain,
                                      const float* t, void* fin, lilicorr_dtype_t dt,
                                      cudaStream_t st) {
  const int M = B * LK;
  if (M == 0) return LILICORR_OK;
  const int grid = ceil_div(M, 8);
  if (dt == LILICORR_F32)
    LL_TRY(launch_k(fusion_input_kernel<float>, grid, 256, 0, st, x, M, LK, D, gain, t, static_cast<float*>(fin)));
  else
    LL_TRY(launch_k(fusion_input_kernel<__nv_bfloat16>, grid, 256, 0, st, x, M, LK, D, gain, t,
                                                             static_cast<__nv_bfloat16*>(fin)));
  return LILICORR_OK;
}

lilicorr_status_t launch_unit_rows(const float* src, int rows, int n, int ld_src, float* dst,
                                   int ld_dst, cudaStream_t st) {
  if (rows == 0) return LILICORR_OK;
  LL_TRY(launch_k(unit_rows_kernel, ceil_div(rows, 8), 256, 0, st, src, rows, n, ld_src, dst, ld_dst));
  return LILICORR_OK;
}

lilicorr_status_t launch_attention(const float* qkv, int B, int L, int K, int D, int n_heads,
                                   const float* dist, const float* same, void* out,
                                   lilicorr_dtype_t out_dt, cudaStream_t st) {
  if (B == 0) return LILICORR_OK;
  const int warps = 8;
  const int LK = L * K;
  const size_t smem = attention_smem_bytes(LK, D / n_heads, warps);
  static bool cfg_f32[64] = {false}, cfg_bf16[64] = {false};
  LL_TRY(allow_max_dynamic_smem(attention_kernel<float>, cfg_f32));
  LL_TRY(allow_max_dynamic_smem(attention_kernel<__nv_bfloat16>, cfg_bf16));
  // split the queries of a (sequence, head) over CTAs until the grid covers the GPU
  int qblocks = ceil_div(2 * num_sms(), B * n_heads);
  qblocks = max(1, min(qblocks, ceil_div(LK, 2 * warps)));
  const int q_per_cta = ceil_div(LK, qblocks);
  qblocks = ceil_div(LK, q_per_cta);
  dim3 grid(B * n_heads, qblocks);
  if (out_dt == LILICORR_F32)
    LL_TRY(launch_k(attention_kernel<float>, grid, warps * 32, smem, st, qkv, L, K, D, n_heads, q_per_cta, dist,
                                                            same, static_cast<float*>(out)));
  else
    LL_TRY(launch_k(attention_kernel<__nv_bfloat16>, grid, warps * 32, smem, st, 
        qkv, L, K, D, n_heads, q_per_cta, dist, same, static_cast<__nv_bfloat16*>(out)));
  return LILICORR_OK;
}

}  // namespace lilicorr
