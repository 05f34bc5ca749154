// Tensor-core linear layer for one tile of rows: C[M, N] = epilogue(A W^T) with M <= 128,
// bf16 A and W, Kd <= 512 (a multiple of 64) — the node-level products of one sequence.
//
// At these sizes a product is a few MFLOP and its time is latency: launch, TMA round
// trips, the accumulator drain. One SM completes about one TMA copy per 0.3 us almost
// independently of its size up to 64 KB, so this kernel moves everything a CTA needs in
// three copies: all of A [128 x Kd] and all of its BN weight rows [BN x Kd] as 3-D boxes
// (64-wide K chunks, 128-byte swizzle), and the residual tile. One CTA per BN output
// columns; one lane issues Kd / 16 tcgen05.mma (M = 128, N = BN) into tensor memory; four
// epilogue warps drain it with tcgen05.ld, add bias / per-sequence bias / SiLU / the
// residual, stage 128-byte-swizzled chunks in the A buffer (free once the products are
// done) and store them with TMA. Every mbarrier wait is bounded (about 2 s).
#include "tc_ptx.cuh"

namespace lilicorr {

namespace {
using namespace tc;

constexpr int SG_THREADS = 192;            // loader, MMA, 4 epilogue warps
constexpr int SG_EPI = 128;
constexpr uint32_t SG_CHUNK = 128 * 128;   // 128 rows x 128 bytes
constexpr long long SG_WAIT = 4000000000ll;

struct SmallEpilogue {
  const float* bias;
  const float* bias_rows; int rows_per_bias;
  int act;
};

__device__ __forceinline__ void sg_bar() { asm volatile("bar.sync 1, %0;" ::"n"(SG_EPI) : "memory"); }

template <int BN, bool OUT_BF16, bool RES>
__global__ void __launch_bounds__(SG_THREADS, 1)
    gemm_small_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapW,
                      const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapR,
                      SmallEpilogue ep, int M, int N, int Kd, uint32_t* status) {
  constexpr int CH = OUT_BF16 ? 64 : 32;   // output columns per 128-byte staging chunk
  constexpr int NCH = BN / CH;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int nk = Kd / 64;
  uint8_t* sA = smem;                                    // nk chunks of 128 x 64 bf16 (and
                                                         // later the NCH staging chunks)
  uint8_t* sB = sA + (size_t)(nk > NCH ? nk : NCH) * SG_CHUNK;   // nk chunks of BN x 64 bf16
  uint8_t* sR = sB + (size_t)nk * BN * 128;              // BN / 32 chunks of 128 x 32 fp32
  __shared__ __align__(8) uint64_t full, acc_full;
  __shared__ uint32_t tmem_base;
  __shared__ volatile int abort_flag;
  __shared__ __align__(16) float s_bias[BN];      // read as float4

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN;
  if (threadIdx.x == 0) {
    mbar_init(&full, 1);
    mbar_init(&acc_full, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(&tmem_base, BN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  pdl_wait();                       // every operand may come from the preceding launch
  if (warp == 0 && lane == 0) {
    const uint32_t bytes = (uint32_t)nk * (SG_CHUNK + BN * 128) + (RES ? BN * 512u : 0u);
    mbar_expect_tx(&full, bytes);
    tma_load_3d(sB, &mapW, &full, 0, n0, 0);
    tma_load_3d(sA, &mapA, &full, 0, 0, 0);
    if (RES)
      for (int j = 0; j < BN / 32; ++j)
        tma_load_2d(sR + (size_t)j * SG_CHUNK, &mapR, &full, n0 + 32 * j, 0);
  }

  if (warp == 1) {
    if (lane == 0) {
      if (!mbar_wait(&full, 0, SG_WAIT)) abort_flag = 1;
      tc_fence_after();
      if (!abort_flag) {
        constexpr uint32_t idesc = instr_desc(128, BN);
        for (int kc = 0; kc < nk; ++kc) {
          const uint64_t ad = smem_desc(sA + (size_t)kc * SG_CHUNK);
          const uint64_t bd = smem_desc(sB + (size_t)kc * BN * 128);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_bf16(tmem, ad + 2ull * k, bd + 2ull * k, idesc, (kc > 0 || k > 0) ? 1u : 0u);
        }
        mma_commit(&acc_full);
      }
    }
  } else if (warp >= 2) {
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const bool leader = (warp == 2 && lane == 0);
    for (int j = threadIdx.x - 64; j < BN; j += SG_EPI)
      s_bias[j] = (ep.bias && n0 + j < N) ? ep.bias[n0 + j] : 0.f;
    if (!abort_flag && !mbar_wait(&acc_full, 0, SG_WAIT)) abort_flag = 1;
    tc_fence_after();
    sg_bar();
    const float* brow = (ep.bias_rows && row < M) ? ep.bias_rows + (size_t)(row / ep.rows_per_bias) * N
                                                  : nullptr;
#pragma unroll 1
    for (int c = 0; c < NCH; ++c) {
      float v[CH];
#pragma unroll
      for (int h = 0; h < CH / 32; ++h) {
        uint32_t r[32];
        tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + c * CH + h * 32, r);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[h * 32 + j] = __uint_as_float(r[j]);
      }
#pragma unroll
      for (int j = 0; j < CH; j += 4) {
        float4 x = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
        const float4 bb = *reinterpret_cast<const float4*>(s_bias + c * CH + j);
        x.x += bb.x; x.y += bb.y; x.z += bb.z; x.w += bb.w;
        if (brow && n0 + c * CH + j < N) {
          const float4 br = *reinterpret_cast<const float4*>(brow + n0 + c * CH + j);
          x.x += br.x; x.y += br.y; x.z += br.z; x.w += br.w;
        }
        if (ep.act == ACT_SILU) {
          if (OUT_BF16) {
            x.x = silu_tanh(x.x); x.y = silu_tanh(x.y); x.z = silu_tanh(x.z); x.w = silu_tanh(x.w);
          } else {
            x.x = silu_f(x.x); x.y = silu_f(x.y); x.z = silu_f(x.z); x.w = silu_f(x.w);
          }
        }
        if (RES) {                                   // fp32 output: 4 columns = 16 bytes
          const int col = c * CH + j;
          const float4 rr = *reinterpret_cast<const float4*>(
              sR + (size_t)(col >> 5) * SG_CHUNK + swz(row, (col & 31) >> 2));
          x.x += rr.x; x.y += rr.y; x.z += rr.z; x.w += rr.w;
        }
        v[j] = x.x; v[j + 1] = x.y; v[j + 2] = x.z; v[j + 3] = x.w;
      }
      uint8_t* stg = sA + (size_t)c * SG_CHUNK;      // the products are done: A is free
      if (OUT_BF16) {
#pragma unroll
        for (int p = 0; p < 8; ++p) {
          uint4 w;
          w.x = pack_bf16x2(v[8 * p + 0], v[8 * p + 1]);
          w.y = pack_bf16x2(v[8 * p + 2], v[8 * p + 3]);
          w.z = pack_bf16x2(v[8 * p + 4], v[8 * p + 5]);
          w.w = pack_bf16x2(v[8 * p + 6], v[8 * p + 7]);
          *reinterpret_cast<uint4*>(stg + swz(row, p)) = w;
        }
      } else {
#pragma unroll
        for (int p = 0; p < 8; ++p)
          *reinterpret_cast<float4*>(stg + swz(row, p)) =
              make_float4(v[4 * p], v[4 * p + 1], v[4 * p + 2], v[4 * p + 3]);
      }
    }
    fence_async_shared();
    sg_bar();
    if (leader && !abort_flag) {
      for (int c = 0; c < NCH; ++c)
        if (n0 + c * CH < N) tma_store_2d(&mapC, sA + (size_t)c * SG_CHUNK, n0 + c * CH, 0);
      tma_store_wait_all();
    }
  }

  tc_fence_before();
  __syncthreads();
  if (abort_flag) {
    if (threadIdx.x == 0) {
      set_status(status, LILICORR_ERR_TIMEOUT);
      const long long t0 = clock64();                // let copies in flight land
      while (clock64() - t0 < SG_WAIT / 10) {
      }
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, BN);
  }
}

// 3-D view (64, rows, cols / 64) of a row-major bf16 matrix with row stride ld elements:
// box (64, box_rows, cols / 64) is every K chunk of box_rows rows, 128-byte swizzled.
bool kchunk_map(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows) {
  const uint64_t dims[3] = {64, (uint64_t)rows, (uint64_t)(cols / 64)};
  const uint64_t strides[3] = {2, (uint64_t)ld * 2, 128};
  const uint32_t box[3] = {64, (uint32_t)box_rows, (uint32_t)(cols / 64)};
  return make_map_nd(m, base, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, dims, strides, box);
}

template <int BN, bool OUT_BF16>
size_t small_smem(int Kd, bool res) {
  constexpr int NCH = BN / (OUT_BF16 ? 64 : 32);
  const int nk = Kd / 64;
  return 1024 + (size_t)(nk > NCH ? nk : NCH) * SG_CHUNK + (size_t)nk * BN * 128 +
         (res ? (size_t)BN * 512 : 0);
}

template <int BN, bool OUT_BF16, bool RES>
lilicorr_status_t launch_small(const GemmArgs& g, cudaStream_t st) {
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(gemm_small_kernel<BN, OUT_BF16, RES>, configured));
  CUtensorMap ma, mw, mc, mr;
  const CUtensorMapDataType bf = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const CUtensorMapDataType f32 = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
  constexpr int CH = OUT_BF16 ? 64 : 32;
  if (!kchunk_map(&ma, g.A, g.M, g.Kd, g.lda, 128)) return LILICORR_ERR_CUDA;
  if (!kchunk_map(&mw, g.W, g.N, g.Kd, g.ldw, BN)) return LILICORR_ERR_CUDA;
  if (!make_map(&mc, g.C, OUT_BF16 ? bf : f32, OUT_BF16 ? 2 : 4, g.M, g.N, g.ldc, 128, CH))
    return LILICORR_ERR_CUDA;
  if (RES) {
    if (!make_map(&mr, g.residual, f32, 4, g.M, g.N, g.ldr, 128, 32)) return LILICORR_ERR_CUDA;
  } else {
    mr = mc;                                   // never read
  }
  SmallEpilogue ep;
  ep.bias = g.bias;
  ep.bias_rows = g.bias_rows;
  ep.rows_per_bias = g.rows_per_bias;
  ep.act = g.act;
  LL_TRY(launch_k(gemm_small_kernel<BN, OUT_BF16, RES>, ceil_div(g.N, BN), SG_THREADS,
                  small_smem<BN, OUT_BF16>(g.Kd, RES), st, ma, mw, mc, mr, ep, g.M, g.N, g.Kd,
                  g.status));
  return LILICORR_OK;
}

template <int BN>
lilicorr_status_t launch_small_f32(const GemmArgs& g, cudaStream_t st) {
  return g.residual ? launch_small<BN, false, true>(g, st) : launch_small<BN, false, false>(g, st);
}

}  // namespace

bool gemm_small_supported(const GemmArgs& g) {
  if (!gemm_tc_supported(g)) return false;
  if (g.M > 128 || g.Kd % 64 || g.Kd > 512) return false;
  if (g.c_dt == LILICORR_BF16 && g.N % 64) return false;    // whole 64-column bf16 chunks
  if (g.c_dt == LILICORR_F32 && g.N % 32) return false;
  return small_smem<64, false>(g.Kd, g.residual != nullptr) <= SMEM_PER_BLOCK_MAX;
}

lilicorr_status_t launch_gemm_small(const GemmArgs& g, cudaStream_t st) {
  if (g.M == 0 || g.N == 0) return LILICORR_OK;
  // 64 output columns per CTA, or 32 when that still leaves few CTAs (more CTAs, each
  // moving its copies in parallel); bf16 outputs stage 64-column chunks
  if (g.c_dt == LILICORR_BF16) return launch_small<64, true, false>(g, st);
  return g.N <= 512 ? launch_small_f32<32>(g, st) : launch_small_f32<64>(g, st);
}

}  // namespace lilicorr
