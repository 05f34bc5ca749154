// Tensor-core linear layer of the bf16 head (5th-generation tensor cores, sm_103a).
//
// C[M, N] = epilogue(A[M, Kd] W[N, Kd]^T) with bf16 A (activations) and W (weights),
// fp32 accumulation in tensor memory. One CTA computes a 128 x BN tile:
//   * warp 0 lane 0 streams 128 x 64 tiles of A and BN x 64 tiles of W into a ring
//     of shared-memory stages with 2-D TMA copies (128-byte swizzle), each stage
//     guarded by a "full" mbarrier (transaction bytes) and an "empty" mbarrier;
//   * warp 1 allocates BN columns of tensor memory, and its lane 0 issues
//     tcgen05.mma (M = 128, N = BN, K = 16) four times per stage, releasing the
//     stage with tcgen05.commit;
//   * all four warps then read the accumulator back with tcgen05.ld (warp w owns
//     rows 32w..32w+31) and apply bias / per-sequence bias / SiLU / residual before
//     storing fp32 or bf16.
// Every wait is bounded (about 2 s); on timeout the CTA records LILICORR_ERR_TIMEOUT in
// the status word, waits (bounded) for its copies in flight, frees its tensor
// memory and exits.
#include <cuda.h>

#include "internal.cuh"

namespace lilicorr {

namespace {

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;                  // 64 bf16 = 128 bytes: one swizzle atom row
constexpr int TC_THREADS = 128;
constexpr long long WAIT_LIMIT_CYCLES = 4000000000ll;   // about 2 s at the SM clock

struct TcEpilogue {
  void* C; int ldc; int c_bf16;
  const float* bias;
  const float* bias_rows; int rows_per_bias;
  const float* residual; int ldr;
  int act;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for the phase of parity `parity` to complete; false after `limit` SM cycles
// (the bound is read from the SM's own cycle counter, which is cheap to poll).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > limit) return false;
  return true;
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row groups
// 1024 bytes apart; start address advanced by 32 bytes per K step of 16 elements.
__device__ __forceinline__ uint64_t smem_desc(const void* tile) {
  const uint64_t addr = smem_u32(tile);
  return ((addr & 0x3FFFFull) >> 4)          // start address
         | (1ull << 16)                      // leading byte offset (unused for this layout)
         | ((1024ull >> 4) << 32)            // stride byte offset: 8 rows x 128 B
         | (1ull << 46)                      // descriptor version
         | (2ull << 61);                     // 128-byte swizzle
}
// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both K-major.
__host__ __device__ constexpr uint32_t instr_desc(int m, int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(m >> 4) << 24);
}
__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate));
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32"
      " {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15,"
      " %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

template <int BN>
struct TcCfg {
  static constexpr int STAGES = BN >= 256 ? 3 : 4;
  static constexpr uint32_t A_BYTES = TC_BM * TC_BK * 2;
  static constexpr uint32_t B_BYTES = BN * TC_BK * 2;
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * (A_BYTES + B_BYTES);
  static constexpr uint32_t TMEM_COLS = BN < 32 ? 32 : BN;
};

template <int BN>
__global__ void __launch_bounds__(TC_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap mapA,
                   const __grid_constant__ CUtensorMap mapW, TcEpilogue ep, int M, int N, int Kd,
                   uint32_t* status) {
  using Cfg = TcCfg<BN>;
  constexpr int S = Cfg::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + S * Cfg::A_BYTES;
  __shared__ __align__(8) uint64_t full[S], empty[S], done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.y * TC_BM, n0 = blockIdx.x * BN;
  const int nk = (Kd + TC_BK - 1) / TC_BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&done, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tmem_base)),
                 "r"(Cfg::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 0 && lane == 0) {
    // ---- producer: TMA into the stage ring
    for (int i = 0; i < nk; ++i) {
      const int s = i % S;
      const uint32_t ph = (uint32_t)(i / S) & 1u;
      if (!mbar_wait(&empty[s], ph ^ 1u, WAIT_LIMIT_CYCLES)) {
        atomicExch(&abort_flag, 1);
        break;
      }
      mbar_expect_tx(&full[s], Cfg::A_BYTES + Cfg::B_BYTES);
      tma_load_2d(sA + (size_t)s * Cfg::A_BYTES, &mapA, &full[s], i * TC_BK, m0);
      tma_load_2d(sB + (size_t)s * Cfg::B_BYTES, &mapW, &full[s], i * TC_BK, n0);
    }
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer
    constexpr uint32_t idesc = instr_desc(TC_BM, BN);
    for (int i = 0; i < nk; ++i) {
      const int s = i % S;
      const uint32_t ph = (uint32_t)(i / S) & 1u;
      if (!mbar_wait(&full[s], ph, WAIT_LIMIT_CYCLES)) {
        atomicExch(&abort_flag, 1);
        break;
      }
      tc_fence_after();
      const uint64_t ad = smem_desc(sA + (size_t)s * Cfg::A_BYTES);
      const uint64_t bd = smem_desc(sB + (size_t)s * Cfg::B_BYTES);
#pragma unroll
      for (int k = 0; k < TC_BK / 16; ++k)
        mma_bf16(tmem, ad + 2ull * k, bd + 2ull * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
      mma_commit(&empty[s]);
    }
    mma_commit(&done);
  }
  __syncwarp();

  // ---- epilogue: TMEM -> registers -> shared (transpose) -> global, row segments.
  // Lane l of warp w owns column (c0 + l) of rows 32w..32w+31 of each 32-column chunk;
  // the chunk's residual values are loaded before they are needed, all 32 in flight
  // (the first chunk's while the tensor cores are still busy).
  const int mrow0 = m0 + warp * 32;
  float res[32];
  auto load_residual = [&](int c0) {
    const int n = n0 + c0 + lane;
#pragma unroll
    for (int rr = 0; rr < 32; ++rr)
      res[rr] = (ep.residual && n < N && mrow0 + rr < M)
                    ? ep.residual[(size_t)(mrow0 + rr) * ep.ldr + n] : 0.f;
  };
  load_residual(0);
  if (!mbar_wait(&done, 0, WAIT_LIMIT_CYCLES)) atomicExch(&abort_flag, 1);
  tc_fence_after();
  __syncthreads();                         // the stage ring is drained: reuse it below
  if (!abort_flag) {
    float* tile = reinterpret_cast<float*>(smem) + warp * 32 * 33;   // this warp's 32 x 32
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 32) {
      uint32_t r[32];
      tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, r);
#pragma unroll
      for (int j = 0; j < 32; ++j) tile[lane * 33 + j] = __uint_as_float(r[j]);
      __syncwarp();
      const int n = n0 + c0 + lane;
      if (n < N) {
        const float bn = ep.bias ? ep.bias[n] : 0.f;
#pragma unroll
        for (int rr = 0; rr < 32; ++rr) {
          const int m = mrow0 + rr;
          if (m < M) {
            float v = tile[rr * 33 + lane] + bn;
            if (ep.bias_rows) v += ep.bias_rows[(size_t)(m / ep.rows_per_bias) * N + n];
            if (ep.act == ACT_SILU) v = silu_f(v);
            v += res[rr];
            if (ep.c_bf16)
              static_cast<__nv_bfloat16*>(ep.C)[(size_t)m * ep.ldc + n] = __float2bfloat16_rn(v);
            else
              static_cast<float*>(ep.C)[(size_t)m * ep.ldc + n] = v;
          }
        }
      }
      if (c0 + 32 < BN) load_residual(c0 + 32);
      __syncwarp();
    }
  }

  // ---- teardown
  tc_fence_before();
  __syncthreads();
  if (abort_flag) {
    if (threadIdx.x == 0) {
      set_status(status, LILICORR_ERR_TIMEOUT);
      // let copies still in flight land before the shared memory is released
      for (int s = 0; s < S && s < nk; ++s) {
        const int last = ((nk - 1 - s) / S) * S + s;
        mbar_wait(&full[s], (uint32_t)(last / S) & 1u, WAIT_LIMIT_CYCLES / 10);
      }
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(Cfg::TMEM_COLS)
                 : "memory");
  }
}

// ----------------------------------------------------------------------------- host side
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D bf16 tensor map over rows x cols (row stride ld elements), box box_rows x 64.
bool make_map(CUtensorMap* map, const void* base, int rows, int cols, int ld, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {(cuuint32_t)TC_BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN>
lilicorr_status_t launch_bn(const GemmArgs& g, uint32_t* status, cudaStream_t st) {
  using Cfg = TcCfg<BN>;
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(gemm_tc_kernel<BN>, configured));
  CUtensorMap ma, mw;
  if (!make_map(&ma, g.A, g.M, g.Kd, g.lda, TC_BM)) return LILICORR_ERR_CUDA;
  if (!make_map(&mw, g.W, g.N, g.Kd, g.ldw, BN)) return LILICORR_ERR_CUDA;
  TcEpilogue ep;
  ep.C = g.C; ep.ldc = g.ldc; ep.c_bf16 = g.c_dt == LILICORR_BF16;
  ep.bias = g.bias; ep.bias_rows = g.bias_rows; ep.rows_per_bias = g.rows_per_bias;
  ep.residual = g.residual; ep.ldr = g.ldr; ep.act = g.act;
  dim3 grid(ceil_div(g.N, BN), ceil_div(g.M, TC_BM));
  gemm_tc_kernel<BN><<<grid, TC_THREADS, Cfg::SMEM, st>>>(ma, mw, ep, g.M, g.N, g.Kd, status);
  return last_launch();
}

}  // namespace

bool gemm_tc_supported(const GemmArgs& g) {
  if (g.a_dt != LILICORR_BF16 || g.w_dt != LILICORR_BF16) return false;
  if (g.M <= 0 || g.N <= 0 || g.Kd <= 0) return false;
  // TMA: 16-byte aligned bases and row strides
  if (!aligned16(g.A) || !aligned16(g.W) || (g.lda % 8) || (g.ldw % 8) || (g.Kd % 8)) return false;
  return encode_fn() != nullptr;
}

lilicorr_status_t launch_gemm_tc(const GemmArgs& g, cudaStream_t st) {
  // column tile: the widest of 256/128/64 that still gives the grid a few waves of CTAs
  const int mt = ceil_div(g.M, TC_BM);
  const int sms = num_sms();
  if (g.N >= 256 && mt * ceil_div(g.N, 256) >= sms) return launch_bn<256>(g, g.status, st);
  if (g.N >= 128 && mt * ceil_div(g.N, 128) >= sms / 2) return launch_bn<128>(g, g.status, st);
  return launch_bn<64>(g, g.status, st);
}

}  // namespace lilicorr
