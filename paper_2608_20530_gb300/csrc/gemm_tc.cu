// Tensor-core linear layer of the bf16 head (5th-generation tensor cores, sm_103a).
//
// C[M, N] = epilogue(A[M, Kd] W[N, Kd]^T) with bf16 A (activations) and W (weights),
// fp32 accumulation in tensor memory. A persistent, warp-specialised kernel: one CTA
// per SM walks output tiles of 128 x BN.
//   * warp 0 (one lane) streams 128 x 64 tiles of A and BN x 64 tiles of W into a ring
//     of shared-memory stages with 2-D TMA copies (128-byte swizzle); each stage has a
//     "full" mbarrier (transaction bytes) and an "empty" mbarrier;
//   * warp 1 allocates two accumulators of BN tensor-memory columns and its lane 0
//     issues tcgen05.mma (M = 128, N = BN, K = 16), four per stage, releasing stages
//     with tcgen05.commit and handing finished accumulators to the epilogue;
//   * warps 2-9 drain an accumulator with tcgen05.ld while the next tile's products
//     run on the other one: two warps per tensor-memory lane quarter, each taking half
//     of every chunk's columns. Per chunk of 128 rows x 128 bytes they add bias /
//     per-sequence bias / SiLU / the residual (brought in by a TMA load), write the
//     chunk into a 128-byte-swizzled staging buffer and store it with one TMA bulk
//     tensor store (double-buffered staging and residual buffers).
// Every mbarrier wait is bounded (about 2 s of SM cycles, or a shorter limit a test hook
// sets); on timeout the kernel records LILICORR_ERR_TIMEOUT in the status word, stops
// issuing work while keeping every thread on its barriers, lets copies in flight land,
// frees its tensor memory, returns.
#include "tc_ptx.cuh"

namespace lilicorr {

namespace {
using namespace tc;

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;                  // 64 bf16 = 128 bytes: one swizzle atom row
constexpr int TC_THREADS = 320;            // producer, MMA, 8 epilogue warps
constexpr int EPI_THREADS = 256;
constexpr uint32_t CHUNK_BYTES = 128 * 128;   // staging chunk: 128 rows x 128 bytes
constexpr long long WAIT_LIMIT_CYCLES = 4000000000ll;   // about 2 s at the SM clock
constexpr float TC_RMS_EPS = 1e-6f;                    // the network's RMSNorm epsilon

__device__ __forceinline__ void epi_bar() {   // the 8 epilogue warps only
  asm volatile("bar.sync 1, %0;" ::"n"(EPI_THREADS) : "memory");
}
// tcgen05.ld of 16 columns (lane = row of the calling warp's quarter), with the wait
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32"
      " {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}


struct TcEpilogue {
  const float* bias;
  const float* bias_rows; int rows_per_bias;
  int has_residual;
  int act;
  // RMSNorm of the output rows folded into the next product (fp32 outputs): the output
  // times `c2_gain` per column, rounded to bf16, into c2 [M, ldc2], and each thread's sum of
  // squares of its part of the row into ss_out[m * SS_LD + 2 * column tile + half]
  __nv_bfloat16* c2; int ldc2; const float* c2_gain; float* ss_out;
  // ...and optionally a second copy times a per-sequence row vector: c3 [M, ldc2] receives
  // bf16(output * c2_gain * c3_t[m / c3_rows_per]) (c3_t [*, N])
  __nv_bfloat16* c3; const float* c3_t; int c3_rows_per;
  int no_c;              // folded producer whose output C nobody reads: only c2 / c3 written
  // ...and its use: the accumulator scaled by rsqrt(sum of ss_in[m * SS_LD + 0..ss_slots) *
  // ss_scale + eps) before the bias
  const float* ss_in; int ss_slots; float ss_scale;
};

template <int BN, bool OUT_BF16>
struct TcCfg {
  static constexpr int STAGES = BN >= 256 ? 3 : 4;
  static constexpr uint32_t A_BYTES = TC_BM * TC_BK * 2;
  static constexpr uint32_t B_BYTES = BN * TC_BK * 2;
  static constexpr int CH = OUT_BF16 ? 64 : 32;        // output columns per 128-byte chunk
  static constexpr int NCH = BN / CH;
  static constexpr uint32_t TMEM_COLS = 2 * BN;         // two accumulators
  static constexpr size_t RING = (size_t)STAGES * (A_BYTES + B_BYTES);
  static constexpr size_t SMEM = 1024 + RING + 4 * (size_t)CHUNK_BYTES + 3 * BN * sizeof(float);
};

// FOLD: the instantiation with the folded-RMSNorm epilogue (c2 / ss_out, ss_in); the
// others leave that code out and keep their registers.
template <int BN, bool OUT_BF16, bool FOLD>
__global__ void __launch_bounds__(TC_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap mapA,
                   const __grid_constant__ CUtensorMap mapW,
                   const __grid_constant__ CUtensorMap mapC,
                   const __grid_constant__ CUtensorMap mapR, TcEpilogue ep, int M, int N, int Kd,
                   uint32_t* status, long long wait_limit, int starve) {
  using Cfg = TcCfg<BN, OUT_BF16>;
  constexpr int S = Cfg::STAGES, CH = Cfg::CH, NCH = Cfg::NCH;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + S * Cfg::A_BYTES;
  uint8_t* s_out = smem + Cfg::RING;                   // 2 staging chunks
  uint8_t* s_res = s_out + 2 * CHUNK_BYTES;            // 2 residual chunks
  float* s_bias = reinterpret_cast<float*>(s_res + 2 * CHUNK_BYTES);
  float* s_gain = s_bias + BN;                         // c2_gain of the tile's columns
  float* s_t = s_gain + BN;                            // c3_t of the tile's sequence
  __shared__ __align__(8) uint64_t full[S], empty[S], acc_full[2], acc_empty[2], res_full[2];
  __shared__ uint32_t tmem_base;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles_n = (N + BN - 1) / BN;
  const int tiles = ((M + TC_BM - 1) / TC_BM) * tiles_n;
  const int nk = (Kd + TC_BK - 1) / TC_BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], EPI_THREADS / 32);
      mbar_init(&res_full[b], 1);
    }
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
  pdl_wait();                      // inputs come from the preceding launch

  if (warp == 0) {
    // ---- producer: TMA into the stage ring, tile after tile (none at all under the
    //      test hook that starves the consumers to exercise their bounded waits)
    if (lane == 0 && !starve) {
      uint32_t g = 0;                            // k-blocks issued so far
      for (int t = blockIdx.x; t < tiles && !abort_flag; t += gridDim.x) {
        const int m0 = (t / tiles_n) * TC_BM, n0 = (t % tiles_n) * BN;
        for (int i = 0; i < nk; ++i, ++g) {
          const int s = (int)(g % S);
          const uint32_t ph = (g / S) & 1u;
          if (!mbar_wait(&empty[s], ph ^ 1u, wait_limit)) {
            abort_flag = 1;
            break;
          }
          mbar_expect_tx(&full[s], Cfg::A_BYTES + Cfg::B_BYTES);
          tma_load_2d(sA + (size_t)s * Cfg::A_BYTES, &mapA, &full[s], i * TC_BK, m0);
          tma_load_2d(sB + (size_t)s * Cfg::B_BYTES, &mapW, &full[s], i * TC_BK, n0);
        }
      }
    }
  } else if (warp == 1) {
    // ---- MMA issuer: one accumulator per tile, alternating
    if (lane == 0) {
      constexpr uint32_t idesc = instr_desc(TC_BM, BN);
      uint32_t g = 0, lt = 0;
      for (int t = blockIdx.x; t < tiles && !abort_flag; t += gridDim.x, ++lt) {
        const uint32_t acc = lt & 1u, aph = (lt >> 1) & 1u;
        if (!mbar_wait(&acc_empty[acc], aph ^ 1u, wait_limit)) {
          abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + acc * BN;
        for (int i = 0; i < nk; ++i, ++g) {
          const int s = (int)(g % S);
          const uint32_t ph = (g / S) & 1u;
          if (!mbar_wait(&full[s], ph, wait_limit)) {
            abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc(sA + (size_t)s * Cfg::A_BYTES);
          const uint64_t bd = smem_desc(sB + (size_t)s * Cfg::B_BYTES);
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)
            mma_bf16(d, ad + 2ull * k, bd + 2ull * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
          mma_commit(&empty[s]);
        }
        mma_commit(&acc_full[acc]);
      }
    }
  } else {
    // ---- epilogue warps 2..9: warp w reads tensor-memory lanes 32*(w%4)..+31 and takes
    //      columns HC*half .. HC*half + HC - 1 of every chunk
    constexpr int HC = CH / 2;
    const int q = warp & 3;
    const int half = (warp - 2) >> 2;
    const int row = q * 32 + lane;               // row inside the tile
    const bool leader = (warp == 2 && lane == 0);
    uint32_t cc = 0, lt = 0;                     // chunks and tiles handled so far
    // residual chunks come in by TMA, one chunk ahead
    auto issue_res = [&](int t, int c, uint32_t k) {
      const int m0 = (t / tiles_n) * TC_BM, n0 = (t % tiles_n) * BN;
      uint64_t* bar = &res_full[k & 1u];
      mbar_expect_tx(bar, CHUNK_BYTES);
      tma_load_2d(s_res + (k & 1u) * CHUNK_BYTES, &mapR, bar, n0 + c * CH, m0);
    };
    if (ep.has_residual && leader && (int)blockIdx.x < tiles) issue_res(blockIdx.x, 0, 0);
    // folded RMSNorm of the input rows: the row's sums of squares, loaded a tile ahead
    float4 ssn[SS_LD / 4];
    auto load_ss = [&](int t) {
      const int mm = (t / tiles_n) * TC_BM + row;
      const float4* src = reinterpret_cast<const float4*>(ep.ss_in + (size_t)mm * SS_LD);
#pragma unroll
      for (int i = 0; i < SS_LD / 4; ++i)
        ssn[i] = (t < tiles && mm < M && 4 * i < ep.ss_slots) ? src[i]
                                                              : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    if (FOLD && ep.ss_in) load_ss(blockIdx.x);
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++lt) {
      const int m0 = (t / tiles_n) * TC_BM, n0 = (t % tiles_n) * BN;
      const uint32_t acc = lt & 1u;
      epi_bar();                                  // s_bias free again
      // c3: when the tile's rows all belong to one sequence, its c3_t row goes to shared
      // memory with the gains; otherwise every thread reads its own row's
      const int tb0 = (FOLD && ep.c3) ? min(m0, M - 1) / ep.c3_rows_per : 0;
      const bool t_shared = (FOLD && ep.c3) && min(m0 + TC_BM - 1, M - 1) / ep.c3_rows_per == tb0;
      for (int j = threadIdx.x - 64; j < BN; j += EPI_THREADS) {
        s_bias[j] = (ep.bias && n0 + j < N) ? ep.bias[n0 + j] : 0.f;
        if (FOLD && !OUT_BF16 && ep.c2) s_gain[j] = n0 + j < N ? ep.c2_gain[n0 + j] : 0.f;
        if (t_shared) s_t[j] = n0 + j < N ? ep.c3_t[(size_t)tb0 * N + n0 + j] : 0.f;
      }
      if (!abort_flag && !mbar_wait(&acc_full[acc], (lt >> 1) & 1u, wait_limit))
        abort_flag = 1;
      tc_fence_after();
      epi_bar();
      const int m = m0 + row;
      const float* brow = (ep.bias_rows && m < M)
                              ? ep.bias_rows + (size_t)(m / ep.rows_per_bias) * N : nullptr;
      float rs = 1.f;                             // folded RMSNorm of the input rows
      if (FOLD && ep.ss_in) {
        float sum = 0.f;                          // slots past ss_slots hold zeros
#pragma unroll
        for (int i = 0; i < SS_LD / 4; ++i) sum += (ssn[i].x + ssn[i].y) + (ssn[i].z + ssn[i].w);
        rs = rsqrtf(sum * ep.ss_scale + TC_RMS_EPS);
        load_ss(t + gridDim.x);
      }
      float ssq = 0.f;                            // this thread's squares of the output row
#pragma unroll 1
      for (int c = 0; c < NCH; ++c, ++cc) {
        const uint32_t b = cc & 1u;
        // prefetch the next chunk's residual (its buffer was drained a chunk ago)
        if (ep.has_residual && leader && !abort_flag) {
          if (c + 1 < NCH) issue_res(t, c + 1, cc + 1);
          else if (t + (int)gridDim.x < tiles) issue_res(t + gridDim.x, 0, cc + 1);
        }
        const int cl = c * CH + half * HC;         // first column of this thread's part
        float v[HC];
        {
          const uint32_t ta = tmem + ((uint32_t)(q * 32) << 16) + acc * BN + cl;
          if constexpr (HC == 32) {
            uint32_t r[32];
            tmem_ld32(ta, r);
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
          } else {
            uint32_t r[16];
            tmem_ld16(ta, r);
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(r[j]);
          }
        }
        if (c == NCH - 1) {
          // accumulator drained: hand it back to the MMA warp
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[acc]);
        }
        if (ep.has_residual && !abort_flag &&
            !mbar_wait(&res_full[b], (cc >> 1) & 1u, wait_limit))
          abort_flag = 1;
#pragma unroll
        for (int j = 0; j < HC; j += 4) {
          const float4 bb = *reinterpret_cast<const float4*>(s_bias + cl + j);
          // the product (scaled per row by a folded RMSNorm) plus the bias
          float4 x = make_float4(fmaf(v[j], rs, bb.x), fmaf(v[j + 1], rs, bb.y),
                                 fmaf(v[j + 2], rs, bb.z), fmaf(v[j + 3], rs, bb.w));
          if (brow && n0 + cl + j < N) {
            const float4 br = *reinterpret_cast<const float4*>(brow + n0 + cl + j);
            x.x += br.x; x.y += br.y; x.z += br.z; x.w += br.w;
          }
          if (ep.act == ACT_SILU) {
            if (OUT_BF16) {
              x.x = silu_tanh(x.x); x.y = silu_tanh(x.y); x.z = silu_tanh(x.z); x.w = silu_tanh(x.w);
            } else {
              x.x = silu_f(x.x); x.y = silu_f(x.y); x.z = silu_f(x.z); x.w = silu_f(x.w);
            }
          }
          if (ep.has_residual) {            // fp32 output only: 4 columns = 16 bytes
            const float4 rr = *reinterpret_cast<const float4*>(
                s_res + b * CHUNK_BYTES + swz(row, (half * HC + j) >> 2));
            x.x += rr.x; x.y += rr.y; x.z += rr.z; x.w += rr.w;
          }
          v[j] = x.x; v[j + 1] = x.y; v[j + 2] = x.z; v[j + 3] = x.w;
        }
        if constexpr (FOLD && !OUT_BF16) {
          if (ep.c2) {                      // the next RMSNorm's input, and its sums
            // the warp holds 32 rows x 32 bytes: lanes 2i and 2i+1 store the two halves
            // of row i (then of row 16 + i), one whole 32-byte sector per pair
            static_assert(HC == 16, "fp32 chunk halves of 16 columns");
            auto store_rows = [&](const uint32_t (&wv)[HC / 2], __nv_bfloat16* dst) {
#pragma unroll
              for (int rd = 0; rd < 2; ++rd) {
                const int src = 16 * rd + (lane >> 1), piece = lane & 1;
                uint32_t o[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const uint32_t a0 = __shfl_sync(0xffffffffu, wv[k], src);
                  const uint32_t a1 = __shfl_sync(0xffffffffu, wv[4 + k], src);
                  o[k] = piece ? a1 : a0;
                }
                const int mr = m0 + q * 32 + src;
                if (mr < M && n0 + cl < N)
                  *reinterpret_cast<uint4*>(dst + (size_t)mr * ep.ldc2 + n0 + cl + 8 * piece) =
                      make_uint4(o[0], o[1], o[2], o[3]);
              }
            };
            float g[HC];
#pragma unroll
            for (int j = 0; j < HC; ++j) g[j] = v[j] * s_gain[cl + j];
            uint32_t wv[HC / 2];
#pragma unroll
            for (int j = 0; j < HC; j += 2) {
              ssq = fmaf(v[j], v[j], fmaf(v[j + 1], v[j + 1], ssq));
              wv[j / 2] = pack_bf16x2(g[j], g[j + 1]);
            }
            store_rows(wv, ep.c2);
            if (ep.c3) {
              const float4* tr = reinterpret_cast<const float4*>(
                  t_shared ? s_t + cl
                           : ep.c3_t + (size_t)(m < M ? m / ep.c3_rows_per : 0) * N + n0 + cl);
#pragma unroll
              for (int j = 0; j < HC; j += 4) {
                const float4 tv = tr[j / 4];
                wv[j / 2] = pack_bf16x2(g[j] * tv.x, g[j + 1] * tv.y);
                wv[j / 2 + 1] = pack_bf16x2(g[j + 2] * tv.z, g[j + 3] * tv.w);
              }
              store_rows(wv, ep.c3);
            }
          }
        }
        epi_bar();          // staging buffer b: its store two chunks ago has been read
        uint8_t* stg = s_out + b * CHUNK_BYTES;
        if (OUT_BF16) {
#pragma unroll
          for (int p = 0; p < 4; ++p) {     // 4 pieces of 8 bf16
            uint4 w;
            w.x = pack_bf16x2(v[8 * p + 0], v[8 * p + 1]);
            w.y = pack_bf16x2(v[8 * p + 2], v[8 * p + 3]);
            w.z = pack_bf16x2(v[8 * p + 4], v[8 * p + 5]);
            w.w = pack_bf16x2(v[8 * p + 6], v[8 * p + 7]);
            *reinterpret_cast<uint4*>(stg + swz(row, 4 * half + p)) = w;
          }
        } else {
#pragma unroll
          for (int p = 0; p < 4; ++p)       // 4 pieces of 4 floats
            *reinterpret_cast<float4*>(stg + swz(row, 4 * half + p)) =
                make_float4(v[4 * p], v[4 * p + 1], v[4 * p + 2], v[4 * p + 3]);
        }
        fence_async_shared();
        epi_bar();
        if (leader && !abort_flag && n0 + c * CH < N && !(FOLD && ep.no_c)) {
          tma_store_2d(&mapC, stg, n0 + c * CH, m0);
          tma_store_wait_read_le1();         // the other buffer is free for the next chunk
        }
      }
      if (FOLD && !OUT_BF16 && ep.c2 && m < M)
        ep.ss_out[(size_t)m * SS_LD + 2 * (t % tiles_n) + half] = ssq;
    }
    if (leader) tma_store_wait_all();
  }

  // ---- teardown
  tc_fence_before();
  __syncthreads();
  if (abort_flag) {
    if (threadIdx.x == 0) {
      set_status(status, LILICORR_ERR_TIMEOUT);
      // let copies still in flight land before the shared memory is released
      const long long t0 = clock64();
      while (clock64() - t0 < wait_limit / 10) {
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

template <int BN, bool OUT_BF16, bool FOLD>
lilicorr_status_t launch_bn(const GemmArgs& g, cudaStream_t st) {
  using Cfg = TcCfg<BN, OUT_BF16>;
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(gemm_tc_kernel<BN, OUT_BF16, FOLD>, configured));
  CUtensorMap ma, mw, mc, mr;
  const CUtensorMapDataType bf = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const CUtensorMapDataType f32 = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
  if (!make_map(&ma, g.A, bf, 2, g.M, g.Kd, g.lda, TC_BM, TC_BK)) return LILICORR_ERR_CUDA;
  if (!make_map(&mw, g.W, bf, 2, g.N, g.Kd, g.ldw, BN, TC_BK)) return LILICORR_ERR_CUDA;
  if (g.residual) {
    if (!make_map(&mr, g.residual, f32, 4, g.M, g.N, g.ldr, TC_BM, 32)) return LILICORR_ERR_CUDA;
  }
  if (g.C) {
    if (!make_map(&mc, g.C, OUT_BF16 ? bf : f32, OUT_BF16 ? 2 : 4, g.M, g.N, g.ldc, TC_BM, Cfg::CH))
      return LILICORR_ERR_CUDA;
  } else {
    mc = g.residual ? mr : ma;                 // never written (no_c)
  }
  if (!g.residual) mr = mc;                    // never read
  TcEpilogue ep;
  ep.bias = g.bias;
  ep.bias_rows = g.bias_rows;
  ep.rows_per_bias = g.rows_per_bias;
  ep.has_residual = g.residual != nullptr;
  ep.act = g.act;
  ep.c2 = static_cast<__nv_bfloat16*>(g.c2);
  ep.ldc2 = g.ldc2;
  ep.c2_gain = g.c2_gain;
  ep.ss_out = g.ss_out;
  ep.ss_in = g.ss_in;
  ep.ss_slots = g.ss_slots;
  ep.c3 = static_cast<__nv_bfloat16*>(g.c3);
  ep.c3_t = g.c3_t;
  ep.c3_rows_per = g.c3_rows_per;
  ep.no_c = g.C == nullptr;
  ep.ss_scale = 1.0f / (float)(g.ss_dim > 0 ? g.ss_dim : g.Kd);
  const int tiles = ceil_div(g.M, TC_BM) * ceil_div(g.N, BN);
  const int grid = tiles < num_sms() ? tiles : num_sms();
  const long long wait = g.wait_limit > 0 ? g.wait_limit : WAIT_LIMIT_CYCLES;
  LL_TRY(launch_k(gemm_tc_kernel<BN, OUT_BF16, FOLD>, grid, TC_THREADS, Cfg::SMEM, st, ma, mw, mc, mr, ep,
                  g.M, g.N, g.Kd, g.status, wait, g.test_starve));
  return LILICORR_OK;
}

// Column tile: the widest of 256/128/64 that still gives every SM a tile.
int tc_column_tile(int M, int N) {
  const int mt = ceil_div(M, TC_BM);
  const int sms = num_sms();
  if (N >= 256 && mt * ceil_div(N, 256) >= sms) return 256;
  if (N >= 128 && mt * ceil_div(N, 128) >= sms / 2) return 128;
  return 64;
}

template <bool OUT_BF16, bool FOLD>
lilicorr_status_t launch_out(const GemmArgs& g, cudaStream_t st) {
  const int bn = tc_column_tile(g.M, g.N);
  if (bn == 256) return launch_bn<256, OUT_BF16, FOLD>(g, st);
  if (bn == 128) return launch_bn<128, OUT_BF16, FOLD>(g, st);
  return launch_bn<64, OUT_BF16, FOLD>(g, st);
}

}  // namespace

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
    else
      (void)cudaGetLastError();
  }
  return fn;
}

bool make_map(CUtensorMap* map, const void* base, CUtensorMapDataType type, size_t es, int rows,
              int cols, int ld, int box_rows, int box_cols) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * es};
  cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, type, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_map_nd(CUtensorMap* map, const void* base, CUtensorMapDataType type, int rank,
                 const uint64_t* dims, const uint64_t* strides_bytes, const uint32_t* box) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || rank < 1 || rank > 5) return false;
  cuuint64_t d[5], st[4];
  cuuint32_t b[5], e[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    b[i] = box[i];
    e[i] = 1;
    if (i > 0) st[i - 1] = strides_bytes[i];
  }
  return fn(map, type, (cuuint32_t)rank, const_cast<void*>(base), d, st, b, e,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int gemm_tc_ss_slots(int M, int N) { return 2 * ceil_div(N, tc_column_tile(M, N)); }

bool gemm_tc_supported(const GemmArgs& g) {
  if (g.a_dt != LILICORR_BF16 || g.w_dt != LILICORR_BF16) return false;
  // folded RMSNorm: fp32 output, whole 32-column groups, 16-byte aligned bf16 copy rows
  if (g.c2 && (g.c_dt != LILICORR_F32 || !g.c2_gain || !g.ss_out || (g.N % 32) ||
               !aligned16(g.c2) || (g.ldc2 % 8) || gemm_tc_ss_slots(g.M, g.N) > SS_LD))
    return false;
  if (g.c3 && (!g.c2 || !g.c3_t || g.c3_rows_per < 1 || !aligned16(g.c3) || !aligned16(g.c3_t)))
    return false;
  if (g.ss_in && (g.ss_slots < 1 || g.ss_slots > SS_LD)) return false;
  if (g.M <= 0 || g.N <= 0 || g.Kd <= 0) return false;
  // TMA: 16-byte aligned bases and row strides, outputs in 16-byte column groups
  // C may be absent only for a folded producer (its bf16 copies are the output)
  if (!g.C && !(g.c2 && g.c_dt == LILICORR_F32)) return false;
  if (!aligned16(g.A) || !aligned16(g.W) || !aligned16(g.C)) return false;
  if ((g.lda % 8) || (g.ldw % 8) || (g.Kd % 8) || (g.N % 8) || (g.ldc % 8)) return false;
  if (g.residual && (g.c_dt != LILICORR_F32 || !aligned16(g.residual) || (g.ldr % 4)))
    return false;
  if (g.bias_rows && (g.N % 4)) return false;
  return encode_fn() != nullptr;
}

lilicorr_status_t launch_gemm_tc(const GemmArgs& g, cudaStream_t st) {
  const bool fold = g.c2 || g.ss_in;
  if (g.c_dt == LILICORR_BF16)
    return fold ? launch_out<true, true>(g, st) : launch_out<true, false>(g, st);
  return fold ? launch_out<false, true>(g, st) : launch_out<false, false>(g, st);
}

}  // namespace lilicorr
