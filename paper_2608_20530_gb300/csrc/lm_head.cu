// The LM-head projection fused with step (1): logits = hidden W_vocab^T are formed tile by
// tile on the tensor cores and consumed in tensor memory by the online log-sum-exp and the
// top-K selection, so the [rows, V] logits never reach HBM (the step before the path in
// the paper's cost breakdown, Table "cost"; Sec. 3.2 top-K pool; App. A "Serving").
//
// A persistent, warp-specialised tcgen05 kernel, one CTA per SM, 192 threads:
//   * warp 0 (one lane) streams 128 x 64 tiles of hidden and 256 x 64 tiles of W_vocab
//     (bf16, 128-byte swizzle) into a four-stage ring with 2-D TMA copies;
//   * warp 1 allocates two 256-column accumulators in tensor memory; its lane 0 issues
//     tcgen05.mma (M = 128, N = 256, K = 16), four per stage, and hands finished
//     accumulators to the epilogue;
//   * warps 2-5 own one row each per thread (tensor-memory lane = row). While the next
//     tile's products run on the other accumulator they read the 256 logits of their row
//     with tcgen05.ld and fold them into the row's running maximum, its sum of exponentials
//     below that maximum and its top-K list (shared memory, sorted; a logit enters only if
//     it beats the list's K-th value).
// Every CTA keeps one 128-row block of hidden and walks vocabulary tiles in increasing
// order (the CTAs of one vocabulary tile run side by side, so W_vocab crosses HBM about
// once). At the end each CTA writes its rows' partial records (the vocabulary-shard format
// of lilicorr_topk_lse_partial: max, sum, K values, K ids); the merge kernel of step (1)
// combines the records of all CTAs into ids, log-probabilities and the log-normaliser.
// Every mbarrier wait is bounded (about 2 s of SM cycles); on timeout the kernel records
// LILICORR_ERR_TIMEOUT, stops issuing work, lets copies in flight land, frees tensor
// memory and returns.
#include "tc_ptx.cuh"

namespace lilicorr {

namespace {
using namespace tc;

constexpr int LH_BM = 128;
constexpr int LH_BN = 256;
constexpr int LH_BK = 64;                  // 64 bf16 = 128 bytes: one swizzle atom row
constexpr int LH_STAGES = 4;
constexpr int LH_THREADS = 192;            // producer, MMA, 4 epilogue warps
constexpr int LH_EPI = 128;
constexpr uint32_t LH_A_BYTES = LH_BM * LH_BK * 2;
constexpr uint32_t LH_B_BYTES = LH_BN * LH_BK * 2;
constexpr size_t LH_SMEM = 1024 + (size_t)LH_STAGES * (LH_A_BYTES + LH_B_BYTES);
constexpr uint32_t LH_TMEM_COLS = 2 * LH_BN;
constexpr long long LH_WAIT = 4000000000ll;
constexpr float LH_LOG2E = 1.4426950408889634f;

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Work split: CTA c keeps row block c % tiles_m and takes vocabulary tiles
// c / tiles_m, c / tiles_m + per, ... with per = gridDim.x / tiles_m.
struct LhShape {
  int rows, H, V, K, tiles_m, tiles_n;
};

__global__ void __launch_bounds__(LH_THREADS, 1)
    lm_head_topk_kernel(const __grid_constant__ CUtensorMap mapA,
                        const __grid_constant__ CUtensorMap mapW, LhShape sh,
                        unsigned char* __restrict__ recs, uint32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + LH_STAGES * LH_A_BYTES;
  __shared__ __align__(8) uint64_t full[LH_STAGES], empty[LH_STAGES], acc_full[2], acc_empty[2];
  __shared__ uint64_t s_list[LILICORR_MAX_K * LH_BM];   // [k][row] running top-K keys
  __shared__ uint32_t tmem_base;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = gridDim.x / sh.tiles_m;
  const int mt = blockIdx.x % sh.tiles_m;
  const int n_first = blockIdx.x / sh.tiles_m;
  const int nk = sh.H / LH_BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < LH_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], LH_EPI / 32);
    }
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(&tmem_base, LH_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  pdl_wait();

  if (warp == 0) {
    // ---- producer
    if (lane == 0) {
      uint32_t g = 0;
      for (int nt = n_first; nt < sh.tiles_n && !abort_flag; nt += per) {
        for (int i = 0; i < nk; ++i, ++g) {
          const int s = (int)(g % LH_STAGES);
          const uint32_t ph = (g / LH_STAGES) & 1u;
          if (!mbar_wait(&empty[s], ph ^ 1u, LH_WAIT)) {
            abort_flag = 1;
            break;
          }
          mbar_expect_tx(&full[s], LH_A_BYTES + LH_B_BYTES);
          tma_load_2d(sA + (size_t)s * LH_A_BYTES, &mapA, &full[s], i * LH_BK, mt * LH_BM);
          tma_load_2d(sB + (size_t)s * LH_B_BYTES, &mapW, &full[s], i * LH_BK, nt * LH_BN);
        }
      }
    }
  } else if (warp == 1) {
    // ---- MMA issuer, accumulators alternating
    if (lane == 0) {
      constexpr uint32_t idesc = instr_desc(LH_BM, LH_BN);
      uint32_t g = 0, lt = 0;
      for (int nt = n_first; nt < sh.tiles_n && !abort_flag; nt += per, ++lt) {
        const uint32_t acc = lt & 1u;
        if (!mbar_wait(&acc_empty[acc], ((lt >> 1) & 1u) ^ 1u, LH_WAIT)) {
          abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + acc * LH_BN;
        for (int i = 0; i < nk; ++i, ++g) {
          const int s = (int)(g % LH_STAGES);
          const uint32_t ph = (g / LH_STAGES) & 1u;
          if (!mbar_wait(&full[s], ph, LH_WAIT)) {
            abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc(sA + (size_t)s * LH_A_BYTES);
          const uint64_t bd = smem_desc(sB + (size_t)s * LH_B_BYTES);
#pragma unroll
          for (int k = 0; k < LH_BK / 16; ++k)
            mma_bf16(d, ad + 2ull * k, bd + 2ull * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
          mma_commit(&empty[s]);
        }
        mma_commit(&acc_full[acc]);
      }
    }
  } else {
    // ---- epilogue: thread (q, lane) owns row q*32 + lane of the block
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int grow = mt * LH_BM + row;
    const bool valid = grow < sh.rows;
    const int K = sh.K;
    float m_run = -INFINITY, s_run = 0.f, thr = -INFINITY;
    int n_in = 0;
    uint32_t lt = 0;
    for (int nt = n_first; nt < sh.tiles_n; nt += per, ++lt) {
      const uint32_t acc = lt & 1u;
      if (!abort_flag && !mbar_wait(&acc_full[acc], (lt >> 1) & 1u, LH_WAIT)) abort_flag = 1;
      tc_fence_after();
      const int n0 = nt * LH_BN;
#pragma unroll 1
      for (int c = 0; c < LH_BN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + acc * LH_BN + c * 32, r);
        if (c == LH_BN / 32 - 1) {
          // accumulator drained: hand it back to the MMA warp
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[acc]);
        }
        if (!valid || abort_flag) continue;
        const int col0 = n0 + c * 32;
        float v[32];
        float cmax = -INFINITY;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          v[j] = col0 + j < sh.V ? __uint_as_float(r[j]) : -INFINITY;
          cmax = fmaxf(cmax, v[j]);
        }
        if (cmax == -INFINITY) continue;              // only columns past the vocabulary
        if (cmax > m_run) {
          s_run *= ex2_approx((m_run - cmax) * LH_LOG2E);
          m_run = cmax;
        }
        const float ml = m_run * LH_LOG2E;
        float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
          a0 += ex2_approx(fmaf(v[j], LH_LOG2E, -ml));
          a1 += ex2_approx(fmaf(v[j + 1], LH_LOG2E, -ml));
          a2 += ex2_approx(fmaf(v[j + 2], LH_LOG2E, -ml));
          a3 += ex2_approx(fmaf(v[j + 3], LH_LOG2E, -ml));
        }
        s_run += (a0 + a1) + (a2 + a3);
        if (cmax > thr) {
          // candidates, in increasing id order: a logit equal to the K-th value has a
          // larger id than every listed one, so only a strictly larger logit enters
          uint32_t hm = 0u;
#pragma unroll
          for (int j = 0; j < 32; ++j) hm |= v[j] > thr ? (1u << j) : 0u;
          while (hm) {
            const int j = __ffs(hm) - 1;
            hm &= hm - 1u;
            float x = v[0];
#pragma unroll
            for (int t = 1; t < 32; ++t) x = j == t ? v[t] : x;
            if (!(x > thr)) continue;                 // the K-th value has risen since
            const uint64_t key = make_key(x, (uint32_t)(col0 + j));
            int i = n_in < K ? n_in++ : K - 1;
            while (i > 0 && s_list[(i - 1) * LH_BM + row] < key) {
              s_list[i * LH_BM + row] = s_list[(i - 1) * LH_BM + row];
              --i;
            }
            s_list[i * LH_BM + row] = key;
            if (n_in == K) thr = key_value(s_list[(K - 1) * LH_BM + row]);
          }
        }
      }
    }
    if (valid && !abort_flag) {
      // this CTA's partial record of row grow: record index n_first (one per CTA of
      // the row block), rows of the record set in order
      unsigned char* rec = recs + ((size_t)n_first * sh.rows + grow) * topk_partial_bytes(K);
      float* rf = reinterpret_cast<float*>(rec);
      int32_t* ri = reinterpret_cast<int32_t*>(rec + 8 + 4 * (size_t)K);
      rf[0] = m_run;
      rf[1] = s_run;
      for (int k = 0; k < K; ++k) {
        const uint64_t key = k < n_in ? s_list[k * LH_BM + row] : 0ull;
        rf[2 + k] = key ? key_value(key) : -INFINITY;
        ri[k] = key ? key_id(key) : -1;
      }
    }
  }

  // ---- teardown
  tc_fence_before();
  __syncthreads();
  if (abort_flag) {
    if (threadIdx.x == 0) {
      set_status(status, LILICORR_ERR_TIMEOUT);
      const long long t0 = clock64();          // let copies in flight land
      while (clock64() - t0 < LH_WAIT / 10) {
      }
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, LH_TMEM_COLS);
  }
}

// ----------------------------------------------------------------------------- few rows
// Up to 16 rows (a batch-1 block): the roles of the operands swap. A vocabulary tile of
// 128 rows of W_vocab is the A operand (M = 128) and the hidden rows the B operand (N = 16),
// so the accumulator holds one vocabulary row per tensor-memory lane and one hidden row per
// column: each of the 128 epilogue threads folds its vocabulary row's logits (one per
// hidden row) into a running maximum and sum per hidden row, and appends the ones above the
// hidden row's current K-th value to that row's candidate list in shared memory (an atomic
// slot). After every tile a warp compacts each list of more than K keys to its K largest
// by rank counting and raises the row's filter to the K-th value; a later logit equal to
// it loses the tie (every CTA meets the vocabulary in increasing id order), so the filter is
// strict. A stage is 18 KB instead of 48 KB (the 128-row hidden tile was mostly padding),
// so the ring is ten deep.
constexpr int LS_BM = 128;                 // vocabulary rows per tile (M)
constexpr int LS_BN = 16;                  // hidden rows (N)
constexpr int LS_STAGES = 10;
constexpr uint32_t LS_A_BYTES = LS_BM * LH_BK * 2;
constexpr uint32_t LS_B_BYTES = LS_BN * LH_BK * 2;
constexpr int LS_CAP = LS_BM + LILICORR_MAX_K;   // candidates of a row between compactions
constexpr size_t LS_SMEM = 1024 + (size_t)LS_STAGES * (LS_A_BYTES + LS_B_BYTES) +
                           (size_t)LS_BN * LS_CAP * sizeof(uint64_t);
constexpr uint32_t LS_TMEM_COLS = 32;      // two 16-column accumulators

// order image of a float as in the candidate keys (-0.0 == +0.0): x > y as floats iff
// ord_f32(x) > ord_f32(y)
__device__ __forceinline__ uint32_t ord_f32(float v) { return (uint32_t)(make_key(v, 0u) >> 32); }

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

__device__ __forceinline__ void ls_bar() {  // the four epilogue warps
  asm volatile("bar.sync 1, %0;" ::"n"(LH_EPI) : "memory");
}

// Compact hidden row j's candidate list (keys in cand[0..n), n <= LS_CAP) to its K largest,
// sorted descending, by one warp; returns the new count. tmp: K keys of scratch.
__device__ __forceinline__ int ls_compact(uint64_t* cand, int n, int K, uint64_t* tmp, int lane) {
  for (int i = lane; i < K; i += 32) tmp[i] = 0ull;
  __syncwarp();
  for (int i = lane; i < n; i += 32) {
    const uint64_t c = cand[i];
    int rank = 0;
    for (int t = 0; t < n; ++t) rank += cand[t] > c ? 1 : 0;
    if (rank < K) tmp[rank] = c;
  }
  __syncwarp();
  const int kept = min(n, K);
  for (int i = lane; i < kept; i += 32) cand[i] = tmp[i];
  __syncwarp();
  return kept;
}

__global__ void __launch_bounds__(LH_THREADS, 1)
    lm_head_rows_kernel(const __grid_constant__ CUtensorMap mapW,
                        const __grid_constant__ CUtensorMap mapH, LhShape sh,
                        unsigned char* __restrict__ recs, uint32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sW = smem;
  uint8_t* sH = smem + LS_STAGES * LS_A_BYTES;
  uint64_t* cand = reinterpret_cast<uint64_t*>(sH + LS_STAGES * LS_B_BYTES);   // [LS_BN][LS_CAP]
  __shared__ __align__(8) uint64_t full[LS_STAGES], empty[LS_STAGES], acc_full[2], acc_empty[2];
  __shared__ uint64_t s_tmp[4][LILICORR_MAX_K];
  __shared__ int cnt[LS_BN];
  __shared__ uint32_t thr_o[LS_BN];         // order image of each row's filter value
  __shared__ float red_m[4][LS_BN], red_s[4][LS_BN];
  __shared__ uint32_t tmem_base;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = gridDim.x;
  const int nk = sh.H / LH_BK;
  const int R = sh.rows, K = sh.K;

  if (threadIdx.x == 0) {
    for (int s = 0; s < LS_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], LH_EPI / 32);
    }
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (threadIdx.x < LS_BN) {
    cnt[threadIdx.x] = 0;
    thr_o[threadIdx.x] = ord_f32(-INFINITY);
  }
  if (warp == 1) tmem_alloc(&tmem_base, LS_TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  pdl_wait();

  if (warp == 0) {
    // ---- producer: a vocabulary tile and the hidden rows' matching columns per stage
    if (lane == 0) {
      uint32_t g = 0;
      for (int nt = blockIdx.x; nt < sh.tiles_n && !abort_flag; nt += per) {
        for (int i = 0; i < nk; ++i, ++g) {
          const int s = (int)(g % LS_STAGES);
          const uint32_t ph = (g / LS_STAGES) & 1u;
          if (!mbar_wait(&empty[s], ph ^ 1u, LH_WAIT)) {
            abort_flag = 1;
            break;
          }
          mbar_expect_tx(&full[s], LS_A_BYTES + LS_B_BYTES);
          tma_load_2d(sW + (size_t)s * LS_A_BYTES, &mapW, &full[s], i * LH_BK, nt * LS_BM);
          tma_load_2d(sH + (size_t)s * LS_B_BYTES, &mapH, &full[s], i * LH_BK, 0);
        }
      }
    }
  } else if (warp == 1) {
    // ---- MMA issuer, accumulators alternating
    if (lane == 0) {
      constexpr uint32_t idesc = instr_desc(LS_BM, LS_BN);
      uint32_t g = 0, lt = 0;
      for (int nt = blockIdx.x; nt < sh.tiles_n && !abort_flag; nt += per, ++lt) {
        const uint32_t acc = lt & 1u;
        if (!mbar_wait(&acc_empty[acc], ((lt >> 1) & 1u) ^ 1u, LH_WAIT)) {
          abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + acc * LS_BN;
        for (int i = 0; i < nk; ++i, ++g) {
          const int s = (int)(g % LS_STAGES);
          const uint32_t ph = (g / LS_STAGES) & 1u;
          if (!mbar_wait(&full[s], ph, LH_WAIT)) {
            abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint64_t ad = smem_desc(sW + (size_t)s * LS_A_BYTES);
          const uint64_t bd = smem_desc(sH + (size_t)s * LS_B_BYTES);
#pragma unroll
          for (int k = 0; k < LH_BK / 16; ++k)
            mma_bf16(d, ad + 2ull * k, bd + 2ull * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
          mma_commit(&empty[s]);
        }
        mma_commit(&acc_full[acc]);
      }
    }
  } else {
    // ---- epilogue: thread (q, lane) owns vocabulary row 32 q + lane of every tile
    const int q = warp & 3;
    const int vrow = q * 32 + lane;
    float m_run[LS_BN], s_run[LS_BN];
#pragma unroll
    for (int j = 0; j < LS_BN; ++j) {
      m_run[j] = -INFINITY;
      s_run[j] = 0.f;
    }
    uint32_t lt = 0;
    for (int nt = blockIdx.x; nt < sh.tiles_n; nt += per, ++lt) {
      const uint32_t acc = lt & 1u;
      if (!abort_flag && !mbar_wait(&acc_full[acc], (lt >> 1) & 1u, LH_WAIT)) abort_flag = 1;
      tc_fence_after();
      uint32_t r[LS_BN];
      tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + acc * LS_BN, r);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[acc]);      // accumulator drained
      const int vid = nt * LS_BM + vrow;
      if (!abort_flag && vid < sh.V) {
#pragma unroll
        for (int j = 0; j < LS_BN; ++j) {
          if (j >= R) break;
          const float x = __uint_as_float(r[j]);
          if (x > m_run[j]) {
            s_run[j] = s_run[j] * ex2_approx((m_run[j] - x) * LH_LOG2E) + 1.f;
            m_run[j] = x;
          } else {
            s_run[j] += ex2_approx((x - m_run[j]) * LH_LOG2E);
          }
          if (ord_f32(x) > *(volatile uint32_t*)&thr_o[j]) {
            const int pos = atomicAdd(&cnt[j], 1);
            if (pos < LS_CAP) cand[j * LS_CAP + pos] = make_key(x, (uint32_t)vid);
          }
        }
      }
      ls_bar();                                  // this tile's candidates are in
      for (int j = q; j < R; j += 4) {
        const int n = min(cnt[j], LS_CAP);
        if (n > K) {
          const int kept = ls_compact(cand + j * LS_CAP, n, K, s_tmp[q], lane);
          if (lane == 0) {
            cnt[j] = kept;
            // later logits equal to the K-th value carry larger ids: they lose the tie
            thr_o[j] = ord_f32(key_value(cand[j * LS_CAP + K - 1]));
          }
        }
      }
      ls_bar();                                  // lists and filters ready for the next tile
    }
    // the CTA's record of each hidden row: (max, sum) over its threads, K largest keys
#pragma unroll
    for (int j = 0; j < LS_BN; ++j) {
      if (j >= R) break;
      const float wm = warp_max(m_run[j]);
      const float ws = warp_sum(m_run[j] == -INFINITY ? 0.f : s_run[j] * ex2_approx((m_run[j] - wm) * LH_LOG2E));
      if (lane == 0) {
        red_m[q][j] = wm;
        red_s[q][j] = ws;
      }
    }
    for (int j = q; j < R; j += 4) {             // sorted, descending
      const int n = min(cnt[j], LS_CAP);
      const int kept = ls_compact(cand + j * LS_CAP, n, K, s_tmp[q], lane);
      if (lane == 0) cnt[j] = kept;
    }
    ls_bar();
    if (!abort_flag && threadIdx.x - 64 < R) {
      const int j = threadIdx.x - 64;
      float gm = -INFINITY;
      for (int w = 0; w < 4; ++w) gm = fmaxf(gm, red_m[w][j]);
      float gs = 0.f;
      for (int w = 0; w < 4; ++w)
        if (red_m[w][j] != -INFINITY) gs += red_s[w][j] * ex2_approx((red_m[w][j] - gm) * LH_LOG2E);
      unsigned char* rec = recs + ((size_t)blockIdx.x * R + j) * topk_partial_bytes(K);
      float* rf = reinterpret_cast<float*>(rec);
      int32_t* ri = reinterpret_cast<int32_t*>(rec + 8 + 4 * (size_t)K);
      rf[0] = gm;
      rf[1] = gs;
      const int n = cnt[j];
      for (int k = 0; k < K; ++k) {
        const uint64_t key = k < n ? cand[j * LS_CAP + k] : 0ull;
        rf[2 + k] = key ? key_value(key) : -INFINITY;
        ri[k] = key ? key_id(key) : -1;
      }
    }
  }

  // ---- teardown
  tc_fence_before();
  __syncthreads();
  if (abort_flag) {
    if (threadIdx.x == 0) {
      set_status(status, LILICORR_ERR_TIMEOUT);
      const long long t0 = clock64();          // let copies in flight land
      while (clock64() - t0 < LH_WAIT / 10) {
      }
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, LS_TMEM_COLS);
  }
}

int lm_head_rows_grid(int V) {
  const int tiles = ceil_div(V, LS_BM);
  return tiles < num_sms() ? tiles : num_sms();
}

// CTAs of the fused kernel: a multiple of the row blocks, at most one per SM and at most
// one per (row block, vocabulary tile).
int lm_head_grid(int rows, int V) {
  const int tiles_m = ceil_div(rows, LH_BM), tiles_n = ceil_div(V, LH_BN);
  int per = num_sms() / tiles_m;
  if (per < 1) per = 1;
  if (per > tiles_n) per = tiles_n;
  return per * tiles_m;
}

}  // namespace

bool lm_head_supported(int rows, int H, int V, int K) {
  return rows > 0 && H >= LH_BK && H % LH_BK == 0 && V >= K && K > 0 && K <= LILICORR_MAX_K &&
         encode_fn() != nullptr;
}

size_t lm_head_records_bytes(int rows, int V, int K) {
  if (rows <= LS_BN) return (size_t)lm_head_rows_grid(V) * rows * topk_partial_bytes(K);
  return (size_t)(lm_head_grid(rows, V) / ceil_div(rows, LH_BM)) * rows * topk_partial_bytes(K);
}

lilicorr_status_t launch_lm_head_topk(const void* hidden, const void* w_vocab, int rows, int H,
                                      int V, int K, void* recs, int32_t* ids, float* logp,
                                      float* lse, uint32_t* status, cudaStream_t st) {
  const CUtensorMapDataType bf = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  LhShape sh;
  sh.rows = rows; sh.H = H; sh.V = V; sh.K = K;
  if (rows <= LS_BN) {
    // few rows: vocabulary tiles as the A operand, the hidden rows as B (N = 16)
    static bool configured_rows[64] = {false};
    LL_TRY(allow_max_dynamic_smem(lm_head_rows_kernel, configured_rows));
    CUtensorMap mw, mh;
    if (!make_map(&mw, w_vocab, bf, 2, V, H, H, LS_BM, LH_BK)) return LILICORR_ERR_CUDA;
    if (!make_map(&mh, hidden, bf, 2, rows, H, H, LS_BN, LH_BK)) return LILICORR_ERR_CUDA;
    sh.tiles_m = 1;
    sh.tiles_n = ceil_div(V, LS_BM);
    const int grid = lm_head_rows_grid(V);
    LL_TRY(launch_k(lm_head_rows_kernel, grid, LH_THREADS, LS_SMEM, st, mw, mh, sh,
                    static_cast<unsigned char*>(recs), status));
    return launch_topk_merge(recs, grid, rows, K, ids, logp, lse, status, st);
  }
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(lm_head_topk_kernel, configured));
  CUtensorMap ma, mw;
  if (!make_map(&ma, hidden, bf, 2, rows, H, H, LH_BM, LH_BK)) return LILICORR_ERR_CUDA;
  if (!make_map(&mw, w_vocab, bf, 2, V, H, H, LH_BN, LH_BK)) return LILICORR_ERR_CUDA;
  sh.tiles_m = ceil_div(rows, LH_BM);
  sh.tiles_n = ceil_div(V, LH_BN);
  const int grid = lm_head_grid(rows, V);
  LL_TRY(launch_k(lm_head_topk_kernel, grid, LH_THREADS, LH_SMEM, st, ma, mw, sh,
                  static_cast<unsigned char*>(recs), status));
  return launch_topk_merge(recs, grid / sh.tiles_m, rows, K, ids, logp, lse, status, st);
}

}  // namespace lilicorr
