// Step (1): per-slot top-K candidates and log-normaliser in one pass over the logits.
//
// Sec. 3.2 keeps each slot's top-K candidate tokens; App. A "Serving" fuses top-K
// extraction with vocabulary-wide logit normalisation. Here every logit is read
// from HBM exactly once:
//   * grid = (splits, rows): each CTA streams one contiguous chunk of one row with
//     16-byte loads, 4 in flight per thread;
//   * every thread keeps an online (max, sum exp) pair, merged by warp shuffles;
//   * every warp keeps its top-K as order-preserving 64-bit keys
//     (value, then lower id first) in shared memory, filtering with a warp-uniform
//     threshold; candidates that pass are appended through a ballot and merged
//     into the list when the buffer fills (rare after the first few vectors);
//   * the last CTA of a row to finish (atomic ticket, no waiting) merges the
//     splits' partial (max, sum, top-K) records and writes ids, logp, lse.
#include "internal.cuh"

namespace lilicorr {

namespace {

constexpr int TK_THREADS = 256;
constexpr int TK_WARPS = TK_THREADS / 32;
constexpr int TK_CAP = 96;             // candidate buffer per warp
constexpr int TK_UNROLL = 4;           // 16-byte loads in flight per thread
constexpr int TK_MAX_SPLITS = 64;
constexpr float LOG2E = 1.4426950408889634f;
constexpr unsigned FULL = 0xffffffffu;

// Order-preserving key: larger value first, equal values by lower id; -0.0 == +0.0.
__device__ __forceinline__ uint64_t make_key(float v, uint32_t id) {
  uint32_t b = __float_as_uint(v);
  if ((b << 1) == 0u) b = 0u;
  const uint32_t o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ((uint64_t)o << 32) | (uint64_t)(0xFFFFFFFFu - id);
}
__device__ __forceinline__ float key_value(uint64_t k) {
  const uint32_t o = (uint32_t)(k >> 32);
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}
__device__ __forceinline__ int32_t key_id(uint64_t k) {
  return (int32_t)(0xFFFFFFFFu - (uint32_t)k);
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t w = __shfl_xor_sync(FULL, v, o);
    v = w > v ? w : v;
  }
  return v;
}

// K largest keys of keys[0..n) (distinct except zeros = empty), by K rounds of
// "largest key below the previous one". Lane r returns the r-th key (0 if none).
__device__ uint64_t warp_select(const uint64_t* keys, int n, int K, int lane) {
  uint64_t prev = ~0ull, mine = 0ull;
  for (int r = 0; r < K; ++r) {
    uint64_t best = 0ull;
    for (int i = lane; i < n; i += 32) {
      const uint64_t k = keys[i];
      if (k < prev && k > best) best = k;
    }
    best = warp_max_u64(best);
    if (lane == r) mine = best;
    prev = best;
    if (best == 0ull) break;
  }
  return mine;
}

struct WarpState {
  uint64_t* list;    // [LILICORR_MAX_K] sorted descending; 0 = empty
  uint64_t* buf;     // [TK_CAP]; list and buf are contiguous: list first
  int nbuf;
  uint64_t thr;      // K-th key of the list (0 while the list is not full)
  float thr_val;     // its value (-inf while not full)
};

// Merge buffer and list into the list. The candidate set is list[0..K) followed by
// buf[0..nbuf) in one contiguous array, so a single selection pass covers both.
__device__ __forceinline__ void warp_flush(WarpState& w, int K, int lane) {
  __syncwarp();
  const uint64_t mine = warp_select(w.list, LILICORR_MAX_K + w.nbuf, K, lane);
  __syncwarp();
  if (lane < K) w.list[lane] = mine;
  w.thr = __shfl_sync(FULL, mine, K - 1);
  w.thr_val = w.thr ? key_value(w.thr) : -INFINITY;
  w.nbuf = 0;
  __syncwarp();
}

// Offer n values (ids id0 + j) of this lane to the warp list. Warp-collective.
template <int N>
__device__ __forceinline__ void warp_offer(WarpState& w, const float (&x)[N], uint32_t id0,
                                           bool hot, int K, int lane) {
#pragma unroll
  for (int j = 0; j < N; ++j) {
    const uint64_t key = make_key(x[j], id0 + (uint32_t)j);
    unsigned m = __ballot_sync(FULL, hot && key > w.thr);
    if (m == 0u) continue;
    if (w.nbuf + __popc(m) > TK_CAP) {
      warp_flush(w, K, lane);
      m = __ballot_sync(FULL, hot && key > w.thr);
      if (m == 0u) continue;
    }
    if ((m >> lane) & 1u) w.buf[w.nbuf + __popc(m & ((1u << lane) - 1u))] = key;
    w.nbuf += __popc(m);
  }
}

template <int N>
__device__ __forceinline__ void lse_update(float& m, float& s, const float (&x)[N], bool valid) {
  if (!valid) return;
  float vmax = x[0];
#pragma unroll
  for (int j = 1; j < N; ++j) vmax = fmaxf(vmax, x[j]);
  if (vmax > m) {
    s *= ex2((m - vmax) * LOG2E);
    m = vmax;
  }
  if (m == -INFINITY) return;
  const float ml = m * LOG2E;
  float acc[N];
#pragma unroll
  for (int j = 0; j < N; ++j) acc[j] = ex2(fmaf(x[j], LOG2E, -ml));
#pragma unroll
  for (int w = 1; w < N; w <<= 1)
#pragma unroll
    for (int j = 0; j + w < N; j += 2 * w) acc[j] += acc[j + w];
  s += acc[0];
}

template <typename T> struct Vec;
template <> struct Vec<uint16_t> {        // bf16
  static constexpr int N = 8;
  __device__ static void unpack(const uint4& v, float (&x)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      x[2 * i] = __uint_as_float(w[i] << 16);
      x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
  __device__ static float scalar(const uint16_t* p, size_t i) { return bf16_to_f32(p[i]); }
};
template <> struct Vec<float> {
  static constexpr int N = 4;
  __device__ static void unpack(const uint4& v, float (&x)[4]) {
    x[0] = __uint_as_float(v.x); x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z); x[3] = __uint_as_float(v.w);
  }
  __device__ static float scalar(const float* p, size_t i) { return p[i]; }
};

struct Rec {            // partial record of one (row, split)
  float m, s;
  uint64_t keys[1];     // [K]
};

template <typename T>
__global__ void __launch_bounds__(TK_THREADS)
topk_lse_kernel(const T* __restrict__ logits, int V, int K, int splits, int chunk_vecs,
                size_t rec_bytes, int32_t* __restrict__ ids, float* __restrict__ logp,
                float* __restrict__ lse, uint32_t* status, uint32_t* counters,
                unsigned char* partials) {
  constexpr int VEC = Vec<T>::N;
  __shared__ uint64_t s_keys[TK_WARPS][LILICORR_MAX_K + TK_CAP];
  __shared__ uint64_t s_merge[TK_MAX_SPLITS * LILICORR_MAX_K];
  __shared__ float s_m[TK_WARPS], s_s[TK_WARPS];
  __shared__ int s_last;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int split = blockIdx.x;
  const int row = blockIdx.y;
  const T* rp = logits + (size_t)row * V;

  // vector-aligned region of this row: [e0, e0 + nvec * VEC)
  const size_t gstart = (size_t)row * V;
  const int e0 = min((int)((VEC - (gstart % VEC)) % VEC), V);
  const int nvec = (V - e0) / VEC;
  const int v_begin = min(split * chunk_vecs, nvec);
  const int v_end = min(v_begin + chunk_vecs, nvec);

  WarpState w;
  w.list = s_keys[warp];
  w.buf = s_keys[warp] + LILICORR_MAX_K;
  w.nbuf = 0;
  w.thr = 0ull;
  w.thr_val = -INFINITY;
  w.list[lane] = 0ull;
  __syncwarp();

  float m = -INFINITY, s = 0.f;

  // scalar head [0, e0) and tail [e0 + nvec*VEC, V): warp 0 of split 0, one element per lane
  if (split == 0 && warp == 0) {
    const int tail0 = e0 + nvec * VEC;
    const int nscalar = e0 + (V - tail0);
    for (int base = 0; base < nscalar; base += 32) {
      const int i = base + lane;
      const bool valid = i < nscalar;
      const int e = valid ? (i < e0 ? i : tail0 + (i - e0)) : 0;
      float x[1] = {valid ? Vec<T>::scalar(rp, e) : -INFINITY};
      lse_update<1>(m, s, x, valid);
      const bool hot = valid && x[0] >= w.thr_val;
      if (__any_sync(FULL, hot)) warp_offer<1>(w, x, (uint32_t)e, hot, K, lane);
    }
  }

  // main stream: 16-byte vectors, TK_UNROLL loads in flight per thread
  const uint4* vp = reinterpret_cast<const uint4*>(rp + e0);
  for (int it = v_begin; it < v_end; it += TK_UNROLL * TK_THREADS) {
    uint4 raw[TK_UNROLL];
#pragma unroll
    for (int u = 0; u < TK_UNROLL; ++u) {
      const int v = it + u * TK_THREADS + tid;
      if (v < v_end) raw[u] = __ldcs(vp + v);
      else raw[u] = make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < TK_UNROLL; ++u) {
      const int v = it + u * TK_THREADS + tid;
      const bool valid = v < v_end;
      float x[VEC];
      Vec<T>::unpack(raw[u], x);
      lse_update<VEC>(m, s, x, valid);
      float vmax = x[0];
#pragma unroll
      for (int j = 1; j < VEC; ++j) vmax = fmaxf(vmax, x[j]);
      const bool hot = valid && vmax >= w.thr_val;
      if (__any_sync(FULL, hot))
        warp_offer<VEC>(w, x, (uint32_t)(e0 + v * VEC), hot, K, lane);
    }
  }
  warp_flush(w, K, lane);

  // (max, sum) of the warp, then of the CTA
  const float wm = warp_max(m);
  float ws = (m == -INFINITY) ? 0.f : s * ex2((m - wm) * LOG2E);
  ws = warp_sum(ws);
  if (lane == 0) { s_m[warp] = wm; s_s[warp] = ws; }
  __syncthreads();

  float cm = -INFINITY, cs = 0.f;
  if (warp == 0) {
    const float pm = lane < TK_WARPS ? s_m[lane] : -INFINITY;
    const float ps = lane < TK_WARPS ? s_s[lane] : 0.f;
    cm = warp_max(pm);
    cs = warp_sum(pm == -INFINITY ? 0.f : ps * ex2((pm - cm) * LOG2E));
  }
  // CTA top-K over the warps' lists (list entries >= K are zero)
  uint64_t mine = 0ull;
  if (warp == 0) {
    // gather the warp lists into s_merge so the selection reads only list entries
    for (int i = lane; i < TK_WARPS * LILICORR_MAX_K; i += 32)
      s_merge[i] = s_keys[i / LILICORR_MAX_K][i % LILICORR_MAX_K];
    __syncwarp();
    mine = warp_select(s_merge, TK_WARPS * LILICORR_MAX_K, K, lane);
  }

  if (splits == 1) {
    if (warp == 0) {
      const float l = cm + logf(cs);
      const bool bad = !(isfinite(l));
      if (lane == 0) {
        lse[row] = l;
        if (bad) set_status(status, LILICORR_ERR_NONFINITE);
      }
      if (lane < K) {
        ids[(size_t)row * K + lane] = key_id(mine);
        logp[(size_t)row * K + lane] = key_value(mine) - l;
      }
    }
    return;
  }

  // publish this split's partial record, then take a ticket
  Rec* rec = reinterpret_cast<Rec*>(partials + ((size_t)row * splits + split) * rec_bytes);
  if (warp == 0) {
    if (lane == 0) { rec->m = cm; rec->s = cs; }
    if (lane < K) rec->keys[lane] = mine;
    __threadfence();
  }
  __syncthreads();
  if (tid == 0) {
    const uint32_t ticket = atomicAdd(&counters[row], 1u);
    s_last = (ticket == (uint32_t)(splits - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // last CTA of the row: merge all splits
  for (int i = tid; i < splits * K; i += TK_THREADS) {
    const Rec* r = reinterpret_cast<const Rec*>(partials + ((size_t)row * splits + i / K) * rec_bytes);
    s_merge[i] = __ldcg(reinterpret_cast<const unsigned long long*>(&r->keys[i % K]));
  }
  __syncthreads();
  if (warp == 0) {
    float pm = -INFINITY, ps = 0.f;
    for (int i = lane; i < splits; i += 32) {
      const Rec* r = reinterpret_cast<const Rec*>(partials + ((size_t)row * splits + i) * rec_bytes);
      const float rm = __ldcg(&r->m), rs = __ldcg(&r->s);
      if (rm == -INFINITY) continue;
      if (rm > pm) { ps = ps * ex2((pm - rm) * LOG2E) + rs; pm = rm; }
      else ps += rs * ex2((rm - pm) * LOG2E);
    }
    const float gm = warp_max(pm);
    const float gs = warp_sum(pm == -INFINITY ? 0.f : ps * ex2((pm - gm) * LOG2E));
    const uint64_t top = warp_select(s_merge, splits * K, K, lane);
    const float l = gm + logf(gs);
    if (lane == 0) {
      lse[row] = l;
      if (!isfinite(l)) set_status(status, LILICORR_ERR_NONFINITE);
      counters[row] = 0u;             // leave the workspace reusable
    }
    if (lane < K) {
      ids[(size_t)row * K + lane] = key_id(top);
      logp[(size_t)row * K + lane] = key_value(top) - l;
    }
  }
}

}  // namespace

TopkPlan topk_plan(int rows, int V, int K, lilicorr_dtype_t dt) {
  const int vec = dt == LILICORR_BF16 ? 8 : 4;
  const int nvec = V / vec;
  const int target_ctas = num_sms() * 4;
  const int min_chunk = 512;                 // vectors (8 KB) per CTA at least
  int splits = ceil_div(target_ctas, rows);
  splits = max(1, min(splits, ceil_div(max(nvec, 1), min_chunk)));
  splits = min(splits, TK_MAX_SPLITS);
  TopkPlan p;
  p.splits = splits;
  p.chunk_vecs = ceil_div(max(nvec, 1), splits);
  p.rec_bytes = align_up(8 + 8 * (size_t)K, 16);
  return p;
}

size_t topk_ws_bytes(int rows, int V, int K, lilicorr_dtype_t dt) {
  const TopkPlan p = topk_plan(rows, V, K, dt);
  return 256 + align_up((size_t)rows * 4, 256) + align_up((size_t)rows * p.splits * p.rec_bytes, 256);
}

lilicorr_status_t launch_topk_lse(const void* logits, lilicorr_dtype_t dt, int rows, int V, int K,
                                  int32_t* ids, float* logp, float* lse, uint32_t* status,
                                  uint32_t* counters, void* partials, cudaStream_t st) {
  if (rows == 0) return LILICORR_OK;
  const TopkPlan p = topk_plan(rows, V, K, dt);
  dim3 grid(p.splits, rows);
  if (dt == LILICORR_BF16)
    topk_lse_kernel<uint16_t><<<grid, TK_THREADS, 0, st>>>(
        static_cast<const uint16_t*>(logits), V, K, p.splits, p.chunk_vecs, p.rec_bytes, ids, logp,
        lse, status, counters, static_cast<unsigned char*>(partials));
  else
    topk_lse_kernel<float><<<grid, TK_THREADS, 0, st>>>(
        static_cast<const float*>(logits), V, K, p.splits, p.chunk_vecs, p.rec_bytes, ids, logp,
        lse, status, counters, static_cast<unsigned char*>(partials));
  return last_launch();
}

}  // namespace lilicorr
