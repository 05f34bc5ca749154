// Step (1): per-slot top-K candidates and log-normaliser in one pass over the logits.
//
// Sec. 3.2 keeps each slot's top-K candidate tokens; App. A "Serving" fuses top-K
// extraction with vocabulary-wide logit normalisation. Here every logit is read
// from HBM exactly once:
//   * grid = (splits, rows): each CTA streams one contiguous chunk of one row with
//     16-byte loads in batches of 4 per thread, the next batch's loads in flight while
//     the current one is reduced;
//   * every thread keeps an online (max, sum exp) pair, merged by warp shuffles;
//   * candidates are order-preserving 64-bit keys (value, then lower id first). Each
//     warp appends the elements that reach its value bound to a key buffer in shared
//     memory (a ballot for the slots). The hot loop costs one compare per batch: a warp
//     looks at a batch only if some lane's batch maximum reaches the bound. The bound
//     is the largest of three lower bounds on the CTA's K-th value: the K-th largest of
//     the warp's 32 running lane maxima (each a distinct element; used until the buffer
//     holds K keys), the K-th key of the buffer (compacted by rank counting whenever it
//     holds 2K keys), and a CTA-wide bound in shared memory. Every warp publishes its
//     r-th largest lane maximum (r = ceil(K / warps)); the smallest of those has r
//     distinct elements at or above it in each of the warps, K in all, so it bounds the
//     CTA's K-th value from below while each warp alone has seen only a fraction of the
//     row;
//   * the arithmetic runs on packed pairs: the batch maxima on raw bf16x2 words, the
//     exponent arguments and the running sums as f32x2 (one instruction per two
//     logits), one ex2 per logit;
//   * the CTA merges its warps' lists by rank counting; with several splits per
//     row the last CTA to finish (atomic ticket, no waiting) merges the splits'
//     partial (max, sum, top-K) records and writes ids, logp and lse.
#include <mutex>

#include "internal.cuh"

namespace lilicorr {

namespace {

constexpr int TK_THREADS = 256;        // CTA size of the few-row plan and of the merges
constexpr int TK_THREADS_MANY = 128;   // CTA size when the rows alone fill the GPU
constexpr int TK_UNROLL = 4;           // 16-byte loads per thread per batch (many rows)
constexpr int TK_UNROLL_FEW = 8;       // ... when few rows are split over many CTAs
constexpr int TK_MAX_SPLITS = 64;
constexpr int TK_MERGE_MAX = 512;      // splits * K keys merged by the last CTA
constexpr int TK_FEW_ROW_CTAS = 256;   // CTAs over all rows when rows are few
constexpr float LOG2E = 1.4426950408889634f;
constexpr unsigned FULL = 0xffffffffu;

// order-preserving 32-bit image of a float (for atomicMax on a threshold)
__device__ __forceinline__ uint32_t ord32(float v) {
  const uint32_t b = __float_as_uint(v);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float unord32(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed fp32 pairs (one register pair, one instruction for both halves).
__device__ __forceinline__ uint64_t pack2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpack2(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.ftz.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.ftz.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// larger of two bf16 pairs, per half (exact; a NaN half yields the other operand's half)
__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Barrier of the NT threads of a CTA (named barrier 1; the same threads as
// __syncthreads).
template <int NT>
__device__ __forceinline__ void csync() {
  asm volatile("bar.sync 1, %0;" ::"n"(NT) : "memory");
}

// Rank counting: each key of keys[0..n) (distinct apart from zeros, which mean "empty")
// counts the keys larger than itself and, if that rank is below K, lands in out[rank].
// Run by `nthreads` threads with indices t; out[0..K) must be zeroed beforehand and
// must not alias keys; the caller synchronises before and after.
__device__ __forceinline__ void rank_place(const uint64_t* keys, int n, int K, uint64_t* out,
                                           int t, int nthreads) {
  for (int i = t; i < n; i += nthreads) {
    const uint64_t c = keys[i];
    if (c == 0ull) continue;
    int rank = 0;
    for (int j = 0; j < n; ++j) rank += keys[j] > c ? 1 : 0;
    if (rank < K) out[rank] = c;
  }
}

// K largest of groups[g][0..K) for g < ngroups (each group sorted descending, zeros =
// empty), CTA-wide. Every group's K-th key bounds the answer's K-th from below, so only
// keys >= the largest such bound survive; they are compacted and rank-counted.
// surv: scratch of TK_MERGE_MAX keys; out[0..K) receives the result. All NT reducing
// threads call.
template <int NT>
__device__ void cta_select(const uint64_t* groups, int ngroups, int stride, int K, uint64_t* surv,
                           int* s_count, uint64_t* s_bound, uint64_t* out) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (warp == 0) {
    uint64_t b = 0ull;
    for (int g = lane; g < ngroups; g += 32) {
      const uint64_t k = groups[(size_t)g * stride + K - 1];
      b = k > b ? k : b;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const uint64_t x = __shfl_xor_sync(FULL, b, o);
      b = x > b ? x : b;
    }
    if (lane == 0) { *s_bound = b; *s_count = 0; }
  }
  for (int i = tid; i < K; i += NT) out[i] = 0ull;
  csync<NT>();
  const uint64_t bound = *s_bound;
  for (int i = tid; i < ngroups * K; i += NT) {
    const uint64_t k = groups[(size_t)(i / K) * stride + i % K];
    if (k != 0ull && k >= bound) surv[atomicAdd(s_count, 1)] = k;
  }
  csync<NT>();
  rank_place(surv, *s_count, K, out, tid, NT);
  csync<NT>();
}

template <int N>
__device__ __forceinline__ float lse_update(float& m, float& s, const float (&x)[N], bool valid) {
  float vmax = x[0];
#pragma unroll
  for (int j = 1; j < N; ++j) vmax = fmaxf(vmax, x[j]);
  if (!valid) return -INFINITY;
  if (vmax > m) {
    s *= ex2((m - vmax) * LOG2E);
    m = vmax;
  }
  if (m == -INFINITY) return vmax;
  const float ml = m * LOG2E;
  float acc[N];
#pragma unroll
  for (int j = 0; j < N; ++j) acc[j] = ex2(fmaf(x[j], LOG2E, -ml));
#pragma unroll
  for (int w = 1; w < N; w <<= 1)
#pragma unroll
    for (int j = 0; j + w < N; j += 2 * w) acc[j] += acc[j + w];
  s += acc[0];
  return vmax;
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
  // largest of the 8 values (NaN ignored), on the packed words
  __device__ static float vmax(const uint4& v) {
    const uint32_t m = max_bf16x2(max_bf16x2(v.x, v.y), max_bf16x2(v.z, v.w));
    return fmaxf(__uint_as_float(m << 16), __uint_as_float(m & 0xFFFF0000u));
  }
  static constexpr uint32_t NEG_INF4 = 0xFF80FF80u;       // two bf16 -inf
};
template <> struct Vec<float> {
  static constexpr int N = 4;
  __device__ static void unpack(const uint4& v, float (&x)[4]) {
    x[0] = __uint_as_float(v.x); x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z); x[3] = __uint_as_float(v.w);
  }
  __device__ static float scalar(const float* p, size_t i) { return p[i]; }
  __device__ static float vmax(const uint4& v) {
    return fmaxf(fmaxf(__uint_as_float(v.x), __uint_as_float(v.y)),
                 fmaxf(__uint_as_float(v.z), __uint_as_float(v.w)));
  }
  static constexpr uint32_t NEG_INF4 = 0xFF800000u;       // fp32 -inf
};

// K-th largest (K <= 32) of one value per lane, by a bitonic sort across the warp.
__device__ __forceinline__ float warp_kth_largest(float v, int K, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const float o = __shfl_xor_sync(FULL, v, stride);
      const bool lower = (lane & stride) == 0, desc = (lane & size) == 0;
      v = (lower == desc) ? fmaxf(v, o) : fminf(v, o);
    }
  return __shfl_sync(FULL, v, K - 1);
}

// r-th largest (1 <= r <= 32) of one value per lane, in the order of ord32 (-0 below +0):
// rounds of a warp-wide maximum over the lanes not yet taken, equal values counted at once
// (at most r rounds; every float's image is above 0, which marks a lane as taken). Cheaper
// than the sorting network for small r (4096 rows of 151,936 at K = 16: 237.6 -> 224.0 us).
__device__ __forceinline__ float warp_rth_largest(float v, int r) {
  uint32_t in = ord32(v);
  for (;;) {
    const uint32_t mx = __reduce_max_sync(FULL, in);
    r -= __popc(__ballot_sync(FULL, in == mx));
    if (r <= 0) return unord32(mx);
    if (in == mx) in = 0u;
  }
}

// A warp's candidates: keys appended to a shared-memory buffer, plus a value bound
// below which no element can be in the CTA's top-K. The bound is the larger of
//   * the K-th largest running maximum over the warp's lanes (each lane's running maximum
//     is a distinct element, so K elements reach it), and
//   * the K-th key of the buffer after a compaction, and the CTA-wide bound (the largest
//     bound any warp of the CTA has published, and the smallest of the warps' published
//     r-th largest lane maxima).
// Appending costs a ballot and a store; the buffer is compacted to its K largest keys by
// rank counting once it holds 2K keys (or when it would overflow).
constexpr int TK_CAP = 96;

// Every warp meets its elements in increasing id order (its share of each batch lies
// above its share of the batch before; the split kernel's scalar head comes first and its
// tail last). So once the buffer holds K keys, a later element whose value equals the
// K-th key's loses that tie, and the warp's own filter may sit just above that value:
// then a run of equal values costs one compaction, not one append per element. Other
// warps meet elements on both sides of this warp's ids, so what the warp publishes (to
// the CTA-wide bound and to the final selection) is the plain bound, publish_bound().
struct WarpCand {
  uint64_t* buf;       // [TK_CAP] in shared memory
  uint64_t* tmp;       // [LILICORR_MAX_K] scratch of the compaction; tmp[K - 1] holds the
                       // K-th key of the last compaction (0: none yet)
  int n;               // keys in buf (warp-uniform)
  float thr;           // the warp's filter (warp-uniform, never decreases)
};

// Smallest float above v (+inf stays +inf).
__device__ __forceinline__ float next_up(float v) {
  if (v == 0.f) return __uint_as_float(1u);
  const uint32_t b = __float_as_uint(v);
  if (b == 0x7F800000u) return v;
  return __uint_as_float((b & 0x80000000u) ? b - 1u : b + 1u);
}

// The warp's bound without the tie step: a value no element of the CTA's top-K lies below.
__device__ __forceinline__ float publish_bound(const WarpCand& w, int K) {
  const uint64_t kth = w.tmp[K - 1];
  if (kth == 0ull) return w.thr;
  const float kv = key_value(kth);
  return w.thr == next_up(kv) ? kv : w.thr;
}

__device__ __forceinline__ void warp_compact(WarpCand& w, int K, int lane) {
  __syncwarp();
  if (lane < K) w.tmp[lane] = 0ull;
  __syncwarp();
  for (int i = lane; i < w.n; i += 32) {
    const uint64_t c = w.buf[i];
    int rank = 0;
    for (int j = 0; j < w.n; ++j) rank += w.buf[j] > c ? 1 : 0;
    if (rank < K) w.tmp[rank] = c;
  }
  __syncwarp();
  const uint64_t mine = lane < K ? w.tmp[lane] : 0ull;
  const uint64_t kth = w.tmp[K - 1];
  __syncwarp();
  if (lane < K) w.buf[lane] = mine;
  w.n = min(w.n, K);
  if (kth) {
    const float kv = key_value(kth);
    if (w.thr <= kv) w.thr = next_up(kv);      // equal values to come lose the tie
  }
  __syncwarp();
}

// This lane's hot values among x[0..N) (ids id0 + j), exactly: at or above the plain bound
// and with a key above the buffer's K-th key (a value equal to that key's needs a lower
// id). For the rest of a vector after a compaction in its middle, whose lanes hold ids on
// both sides of the new K-th key.
template <int N>
__device__ __forceinline__ uint32_t hot_mask_exact(const WarpCand& w, const float (&x)[N],
                                                   uint32_t id0, bool valid, int K) {
  const uint64_t kth = w.tmp[K - 1];
  const float kv = key_value(kth);                // NaN for kth == 0: no tie to break
  const uint32_t kid = (uint32_t)key_id(kth);
  const float lo = publish_bound(w, K);
  uint32_t hm = 0u;
#pragma unroll
  for (int j = 0; j < N; ++j)
    hm |= (valid && x[j] >= lo && (x[j] != kv || id0 + (uint32_t)j < kid)) ? (1u << j) : 0u;
  return hm;
}

// Append this lane's values that reach the filter. Warp-collective: one ballot round per
// hot element of the busiest lane.
template <int N>
__device__ __forceinline__ void warp_append(WarpCand& w, const float (&x)[N], uint32_t id0,
                                            bool valid, int K, int lane) {
  uint32_t hm = 0u;
#pragma unroll
  for (int j = 0; j < N; ++j) hm |= (valid && x[j] >= w.thr) ? (1u << j) : 0u;
  while (__any_sync(FULL, hm != 0u)) {
    if (w.n + 32 > TK_CAP) {
      warp_compact(w, K, lane);
      hm &= hot_mask_exact<N>(w, x, id0, valid, K);
      if (!__any_sync(FULL, hm != 0u)) break;
    }
    const bool has = hm != 0u;
    const int j = has ? __ffs(hm) - 1 : 0;
    hm &= hm - 1u;
    float xv = x[0];
#pragma unroll
    for (int t = 1; t < N; ++t) xv = (j == t) ? x[t] : xv;
    const unsigned mk = __ballot_sync(FULL, has);
    if (has) w.buf[w.n + __popc(mk & ((1u << lane) - 1u))] = make_key(xv, id0 + (uint32_t)j);
    w.n += __popc(mk);
  }
}

// A batch: U 16-byte vectors per thread (vectors it + u*NT + tid, NT threads).
// CHECK = false: every vector is inside the chunk (no predicates); otherwise vectors past
// v_end read as -inf, which adds nothing to the sum and never becomes a candidate (the
// reduction below also skips vectors outside [v_lo, v_end) as candidates).
template <typename T, int NT, int U, bool CHECK>
__device__ __forceinline__ void load_batch(const uint4* __restrict__ vp, int it, int v_end, int tid,
                                           uint4 (&raw)[U]) {
  constexpr uint32_t NI = Vec<T>::NEG_INF4;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int v = it + u * NT + tid;
    raw[u] = (!CHECK || v < v_end) ? __ldcs(vp + v) : make_uint4(NI, NI, NI, NI);
  }
}

// The sum of exp(x - m) over one 16-byte vector, added into two packed accumulators (the
// values are unpacked pair by pair, so the raw words stay the only copy in registers).
template <typename T>
__device__ __forceinline__ void exp_vec(const uint4& r, uint64_t l2, uint64_t nm, uint64_t& a0,
                                        uint64_t& a1) {
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
  if constexpr (sizeof(T) == 2) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float t0, t1;
      unpack2(fma2(pack2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xFFFF0000u)), l2, nm),
              t0, t1);
      const uint64_t e = pack2(ex2(t0), ex2(t1));
      if (i & 1) a1 = add2(a1, e); else a0 = add2(a0, e);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; i += 2) {
      float t0, t1;
      unpack2(fma2(pack2(__uint_as_float(w[i]), __uint_as_float(w[i + 1])), l2, nm), t0, t1);
      const uint64_t e = pack2(ex2(t0), ex2(t1));
      if ((i >> 1) & 1) a1 = add2(a1, e); else a0 = add2(a0, e);
    }
  }
}

// Reduce one loaded batch: the online (max, sum exp) with one rescale check per batch, then
// the candidates, which the warp looks at only if some lane's batch maximum reaches the
// bound. s_wtop[warp]: the warps' published r-th largest lane maxima (r = ceil(K / warps)).
template <typename T, int NT, int U, bool CHECK>
__device__ __forceinline__ void process_batch(const uint4 (&raw)[U], int it, int v_lo,
                                              int v_end, uint32_t id_base, int K, int tid, int lane,
                                              float& m, float& s, WarpCand& w,
                                              uint32_t* s_cta_thr, float* s_wtop) {
  constexpr int VEC = Vec<T>::N;
  float vmx[U];
  float bmax = -INFINITY;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    vmx[u] = Vec<T>::vmax(raw[u]);
    bmax = fmaxf(bmax, vmx[u]);
  }
  // online log-sum-exp, one rescale per batch (rarely taken after the first batches)
  if (bmax > m) {
    s *= ex2((m - bmax) * LOG2E);
    m = bmax;
  }
  if (m != -INFINITY) {
    const float ml = m * LOG2E;
    const uint64_t l2 = pack2(LOG2E, LOG2E), nm = pack2(-ml, -ml);
    uint64_t a0 = pack2(0.f, 0.f), a1 = a0;
#pragma unroll
    for (int u = 0; u < U; ++u) exp_vec<T>(raw[u], l2, nm, a0, a1);
    float p0, p1, p2, p3;
    unpack2(a0, p0, p1);
    unpack2(a1, p2, p3);
    s += (p0 + p1) + (p2 + p3);
  }
  // candidates: only when some lane's batch maximum reaches the current filter
  w.thr = fmaxf(w.thr, unord32(*(volatile uint32_t*)s_cta_thr));
  if (!__any_sync(FULL, bmax >= w.thr)) return;
  {
    // the CTA-wide bound from the warps' published lane maxima
    constexpr int NW = NT / 32;
    const int r = (K + NW - 1) / NW;
    const float mine = warp_rth_largest(m, r);
    volatile float* wtop = s_wtop;
    if (lane == 0) wtop[tid >> 5] = mine;             // lane maxima only grow
    __syncwarp();
    float cb = INFINITY;
#pragma unroll
    for (int i = 0; i < NW; ++i) cb = fminf(cb, wtop[i]);
    if (cb > w.thr) {
      w.thr = cb;
      if (lane == 0) atomicMax(s_cta_thr, ord32(cb));
    }
  }
  if (!__any_sync(FULL, bmax >= w.thr)) return;
  if (w.n < K) {
    // until the buffer holds K keys: the K-th largest running lane maximum
    const float tb = warp_kth_largest(m, K, lane);
    if (tb > w.thr) {
      w.thr = tb;
      if (lane == 0) atomicMax(s_cta_thr, ord32(tb));
    }
  }
#pragma unroll
  for (int u = 0; u < U; ++u) {
    if (!__any_sync(FULL, vmx[u] >= w.thr)) continue;
    const int v = it + u * NT + tid;
    float x[VEC];
    Vec<T>::unpack(raw[u], x);
    warp_append<VEC>(w, x, id_base + (uint32_t)(v * VEC), !CHECK || (v >= v_lo && v < v_end), K,
                     lane);
  }
  if (w.n >= 2 * K) {                                  // the buffer's K-th key bounds it
    warp_compact(w, K, lane);
    if (lane == 0) atomicMax(s_cta_thr, ord32(publish_bound(w, K)));
  }
}

// Stream vectors [v_begin, v_end) through process_batch with the next batch's loads in
// flight while the current one is reduced; full batches in the loop, the ragged last one
// after it.
template <typename T, int NT, int U>
__device__ __forceinline__ void stream_chunk(const uint4* __restrict__ vp, int v_begin, int v_end,
                                             uint32_t id_base, int K, int tid, int lane, float& m,
                                             float& s, WarpCand& w, uint32_t* s_cta_thr,
                                             float* s_wtop) {
  constexpr int STEP = U * NT;
  const int full_end = v_begin + (v_end - v_begin) / STEP * STEP;
  uint4 cur[U], nxt[U];
  if (v_begin < full_end) load_batch<T, NT, U, false>(vp, v_begin, v_end, tid, cur);
#pragma unroll 1
  for (int it = v_begin; it < full_end; it += STEP) {
    if (it + STEP < full_end) load_batch<T, NT, U, false>(vp, it + STEP, v_end, tid, nxt);
    process_batch<T, NT, U, false>(cur, it, it, v_end, id_base, K, tid, lane, m, s, w, s_cta_thr,
                                   s_wtop);
#pragma unroll
    for (int u = 0; u < U; ++u) cur[u] = nxt[u];
  }
  if (full_end < v_end) {
    load_batch<T, NT, U, true>(vp, full_end, v_end, tid, cur);
    process_batch<T, NT, U, true>(cur, full_end, full_end, v_end, id_base, K, tid, lane, m, s, w,
                                  s_cta_thr, s_wtop);
  }
}

// Elements [e_begin, e_end) of row rp, one per lane (the few outside the 16-byte vectors).
template <typename T>
__device__ __forceinline__ void scalar_part(const T* rp, int e_begin, int e_end, int K, int lane,
                                            float& m, float& s, WarpCand& w) {
  for (int base = e_begin; base < e_end; base += 32) {
    const int e = base + lane;
    const bool valid = e < e_end;
    float x[1] = {valid ? Vec<T>::scalar(rp, e) : -INFINITY};
    lse_update<1>(m, s, x, valid);
    warp_append<1>(w, x, (uint32_t)(valid ? e : 0), valid, K, lane);
  }
}

struct Rec {            // partial record of one (row, split)
  float m, s;
  uint64_t keys[1];     // [K]
};

// Where a row's result goes: the final outputs (ids, logp, lse), or, for one vocabulary
// shard, the row's public partial record (running max, sum of exp below it, the shard's
// top-K values and ids with the shard's id offset added; empty entries -inf / -1).
struct PartialOut {
  unsigned char* rec;       // [rows][partial_bytes(K)], or null for the final outputs
  int32_t id_offset;
};

// Warp 0 of the CTA that completes row `row`: (m, s) of the row, its top-K keys in s_top.
__device__ __forceinline__ void write_row(int row, int K, float m, float s, const uint64_t* s_top,
                                          const PartialOut& pout, int32_t* ids, float* logp,
                                          float* lse, uint32_t* status, int lane) {
  if (pout.rec) {
    unsigned char* r = pout.rec + (size_t)row * topk_partial_bytes(K);
    float* rf = reinterpret_cast<float*>(r);
    int32_t* ri = reinterpret_cast<int32_t*>(r + 8 + 4 * (size_t)K);
    if (lane == 0) { rf[0] = m; rf[1] = s; }
    if (lane < K) {
      const uint64_t k = s_top[lane];
      rf[2 + lane] = k ? key_value(k) : -INFINITY;
      ri[lane] = k ? key_id(k) + pout.id_offset : -1;
    }
    return;
  }
  const float l = m + logf(s);
  if (lane == 0) {
    lse[row] = l;
    if (!isfinite(l)) set_status(status, LILICORR_ERR_NONFINITE);
  }
  if (lane < K) {
    const uint64_t k = s_top[lane];
    ids[(size_t)row * K + lane] = key_id(k);
    logp[(size_t)row * K + lane] = key_value(k) - l;
  }
}

// Shared memory of one CTA's row reduction.
template <int NW>
struct TkShared {
  uint64_t buf[NW][TK_CAP];             // the warps' candidates
  uint64_t tmp[NW][LILICORR_MAX_K];
  uint64_t keys[TK_MERGE_MAX];          // the pieces' lists (merging CTA)
  uint64_t merge[TK_MERGE_MAX];
  uint64_t top[LILICORR_MAX_K];
  uint64_t bound;
  float m[NW], s[NW];
  float wtop[NW];                       // the warps' r-th largest lane maxima
  uint32_t cta_thr;                     // CTA-wide value bound (order image)
  int last, count;
};

// Close this CTA's piece of row `row` (all NT reducing threads, same arguments): the
// piece's (max, sum exp) and top-K from the warps' states, then either the row's outputs
// (its only piece) or the piece's partial record and a ticket. The CTA that takes the
// row's last ticket (atomic, no waiting) merges the `npieces` records (row_recs,
// rec_bytes apart) and writes the row.
template <int NT>
__device__ void finish_piece(TkShared<NT / 32>& sh, WarpCand& w, float m, float s, int row, int K,
                             int npieces, int piece, unsigned char* row_recs, size_t rec_bytes,
                             uint32_t* counters, const PartialOut& pout, int32_t* ids,
                             float* logp, float* lse, uint32_t* status) {
  constexpr int NW = NT / 32;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // (max, sum) of the warp, then of the CTA
  const float wm = warp_max(m);
  float ws = (m == -INFINITY) ? 0.f : s * ex2((m - wm) * LOG2E);
  ws = warp_sum(ws);
  const float pb = publish_bound(w, K);
  if (lane == 0) {
    sh.m[warp] = wm;
    sh.s[warp] = ws;
    atomicMax(&sh.cta_thr, ord32(pb));
  }
  // CTA top-K: keys of every warp's buffer at or above the CTA-wide bound, rank-counted
  // (the bound never exceeds the CTA's K-th value, so the K largest keys all survive)
  if (tid == 0) sh.count = 0;
  for (int i = tid; i < LILICORR_MAX_K; i += NT) sh.top[i] = 0ull;
  csync<NT>();
  {
    const float bound = unord32(sh.cta_thr);
    const int nw = w.n;
    for (int i = lane; i < nw; i += 32) {
      const uint64_t k = w.buf[i];
      if (key_value(k) >= bound) {
        const int pos = atomicAdd(&sh.count, 1);
        if (pos < TK_MERGE_MAX) sh.merge[pos] = k;
      }
    }
  }
  csync<NT>();
  if (sh.count > TK_MERGE_MAX) {
    // more survivors than the merge area holds (only with massive ties at the bound):
    // compact every warp's buffer to its own top-K first, then merge those
    warp_compact(w, K, lane);
    if (lane < LILICORR_MAX_K) sh.keys[warp * LILICORR_MAX_K + lane] = lane < w.n ? w.buf[lane] : 0ull;
    csync<NT>();
    cta_select<NT>(sh.keys, NW, LILICORR_MAX_K, K, sh.merge, &sh.count, &sh.bound, sh.top);
  } else {
    rank_place(sh.merge, sh.count, K, sh.top, tid, NT);
    csync<NT>();
  }

  float cm = -INFINITY, cs = 0.f;
  if (warp == 0) {
    const float pm = lane < NW ? sh.m[lane] : -INFINITY;
    const float ps = lane < NW ? sh.s[lane] : 0.f;
    cm = warp_max(pm);
    cs = warp_sum(pm == -INFINITY ? 0.f : ps * ex2((pm - cm) * LOG2E));
  }
  if (npieces == 1) {
    if (warp == 0) write_row(row, K, cm, cs, sh.top, pout, ids, logp, lse, status, lane);
    return;
  }

  // publish this piece's record, then take a ticket
  Rec* rec = reinterpret_cast<Rec*>(row_recs + (size_t)piece * rec_bytes);
  if (warp == 0) {
    if (lane == 0) { rec->m = cm; rec->s = cs; }
    if (lane < K) rec->keys[lane] = sh.top[lane];
    __threadfence();
  }
  csync<NT>();
  if (tid == 0) {
    const uint32_t ticket = atomicAdd(&counters[row], 1u);
    sh.last = (ticket == (uint32_t)(npieces - 1));
  }
  csync<NT>();
  if (!sh.last) return;
  __threadfence();

  // last CTA of the row: merge all pieces (their lists staged in shared memory)
  const int n = npieces * K;
  for (int i = tid; i < n; i += NT) {
    const Rec* r = reinterpret_cast<const Rec*>(row_recs + (size_t)(i / K) * rec_bytes);
    sh.keys[i] = __ldcg(reinterpret_cast<const unsigned long long*>(&r->keys[i % K]));
  }
  csync<NT>();
  cta_select<NT>(sh.keys, npieces, K, K, sh.merge, &sh.count, &sh.bound, sh.top);
  if (warp == 0) {
    float pm = -INFINITY, ps = 0.f;
    for (int i = lane; i < npieces; i += 32) {
      const Rec* r = reinterpret_cast<const Rec*>(row_recs + (size_t)i * rec_bytes);
      const float rm = __ldcg(&r->m), rs = __ldcg(&r->s);
      if (rm == -INFINITY) continue;
      if (rm > pm) { ps = ps * ex2((pm - rm) * LOG2E) + rs; pm = rm; }
      else ps += rs * ex2((rm - pm) * LOG2E);
    }
    const float gm = warp_max(pm);
    const float gs = warp_sum(pm == -INFINITY ? 0.f : ps * ex2((pm - gm) * LOG2E));
    if (lane == 0) counters[row] = 0u;             // leave the workspace reusable
    write_row(row, K, gm, gs, sh.top, pout, ids, logp, lse, status, lane);
  }
}

// U vectors per thread per batch: 4 with up to 1024 / NT CTAs per SM (64 registers), 8 for
// the split plan of few rows (at most two CTAs per SM; more bytes in flight per thread).
template <typename T, int NT, int U>
__global__ void __launch_bounds__(NT, (U > 4 ? 512 : 1024) / NT)
topk_lse_kernel(const T* __restrict__ logits, int V, int K, int splits, int chunk_vecs,
                size_t rec_bytes, int32_t* __restrict__ ids, float* __restrict__ logp,
                float* __restrict__ lse, uint32_t* status, uint32_t* counters,
                unsigned char* partials, PartialOut pout) {
  pdl_wait();
  constexpr int VEC = Vec<T>::N;
  constexpr int NW = NT / 32;
  __shared__ TkShared<NW> sh;

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

  WarpCand w;
  w.buf = sh.buf[warp];
  w.tmp = sh.tmp[warp];
  w.n = 0;
  w.thr = -INFINITY;
  if (lane == 0) w.tmp[K - 1] = 0ull;
  if (tid == 0) sh.cta_thr = ord32(-INFINITY);
  if (tid < NW) sh.wtop[tid] = -INFINITY;
  __syncthreads();

  float m = -INFINITY, s = 0.f;

  // scalar head [0, e0), before the vectors, and scalar tail [e0 + nvec*VEC, V), after
  // them: warp 0 of split 0, one element per lane (so that warp meets its ids in order)
  const int tail0 = e0 + nvec * VEC;
  const bool scalars = split == 0 && warp == 0;
  if (scalars) scalar_part<T>(rp, 0, e0, K, lane, m, s, w);

  // main stream: batches of 16-byte vectors, the next one's loads in flight
  const uint4* vp = reinterpret_cast<const uint4*>(rp + e0);
  stream_chunk<T, NT, U>(vp, v_begin, v_end, (uint32_t)e0, K, tid, lane, m, s, w, &sh.cta_thr,
                         sh.wtop);
  if (scalars) scalar_part<T>(rp, tail0, V, K, lane, m, s, w);
  finish_piece<NT>(sh, w, m, s, row, K, splits, split,
                   partials + (size_t)row * splits * rec_bytes, rec_bytes, counters, pout, ids,
                   logp, lse, status);
}

// Merge of P vocabulary shards' partial records of one row (one CTA per row): the union
// of the shards' top-K lists holds the row's top-K, and (m, s) pairs combine as in the
// split merge above.
__global__ void __launch_bounds__(TK_THREADS)
topk_merge_kernel(const unsigned char* __restrict__ recs, int P, int rows, int K,
                  int32_t* __restrict__ ids, float* __restrict__ logp, float* __restrict__ lse,
                  uint32_t* status) {
  pdl_wait();
  extern __shared__ uint64_t s_dyn[];   // [P*K] keys, [P*K] survivors, then P (max, sum) pairs
  uint64_t* s_keys = s_dyn;
  uint64_t* s_merge = s_dyn + (size_t)P * K;
  float2* s_ms = reinterpret_cast<float2*>(s_dyn + 2 * (size_t)P * K);
  __shared__ uint64_t s_top[LILICORR_MAX_K];
  __shared__ int s_count;
  __shared__ uint64_t s_bound;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, row = blockIdx.x;
  const size_t rb = topk_partial_bytes(K);
  for (int i = tid; i < P * K; i += TK_THREADS) {
    const unsigned char* r = recs + ((size_t)(i / K) * rows + row) * rb;
    const float v = reinterpret_cast<const float*>(r)[2 + i % K];
    const int32_t id = reinterpret_cast<const int32_t*>(r + 8 + 4 * (size_t)K)[i % K];
    s_keys[i] = id < 0 ? 0ull : make_key(v, (uint32_t)id);
  }
  for (int p = tid; p < P; p += TK_THREADS) {     // the records' (max, sum), same pass
    const float* r = reinterpret_cast<const float*>(recs + ((size_t)p * rows + row) * rb);
    s_ms[p] = make_float2(r[0], r[1]);
  }
  __syncthreads();
  cta_select<TK_THREADS>(s_keys, P, K, K, s_merge, &s_count, &s_bound, s_top);
  if (warp == 0) {
    float pm = -INFINITY, ps = 0.f;
    for (int p = lane; p < P; p += 32) {
      const float rm = s_ms[p].x, rs = s_ms[p].y;
      if (rm == -INFINITY) continue;
      if (rm > pm) { ps = ps * ex2((pm - rm) * LOG2E) + rs; pm = rm; }
      else ps += rs * ex2((rm - pm) * LOG2E);
    }
    const float gm = warp_max(pm);
    const float gs = warp_sum(pm == -INFINITY ? 0.f : ps * ex2((pm - gm) * LOG2E));
    const PartialOut none{nullptr, 0};
    write_row(row, K, gm, gs, s_top, none, ids, logp, lse, status, lane);
  }
}

}  // namespace

TopkPlan topk_plan(int rows, int V, int K, lilicorr_dtype_t dt) {
  const int vec = dt == LILICORR_BF16 ? 8 : 4;
  const int nvec = V / vec;
  const int sms = num_sms();
  const int min_chunk = 256;                 // vectors (4 KB) per CTA at least
  int splits = 1, threads = TK_THREADS, unroll = TK_UNROLL;
  if (rows * 2 < sms * 4) {
    // Few rows (not filling half of the 4-per-SM slots): split each over about 256 CTAs of
    // 256 threads in all (a sweep over 16-256 rows of a 151,936-wide vocabulary put the
    // optimum at 192-256 CTAs: more pieces add partial records and merge work faster than
    // they shorten the stream).
    splits = ceil_div(TK_FEW_ROW_CTAS, rows);
    unroll = TK_UNROLL_FEW;       // 16 rows of 151,936: 11.3 -> 10.5 us
  } else if (rows >= 16 * sms) {
    // Many rows per SM: one CTA of 128 threads per row, up to 8 resident per SM, so each SM
    // always has rows in flight while others finish (4096 rows of 151,936: 233 us against
    // 256 us with 256-thread CTAs). Splitting rows never paid: every piece repeats the
    // candidate bound's warm-up and adds a merge (+30-40 % at 512-4096 rows).
    threads = TK_THREADS_MANY;
  }
  splits = max(1, min(splits, ceil_div(max(nvec, 1), min_chunk)));
  splits = min(splits, min(TK_MAX_SPLITS, TK_MERGE_MAX / K));
  TopkPlan p;
  p.splits = splits;
  p.threads = threads;
  p.unroll = unroll;
  p.chunk_vecs = ceil_div(max(nvec, 1), splits);
  p.pieces = splits;
  p.rec_bytes = align_up(8 + 8 * (size_t)K, 16);
  return p;
}

size_t topk_ws_bytes(int rows, int V, int K, lilicorr_dtype_t dt) {
  const TopkPlan p = topk_plan(rows, V, K, dt);
  return 256 + align_up((size_t)rows * 4, 256) + align_up((size_t)rows * p.pieces * p.rec_bytes, 256);
}

template <typename T>
lilicorr_status_t launch_plan(const TopkPlan& p, const T* x, int rows, int V, int K, int32_t* ids,
                              float* logp, float* lse, uint32_t* status, uint32_t* counters,
                              unsigned char* part, const PartialOut& pout, cudaStream_t st) {
  const dim3 grid(p.splits, rows);
  if (p.threads == TK_THREADS_MANY)
    return launch_k(topk_lse_kernel<T, TK_THREADS_MANY, TK_UNROLL>, grid, TK_THREADS_MANY, 0, st,
                    x, V, K, p.splits, p.chunk_vecs, p.rec_bytes, ids, logp, lse, status, counters,
                    part, pout);
  if (p.unroll == TK_UNROLL_FEW)
    return launch_k(topk_lse_kernel<T, TK_THREADS, TK_UNROLL_FEW>, grid, TK_THREADS, 0, st, x, V,
                    K, p.splits, p.chunk_vecs, p.rec_bytes, ids, logp, lse, status, counters, part,
                    pout);
  return launch_k(topk_lse_kernel<T, TK_THREADS, TK_UNROLL>, grid, TK_THREADS, 0, st, x, V, K,
                  p.splits, p.chunk_vecs, p.rec_bytes, ids, logp, lse, status, counters, part,
                  pout);
}

lilicorr_status_t launch_topk_lse(const void* logits, lilicorr_dtype_t dt, int rows, int V, int K,
                                  int32_t* ids, float* logp, float* lse, uint32_t* status,
                                  uint32_t* counters, void* partials, cudaStream_t st,
                                  void* partial_out, int32_t id_offset) {
  const PartialOut pout{static_cast<unsigned char*>(partial_out), id_offset};
  if (rows == 0) return LILICORR_OK;
  const TopkPlan p = topk_plan(rows, V, K, dt);
  unsigned char* part = static_cast<unsigned char*>(partials);
  if (dt == LILICORR_BF16)
    return launch_plan(p, static_cast<const uint16_t*>(logits), rows, V, K, ids, logp, lse, status,
                       counters, part, pout, st);
  return launch_plan(p, static_cast<const float*>(logits), rows, V, K, ids, logp, lse, status,
                     counters, part, pout, st);
}

lilicorr_status_t launch_topk_merge(const void* partials, int P, int rows, int K, int32_t* ids,
                                    float* logp, float* lse, uint32_t* status, cudaStream_t st) {
  if (rows == 0) return LILICORR_OK;
  if (P < 1 || K < 1 || P * K > TOPK_MERGE_KEYS_MAX) return LILICORR_ERR_SHAPE;
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(topk_merge_kernel, configured));
  LL_TRY(launch_k(topk_merge_kernel, rows, TK_THREADS,
                  2 * (size_t)P * K * sizeof(uint64_t) + (size_t)P * sizeof(float2), st,
                  static_cast<const unsigned char*>(partials), P, rows, K, ids, logp, lse, status));
  return LILICORR_OK;
}

}  // namespace lilicorr

// ----------------------------------------------------------------------------- no-allocation variant
// Scratch of lilicorr_topk_lse_noalloc: a fixed array in the library's device image, so
// the call needs no workspace from its caller. Every GPU that loads the library holds it
// until the process exits.
namespace lilicorr {
namespace {

constexpr size_t NOALLOC_SCRATCH_BYTES = 4u << 20;   // 4 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_SCRATCH_BYTES];

std::mutex g_noalloc_mutex;
void* g_noalloc_ptr[64] = {};

// Device address of the scratch on the current device. In host code the array's name
// stands for a host-side shadow, not a device address; cudaGetSymbolAddress (called once
// per device, with that device current) gives the address the kernel must receive.
lilicorr_status_t noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    (void)cudaGetLastError();
    return LILICORR_ERR_CUDA;
  }
  if (dev < 0 || dev >= 64) return LILICORR_ERR_ARG;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) {
      (void)cudaGetLastError();
      return LILICORR_ERR_CUDA;
    }
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return LILICORR_OK;
}

}  // namespace
}  // namespace lilicorr

extern "C" size_t lilicorr_topk_lse_noalloc_max_bytes(void) {
  return lilicorr::NOALLOC_SCRATCH_BYTES;
}

extern "C" lilicorr_status_t lilicorr_topk_lse_noalloc(const void* logits, lilicorr_dtype_t dtype,
                                                       int rows, int V, int K, int32_t* ids,
                                                       float* logp, float* lse,
                                                       cudaStream_t stream) {
  using namespace lilicorr;
  if (dtype != LILICORR_F32 && dtype != LILICORR_BF16) return LILICORR_ERR_DTYPE;
  if (rows < 0 || V <= 0 || K <= 0 || K > LILICORR_MAX_K || K > V) return LILICORR_ERR_SHAPE;
  if (rows == 0) return LILICORR_OK;
  if (!logits || !ids || !logp || !lse) return LILICORR_ERR_ARG;
  if (!aligned16(logits)) return LILICORR_ERR_ARG;
  if (topk_ws_bytes(rows, V, K, dtype) > NOALLOC_SCRATCH_BYTES) return LILICORR_ERR_WORKSPACE;
  void* ws = nullptr;
  LL_TRY(noalloc_scratch(&ws));
  unsigned char* w = static_cast<unsigned char*>(ws);
  // the status word and the per-row tickets must start at zero; the array keeps whatever
  // the previous call left, so clear them on the caller's stream first
  const size_t counters_bytes = align_up((size_t)rows * 4, 256);
  LL_CUDA_TRY(cudaMemsetAsync(w, 0, 256 + counters_bytes, stream));
  return launch_topk_lse(logits, dtype, rows, V, K, ids, logp, lse,
                         reinterpret_cast<uint32_t*>(w), reinterpret_cast<uint32_t*>(w + 256),
                         w + 256 + counters_bytes, stream);
}
