// Step (2), candidate-dependent part, on a thread-block cluster of four CTAs per sequence:
// the node features, the two-layer scoring Transformer, the fusion layer and the out / in
// heads (Sec. 3.2; App. A) for the bf16 head with D = 256, 8 heads, FFN 2D, L*K <= 128;
// optionally followed by steps (3) and (4) for the sequence (Eq. "pair", Sec. 3.5).
//
// The L*K nodes (zero-padded to 128) are the rows of every tensor-core tile, as in the
// one-CTA kernel (net_fused.cu), but the columns are split over the cluster: CTA c of the
// cluster owns columns 64c..64c+63 of the residual stream x (fp32, in its tensor memory),
// heads 2c, 2c+1 and FFN hidden units 128c..128c+127. Each product computes only the CTA's
// output slice:
//   conf2, W_o, W_2     x[:, slice] += A W[slice, :]^T            (N = 64)
//   q|k|v               the q, k, v rows of head pair c            (N = 192)
//   W_1                 FFN hidden units 128c..128c+127            (N = 128)
//   heads               o[:, 64c..64c+63] and i[:, 64c..64c+63]    (N = 128)
// while the fusion layer runs in full on every CTA (u is consumed locally by the heads).
// The operands that need every CTA's slice are all-gathered through distributed shared
// memory: each CTA writes its slice of the RMSNorm operand (before q|k|v and before W_1),
// of the attention output (before W_o), of the FFN hidden state (before W_2) and of the
// fusion input [xf | xf*t] into its own operand buffer, and one thread copies those bytes
// into the same place in the three peers with one bulk shared::cluster copy each, which
// completes the receiving CTA's mbarrier for that exchange; the receiving MMA lane waits
// on it (acquire, cluster scope). RMSNorm statistics (per-row sums of squares of each
// CTA's 64 columns) travel as st.async words to the same kind of barrier.
// Buffer reuse is ordered by the exchanges themselves: a CTA produces the next payload for
// a buffer only after an exchange that needs every CTA's contribution, which each CTA
// makes only once its own readers of that buffer are done (e.g. W_1's input lands in ACT
// after the second RMSNorm exchange, which needs the sender's W_o output, which needs this
// CTA's attention output, written after its attention finished reading q, k, v in ACT).
// The one exception, the hidden state that overwrites the peers' W_1 operand, waits for a
// word from every peer that its W_1 product is done (w1f).
// With the tail enabled, each CTA sums its 64 columns' part of every pair dot product and
// squared norm; the first CTA adds the peers' records (read across the cluster, in rank
// order), forms the cosine scores and runs the greedy walk.
//
// Roles (576 threads): warp 0 lane 0 streams the weight slices by TMA through a ring of
// eight 8 KB slots, warp 1 allocates tensor memory and walks the product schedule (lane 0
// issues tcgen05.mma), warps 2-17 are row
// workers (thread = row r = 32 (warp % 4) + lane and column group cg = (warp - 2) / 4:
// 16 columns of the x slice, or 64 columns of a full-width drain). Every mbarrier wait is
// bounded (about 2 s); on timeout the CTA records LILICORR_ERR_TIMEOUT, stops issuing and
// runs its remaining waits through (the other CTAs of the cluster then time out too).
#include <new>

#include "net_common.cuh"
#include "walk.cuh"

namespace lilicorr {

namespace {
using namespace tc;
using namespace net;

constexpr int NC_CC = 4;                  // CTAs per sequence
constexpr int NC_D = 256, NC_F = 512, NC_NH = 8, NC_HD = 32, NC_M = 128;
constexpr int NC_SL = NC_D / NC_CC;       // 64 columns of x per CTA
constexpr int NC_SLOTS = 8;               // weight ring: 8 slots of 64 rows x 64 k
constexpr int NC_MAX_LAYERS = 4;
constexpr int NC_MAX_L = 64;
constexpr int NC_RW = 512;                // row-worker threads
constexpr int NC_THREADS = 64 + NC_RW;
constexpr uint32_t NC_SLOT = 64 * 128;
constexpr uint32_t NC_TMEM = 512;
constexpr uint32_t X_COL = 0, SCR_COL = 256;
constexpr long long NC_WAIT = 4000000000ll;
constexpr float NC_LOG2E = 1.4426950408889634f;
constexpr float NC_RMS_EPS = 1e-6f;
constexpr uint32_t QKV_SET = 3 * 8192;    // q, k, v of one head

// shared memory (offsets from the 1024-aligned base)
constexpr uint32_t OFF_RING = 0;
constexpr uint32_t OFF_ACT = OFF_RING + NC_SLOTS * NC_SLOT;        // 4 chunks
constexpr uint32_t OFF_HF = OFF_ACT + 4 * CHUNK;                   // 4 chunks
constexpr uint32_t OFF_VEC = OFF_HF + 4 * CHUNK;
constexpr int V_AN = 0, V_FN = 64, V_BO = 128, V_B2 = 192, V_FIN = 320, V_C2B = 384, V_T = 448,
              V_B1 = 512, V_BQKV = 1024, V_C1W = 1792, V_C1B = 3072, V_CB = 3328,
              V_BOI = 3584, V_ANC = 3712, V_TF = 3776, V_END = 4032;
constexpr uint32_t OFF_SS = OFF_VEC + V_END * 4;                   // [4][128] local partials
// [2][4][128] the cluster's partials: [0] for the first RMSNorm of a layer and the final
// one, [1] for the second (a peer can send the next statistics before this CTA has read
// the previous ones, never before it read the ones two exchanges back)
constexpr uint32_t OFF_SSX = OFF_SS + 4 * NC_M * 4;
constexpr uint32_t OFF_DIST = OFF_SSX + 2 * NC_CC * NC_M * 4;      // [8][127]
constexpr uint32_t OFF_SAME = OFF_DIST + NC_NH * (2 * NC_MAX_L - 1) * 4;
constexpr uint32_t OFF_SLOT = OFF_SAME + NC_NH * 4;                // [128]
constexpr uint32_t OFF_IDS = OFF_SLOT + NC_M;                      // [128]
constexpr uint32_t OFF_BAR = (OFF_IDS + NC_M * 4 + 63) & ~63u;
constexpr int N_DONE = 2 + 4 * NC_MAX_LAYERS + 1, N_READY = N_DONE, N_XG = 3 + 6 * NC_MAX_LAYERS;
constexpr int X_C1 = N_XG - 1;            // exchange of the confidence MLP's first layer
constexpr int N_W1F = NC_MAX_LAYERS;
constexpr uint32_t NC_SMEM_USED = OFF_BAR + (2 * NC_SLOTS + N_DONE + N_READY + N_XG + N_W1F + 1) * 8;
constexpr size_t NC_SMEM = 1024 + NC_SMEM_USED;
static_assert(NC_SMEM <= 227 * 1024, "shared memory of the cluster network kernel");
static_assert(OFF_ACT % 1024 == 0 && OFF_HF % 1024 == 0, "swizzle atoms");

// bytes a CTA receives from its three peers per exchange
constexpr uint32_t XB_SS = (NC_CC - 1) * NC_M * 4;
constexpr uint32_t XB_SLICE = (NC_CC - 1) * NC_M * NC_SL * 2;
constexpr uint32_t XB_H = (NC_CC - 1) * NC_M * (NC_F / NC_CC) * 2;   // 128 hidden units each

enum { G_CONF2, G_QKV, G_WO, G_W1, G_W2, G_FUSE, G_WOI };

// events: MMA -> row workers (done), row workers -> MMA (ready, 16 warp arrivals),
// exchanges (xg: the peers' bytes) and the hand-shake of the FFN hidden state (w1f: the
// three peers' W_1 products are done, so their ACT buffers may be overwritten). One
// sequence per cluster: every event completes once.
__device__ __forceinline__ int lb(int l) { return 1 + 4 * l; }
__device__ __forceinline__ int xb(int l) { return 6 * l; }
// done
__device__ __forceinline__ int D_QKV(int l) { return lb(l); }
__device__ __forceinline__ int D_WO(int l) { return lb(l) + 1; }
__device__ __forceinline__ int D_W1(int l) { return lb(l) + 2; }
__device__ __forceinline__ int D_LAYER(int l) { return lb(l) + 3; }
// ready
__device__ __forceinline__ int R_XN(int l) { return lb(l); }
__device__ __forceinline__ int R_ATT(int l) { return lb(l) + 1; }
__device__ __forceinline__ int R_XN2(int l) { return lb(l) + 2; }
__device__ __forceinline__ int R_H(int l) { return lb(l) + 3; }
// exchanges
__device__ __forceinline__ int X_SS(int l) { return xb(l); }
__device__ __forceinline__ int X_XN(int l) { return xb(l) + 1; }
__device__ __forceinline__ int X_ATT(int l) { return xb(l) + 2; }
__device__ __forceinline__ int X_SS2(int l) { return xb(l) + 3; }
__device__ __forceinline__ int X_XN2(int l) { return xb(l) + 4; }
__device__ __forceinline__ int X_H(int l) { return xb(l) + 5; }

struct ClusterMaps {
  CUtensorMap conf2, fuse, woi;
  CUtensorMap wqkv[NC_MAX_LAYERS], wo[NC_MAX_LAYERS], w1[NC_MAX_LAYERS], w2[NC_MAX_LAYERS];
};

struct ClusterArgs {
  int B, L, K, LK, V, n_layers, d2;
  const int32_t* ids;
  const float* logp;
  const float* hproj;       // [B*L, D]
  const float* t;           // [B, D]
  const float* cb;          // [B, D]: t block of the fusion layer plus its bias
  const float* fold;        // [V, D]
  const float *slot, *rank, *conf1_w, *conf1_b, *conf2_b;
  const float* bqkv[NC_MAX_LAYERS];
  const float* bo[NC_MAX_LAYERS];
  const float* b1[NC_MAX_LAYERS];
  const float* b2[NC_MAX_LAYERS];
  const float* an[NC_MAX_LAYERS];
  const float* fn[NC_MAX_LAYERS];
  const float* dist[NC_MAX_LAYERS];
  const float* same[NC_MAX_LAYERS];
  const float* final_norm;
  const float* boi;
  float* oi;                // [B*LK, d2]
  uint32_t* status;
  int tail;                 // the pair scores and the greedy walk in the kernel's tail
  ClusterTail tl;
};

// K chunks and weight rows per chunk of each product slice
__device__ __forceinline__ int n_chunks(int kind) {
  return (kind == G_W2 || kind == G_FUSE) ? 8 : 4;
}
__device__ __forceinline__ int tile_rows(int kind) {
  switch (kind) {
    case G_QKV: return 192;
    case G_FUSE: return 256;
    case G_W1: case G_WOI: return 128;
    default: return NC_SL;
  }
}

__device__ __forceinline__ void load_chunk(const ClusterMaps& m, int kind, int l, int h, int kc,
                                           int me, void* dst, uint64_t* bar) {
  switch (kind) {
    case G_CONF2: tma_load_3d(dst, &m.conf2, bar, 0, NC_SL * me, kc); break;
    case G_QKV: tma_load_5d(dst, &m.wqkv[l], bar, 0, 0, me, 0, kc); break;
    case G_WO: tma_load_3d(dst, &m.wo[l], bar, 0, NC_SL * me, kc); break;
    case G_W1: tma_load_3d(dst, &m.w1[l], bar, 0, 128 * me, kc); break;
    case G_W2: tma_load_3d(dst, &m.w2[l], bar, 0, NC_SL * me, kc); break;
    case G_FUSE: tma_load_3d(dst, &m.fuse, bar, 0, 0, kc); break;
    default:   // out rows 64me.. and in rows d + 64me.. of [W_o; W_i]: both halves of
               // this CTA's 64 columns of the out and in vectors
      tma_load_3d(dst, &m.woi, bar, 0, NC_SL * me, kc);
      tma_load_3d(static_cast<uint8_t*>(dst) + NC_SLOT, &m.woi, bar, 0, 4 * NC_SL + NC_SL * me, kc);
      break;
  }
}

template <class Op>
__device__ __forceinline__ void schedule(const ClusterArgs& a, Op& op) {
  op.gemm(G_CONF2, 0, 0);
  for (int l = 0; l < a.n_layers; ++l) {
    op.gemm(G_QKV, l, 0);
    op.gemm(G_WO, l, 0);
    op.gemm(G_W1, l, 0);
    op.gemm(G_W2, l, 0);
  }
  op.gemm(G_FUSE, 0, 0);
  op.gemm(G_WOI, 0, 0);
}

struct Shared {
  uint8_t* base;
  uint64_t *full, *empty, *done, *ready, *xg, *w1f, *prb;
  volatile int* abort;
};

__device__ __forceinline__ bool ev_wait(uint64_t* bar, volatile int* abort) {
  if (*abort) return false;
  if (!mbar_wait_sleep(bar, 0, NC_WAIT)) {
    *abort = 1;
    return false;
  }
  return true;
}
__device__ __forceinline__ bool xg_wait(uint64_t* bar, volatile int* abort) {
  if (*abort) return false;
  if (!mbar_wait_cluster_sleep(bar, 0, NC_WAIT)) {
    *abort = 1;
    return false;
  }
  return true;
}

// The weight ring: a K chunk of a product slice (64 rows per slot) sits in consecutive
// slots, starting over at slot 0 where it would run past the last one; producer and
// issuer walk the same schedule, so they skip the same slots. Each slot has its own
// phase (bit `slot` of a mask): full is armed on a chunk's first slot, empty is signalled
// for every slot of it.
__device__ __forceinline__ int ring_place(uint32_t& pos, int slots) {
  int first = (int)(pos % NC_SLOTS);
  if (first + slots > NC_SLOTS) {
    pos += NC_SLOTS - first;
    first = 0;
  }
  pos += slots;
  return first;
}

struct Producer {
  const ClusterMaps* m;
  Shared sh;
  int me;
  uint32_t pos, ph;
  __device__ void gemm(int kind, int l, int h) {
    const int nk = n_chunks(kind), ns = tile_rows(kind) / 64;
    const uint32_t bytes = (uint32_t)tile_rows(kind) * 128u;
    for (int kc = 0; kc < nk; ++kc) {
      const int s0 = ring_place(pos, ns);
      for (int i = s0; i < s0 + ns; ++i) {
        if (!mbar_wait(&sh.empty[i], ((ph >> i) & 1u) ^ 1u, NC_WAIT)) *sh.abort = 1;
        ph ^= 1u << i;
      }
      if (*sh.abort) continue;
      mbar_expect_tx(&sh.full[s0], bytes);
      load_chunk(*m, kind, l, h, kc, me, sh.base + OFF_RING + (size_t)s0 * NC_SLOT, &sh.full[s0]);
    }
  }
};

struct Issuer {
  const ClusterArgs* a;
  Shared sh;
  uint32_t pos, ph, tmem;
  __device__ void gemm(int kind, int l, int h) {
    const int nl = a->n_layers;
    // what the product waits for: the row workers' part, and for gathered operands the
    // peers' slices
    int rd = -1, xw = -1, dn = -1;
    switch (kind) {
      case G_CONF2: rd = 0; xw = X_C1; dn = 0; break;
      case G_QKV: rd = R_XN(l); xw = X_XN(l); dn = D_QKV(l); break;
      case G_WO: rd = R_ATT(l); xw = X_ATT(l); dn = D_WO(l); break;
      case G_W1: rd = R_XN2(l); xw = X_XN2(l); dn = D_W1(l); break;
      case G_W2: rd = R_H(l); xw = X_H(l); dn = D_LAYER(l); break;
      case G_FUSE: rd = lb(nl); xw = xb(nl) + 1; dn = lb(nl); break;
      default: rd = lb(nl) + 1; dn = lb(nl) + 1; break;
    }
    const bool lead = (threadIdx.x & 31) == 0;     // the lane that issues and commits
    ev_wait(&sh.ready[rd], sh.abort);
    if (xw >= 0) xg_wait(&sh.xg[xw], sh.abort);
    __syncwarp();
    tc_fence_after();
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // peers' copied data
    const int nk = n_chunks(kind), ns = tile_rows(kind) / 64;
    const bool onto_x = kind == G_CONF2 || kind == G_WO || kind == G_W2;
    const uint32_t d = tmem + (onto_x ? X_COL : SCR_COL);
    const uint32_t idesc = instr_desc(128, tile_rows(kind));
    for (int kc = 0; kc < nk; ++kc) {
      uint32_t a_off;                               // the A operand's K chunk
      switch (kind) {
        case G_WO: a_off = OFF_HF + kc * CHUNK; break;                  // attention output
        case G_W2: a_off = kc < 4 ? OFF_HF + kc * CHUNK : OFF_ACT + (kc - 4) * CHUNK; break;
        case G_FUSE: a_off = kc < 4 ? OFF_ACT + kc * CHUNK : OFF_HF + (kc - 4) * CHUNK; break;
        default: a_off = OFF_ACT + kc * CHUNK; break;
      }
      const int s0 = ring_place(pos, ns);
      const uint32_t par = (ph >> s0) & 1u;
      ph ^= 1u << s0;
      const bool full = ev_wait_full(s0, par);
      __syncwarp();
      if (!full) continue;
      tc_fence_after();
      const uint64_t ad = smem_desc(sh.base + a_off);
      const uint64_t bd = smem_desc(sh.base + OFF_RING + (size_t)s0 * NC_SLOT);
      if (lead) {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_bf16(d, ad + 2ull * k, bd + 2ull * k, idesc, (onto_x || kc > 0 || k > 0) ? 1u : 0u);
        for (int i = s0; i < s0 + ns; ++i) mma_commit(&sh.empty[i]);
      }
      __syncwarp();
    }
    if (!*sh.abort && lead) mma_commit(&sh.done[dn]);
    __syncwarp();
  }
  __device__ bool ev_wait_full(int s, uint32_t ph) {
    if (*sh.abort) return false;
    if (!mbar_wait(&sh.full[s], ph, NC_WAIT)) {
      *sh.abort = 1;
      return false;
    }
    return true;
  }
};

__device__ __forceinline__ void rw_bar() { named_bar(1, NC_RW); }
__device__ __forceinline__ void set_bar(int set) { named_bar(2 + set, NC_RW / 2); }

// One warp's arrival on a row-worker -> MMA event, after its shared-memory writes
// (generic proxy, read by the tensor cores through the async proxy) and tensor-memory
// stores.
__device__ __forceinline__ void rw_signal(uint64_t* bar, int lane) {
  fence_async_shared();
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(bar);
}

// Shared-memory addresses of this CTA's three peers: the peer q-th after this CTA in the
// cluster holds offset o of its shared memory at base[q - 1] + o (mapa is linear).
struct Peers {
  uint32_t local, base[NC_CC - 1];
  __device__ uint32_t at(int q, const void* p) const {
    return base[q - 1] + (smem_u32(p) - local);
  }
};

// 16 values (row r, columns 16cg.. of this CTA's slice) as bf16 into chunk `me` of an
// operand buffer (two 16-byte pieces).
__device__ __forceinline__ void put16(uint8_t* buf, int me, int r, int cg, const float (&v)[16]) {
  uint8_t* ch = buf + (size_t)me * CHUNK;
#pragma unroll
  for (int p = 0; p < 2; ++p) *reinterpret_cast<uint4*>(ch + swz(r, 2 * cg + p)) = pack8(v + 8 * p);
}
// After every row worker wrote its part of `bytes` at src here: the same bytes into the
// same place in the three peers by the bulk-copy engine, counted on their exchange barrier
// `xbar` (one thread issues; it waits until the source has been read).
__device__ __forceinline__ void send_all(const void* src, uint32_t bytes, uint64_t* xbar, int tid,
                                         const Peers& pe) {
  fence_async_shared();
  rw_bar();
  if (tid == 0) {
#pragma unroll
    for (int q = 1; q < NC_CC; ++q) bulk_to_peer(pe.at(q, src), src, bytes, pe.at(q, xbar));
    bulk_wait_read();
  }
}

// A pre-norm RMSNorm feeding a product: RMSNorm(x) diag(g) W^T = diag(r) (x diag(g)) W^T
// with r the rows' 1 / rms, so the operand is x * g (bf16; the rounding is relative, as
// for the normalised value) and each row's r is applied in the drain of the product's
// accumulator. The operand therefore does not wait for the statistics — except where the
// peers' operand buffer may still be read by their previous product (the first RMSNorm of
// a layer and the final one write into buffers W_2 reads): there the statistics exchange,
// which needs every CTA's finished x, goes first and doubles as the hand-shake.
// norm_stats: this thread's 16 columns of x (+ bias, written back to tensor memory when
// write_back) into v, and the CTA's 64-column sum of squares of each row to every CTA
// (exchange `xss`).
__device__ void norm_stats(uint32_t tx, const float* bias, bool write_back, int cg, int r, int me,
                           float* s_ss, float* s_ssx, uint64_t* xss, const Peers& pe,
                           float (&v)[16]) {
  ld16f(tx + 16 * cg, v);
  float ss = 0.f;
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    if (bias) v[e] += bias[16 * cg + e];
    ss = fmaf(v[e], v[e], ss);
  }
  if (bias && write_back) {
    st16f(tx + 16 * cg, v);
    tmem_wait_st();
  }
  s_ss[cg * NC_M + r] = ss;
  rw_bar();
  if (cg == 0) {
    const float part = (s_ss[r] + s_ss[NC_M + r]) + (s_ss[2 * NC_M + r] + s_ss[3 * NC_M + r]);
    float* dst = s_ssx + me * NC_M + r;
    *dst = part;
#pragma unroll
    for (int q = 1; q < NC_CC; ++q) st_peer4(pe.at(q, dst), __float_as_uint(part), pe.at(q, xss));
  }
}
// norm_operand: v * gain into chunk me of `buf`, here and in the peers (exchange `xop`).
__device__ void norm_operand(float (&v)[16], const float* gain, uint8_t* buf, uint64_t* xop,
                             int cg, int r, int me, int tid, const Peers& pe) {
#pragma unroll
  for (int e = 0; e < 16; ++e) v[e] *= gain[16 * cg + e];
  put16(buf, me, r, cg, v);
  send_all(buf + (size_t)me * CHUNK, CHUNK, xop, tid, pe);
}
// norm_recv: 1 / rms of row r over the 256 columns, once every CTA's partial is here.
// A rw_bar separates it from the next norm_stats, which rewrites s_ss / s_ssx.
__device__ float norm_recv(int r, float* s_ssx, uint64_t* xss, volatile int* abort) {
  xg_wait(xss, abort);
  rw_bar();                                  // the local partial
  const float tot = (s_ssx[r] + s_ssx[NC_M + r]) + (s_ssx[2 * NC_M + r] + s_ssx[3 * NC_M + r]);
  return rsqrtf(tot / (float)NC_D + NC_RMS_EPS);
}

// Drain this thread's 64 of 256 scratch columns: SiLU(rs * v + bias) -> bf16 into buf
// (local); rs is the row's RMSNorm factor of the product's input.
__device__ void drain_silu(uint8_t* buf, uint32_t tscr, const float* bias, float rs, int cg, int r) {
#pragma unroll 1
  for (int j = 0; j < 2; ++j) {
    const int c0 = 64 * cg + 32 * j;
    float v[32];
    ld32f(tscr + c0, v);
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
      v[e] = fmaf(rs, v[e], bias[c0 + e]);
      v[e + 1] = fmaf(rs, v[e + 1], bias[c0 + e + 1]);
      silu2(v[e], v[e + 1]);
    }
    put32(buf, r, c0, v);
  }
}

// The drafter-state, slot and rank table rows of this CTA's slice in HF chunks 2-3: 256-byte rows
// (64 fp32) whose 16-byte pieces are XOR-swizzled by row; c is a multiple of 4 below 64.
__device__ __forceinline__ float* tab_at(uint8_t* sm, int row, int c) {
  return reinterpret_cast<float*>(sm + OFF_HF + 2 * CHUNK) + (size_t)row * NC_SL +
         ((((c >> 2) ^ (row & 7))) << 2);
}

// Layer l's vectors (this CTA's slices of the norm gains, b_o and b_2; b_1, the q|k|v
// biases, the relative-position and same-slot biases) into shared memory by asynchronous
// copies: issued once the previous readers are past a barrier, completed (and the biases
// scaled by log2 e) by layer_vectors_finish from the same thread before a barrier.
__device__ void layer_vectors_issue(const ClusterArgs& a, int l, float* vec, float* s_dist,
                                    float* s_same, int tid, int c0s, int nd) {
  for (int i = tid; i < 4 * (NC_SL / 4); i += NC_RW) {
    const int part = i / (NC_SL / 4), c = 4 * (i % (NC_SL / 4));
    const float* src = part == 0 ? a.an[l] : part == 1 ? a.fn[l] : part == 2 ? a.bo[l] : a.b2[l];
    float* dst = vec + (part == 0 ? V_AN : part == 1 ? V_FN : part == 2 ? V_BO : V_B2 + (l & 1) * NC_SL);
    cp_async16(dst + c, src + c0s + c);
  }
  for (int i = tid; i < NC_F / 4; i += NC_RW) cp_async16(vec + V_B1 + 4 * i, a.b1[l] + 4 * i);
  for (int i = tid; i < 3 * NC_D / 4; i += NC_RW) cp_async16(vec + V_BQKV + 4 * i, a.bqkv[l] + 4 * i);
  for (int i = tid; i < NC_NH * nd / 4; i += NC_RW) cp_async16(s_dist + 4 * i, a.dist[l] + 4 * i);
  if (tid < NC_NH / 4) cp_async16(s_same + 4 * tid, a.same[l] + 4 * tid);
}
__device__ void layer_vectors_finish(float* s_dist, float* s_same, int tid, int nd) {
  cp_async_wait_all();
  for (int i = tid; i < NC_NH * nd / 4; i += NC_RW)
#pragma unroll
    for (int e = 0; e < 4; ++e) s_dist[4 * i + e] *= NC_LOG2E;
  if (tid < NC_NH / 4)
#pragma unroll
    for (int e = 0; e < 4; ++e) s_same[4 * tid + e] *= NC_LOG2E;
}

__global__ void __launch_bounds__(NC_THREADS, 1)
    net_cluster_kernel(const __grid_constant__ ClusterMaps maps, const __grid_constant__ ClusterArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint32_t tmem_base;
  __shared__ volatile int abort_flag;
  Shared sh;
  sh.base = sm;
  sh.full = reinterpret_cast<uint64_t*>(sm + OFF_BAR);
  sh.empty = sh.full + NC_SLOTS;
  sh.done = sh.empty + NC_SLOTS;
  sh.ready = sh.done + N_DONE;
  sh.xg = sh.ready + N_READY;
  sh.w1f = sh.xg + N_XG;
  sh.prb = sh.w1f + N_W1F;
  sh.abort = &abort_flag;
  float* s_ss = reinterpret_cast<float*>(sm + OFF_SS);
  float* s_ssx = reinterpret_cast<float*>(sm + OFF_SSX);
  float* s_dist = reinterpret_cast<float*>(sm + OFF_DIST);
  float* s_same = reinterpret_cast<float*>(sm + OFF_SAME);
  uint8_t* s_slot = sm + OFF_SLOT;
  int32_t* s_ids = reinterpret_cast<int32_t*>(sm + OFF_IDS);
  float* vec = reinterpret_cast<float*>(sm + OFF_VEC);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int me = (int)cluster_rank();
  const int b = blockIdx.x / NC_CC;                  // the cluster's sequence
  const int nl = a.n_layers;
  if (threadIdx.x == 0) {
    for (int s = 0; s < NC_SLOTS; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], 1);
    }
    for (int e = 0; e < N_DONE; ++e) {
      mbar_init(&sh.done[e], 1);
      mbar_init(&sh.ready[e], NC_RW / 32);
    }
    for (int e = 0; e < N_XG; ++e) mbar_init(&sh.xg[e], 1);
    for (int e = 0; e < N_W1F; ++e) mbar_init(&sh.w1f[e], NC_CC - 1);
    mbar_init(sh.prb, NC_CC - 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    // every exchange barrier: this CTA's own arrival now, the peers' bytes later
    for (int l = 0; l < nl; ++l) {
      mbar_expect_tx(&sh.xg[X_SS(l)], XB_SS);
      mbar_expect_tx(&sh.xg[X_XN(l)], XB_SLICE);
      mbar_expect_tx(&sh.xg[X_ATT(l)], XB_SLICE);
      mbar_expect_tx(&sh.xg[X_SS2(l)], XB_SS);
      mbar_expect_tx(&sh.xg[X_XN2(l)], XB_SLICE);
      mbar_expect_tx(&sh.xg[X_H(l)], XB_H);
    }
    mbar_expect_tx(&sh.xg[xb(nl)], XB_SS);
    mbar_expect_tx(&sh.xg[xb(nl) + 1], XB_SLICE);
    mbar_expect_tx(&sh.xg[X_C1], XB_SLICE);
  }
  const int c0s = NC_SL * me;                        // first column of this CTA's slice
  const int nd = 2 * a.L - 1;
  if (warp >= 2) {
    // weights only, before the wait on earlier launches: the confidence network
    // (W_c1 transposed to [5][D]) and biases, the slice parts of b_c2, the final gain and
    // the out / in head biases, the slot and rank tables, the first layer's vectors
    const int tid = threadIdx.x - 64;
    for (int i = tid; i < NC_D * LILICORR_N_CONF; i += NC_RW)
      cp_async4(vec + V_C1W + (i % LILICORR_N_CONF) * NC_D + i / LILICORR_N_CONF, a.conf1_w + i);
    for (int i = tid; i < NC_D / 4; i += NC_RW) cp_async16(vec + V_C1B + 4 * i, a.conf1_b + 4 * i);
    for (int i = tid; i < NC_SL / 4; i += NC_RW) {
      cp_async16(vec + V_C2B + 4 * i, a.conf2_b + c0s + 4 * i);
      cp_async16(vec + V_FIN + 4 * i, a.final_norm + c0s + 4 * i);
    }
    for (int i = tid; i < 2 * NC_SL / 4; i += NC_RW)     // out, then in biases of the slice
      cp_async16(vec + V_BOI + 4 * i, a.boi + (i < NC_SL / 4 ? 0 : a.d2 / 2) + c0s + 4 * (i % (NC_SL / 4)));
    for (int i = tid; i < (a.L + a.K) * (NC_SL / 4); i += NC_RW) {
      const int row = a.L + i / (NC_SL / 4), c = (i % (NC_SL / 4)) * 4;
      const float* src = row < 2 * a.L ? a.slot + (size_t)(row - a.L) * NC_D + c0s + c
                                       : a.rank + (size_t)(row - 2 * a.L) * NC_D + c0s + c;
      cp_async16(tab_at(sm, row, c), src);
    }
    layer_vectors_issue(a, 0, vec, s_dist, s_same, tid, c0s, nd);
  }
  if (warp == 1) tmem_alloc(&tmem_base, NC_TMEM);
  tc_fence_before();
  cluster_sync();                  // every CTA's barriers exist before any peer signals them
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  if (warp == 0 && lane == 0)      // the weight stream needs nothing from earlier launches
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  else
    pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      Producer p{&maps, sh, me, 0u, 0u};
      schedule(a, p);
    }
  } else if (warp == 1) {       // the whole warp walks the schedule (warp-uniform
    Issuer is{&a, sh, 0u, 0u, tmem};   // descriptors); one lane issues
    schedule(a, is);
  } else {
    // ------------------------------------------------------------ row workers
    const int cg = (warp - 2) >> 2;
    const int set = cg >> 1;                         // head of the pair in the attention core
    const int wi = (warp - 2) & 7;                   // warp inside the set: queries 16wi..+15
    const int q = warp & 3;
    const int r = q * 32 + lane;                     // node row
    const int wr = warp - 2;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const uint32_t tx = tmem + lane_off + X_COL, tscr = tmem + lane_off + SCR_COL;
    const int L = a.L, K = a.K, LK = a.LK;
    const int tid = threadIdx.x - 64;
    const bool ok = r < LK;
    Peers pe;
    pe.local = smem_u32(sm);
#pragma unroll
    for (int qq = 1; qq < NC_CC; ++qq) pe.base[qq - 1] = peer_addr(pe.local, (uint32_t)((me + qq) % NC_CC));
    // the sequence's vectors from earlier launches: the fusion layer's t block and t
    for (int i = tid; i < NC_D / 4; i += NC_RW) cp_async16(vec + V_CB + 4 * i, a.cb + (size_t)b * NC_D + 4 * i);
    for (int i = tid; i < NC_SL / 4; i += NC_RW) {
      cp_async16(vec + V_T + 4 * i, a.t + (size_t)b * NC_D + c0s + 4 * i);
      if (a.tail) cp_async16(vec + V_ANC + 4 * i, a.tl.anchor + (size_t)b * (a.d2 / 2) + c0s + 4 * i);
    }
    for (int i = tid; i < NC_D / 4; i += NC_RW)          // all of t (the x*t block)
      cp_async16(vec + V_TF + 4 * i, a.t + (size_t)b * NC_D + 4 * i);

    // ---- nodes: x[:, slice] = fold[id] + W_h h_s + b_h + slot[s] + rank[k] + b_c2, and
    //      c1 = SiLU(W_c1 f + b_c1) over all 256 columns (the conf2 operand)
    {
      float f[LILICORR_N_CONF] = {0.f, 0.f, 0.f, 0.f, 0.f};
      if (ok) {
        const int s = r / K, k = r % K;
        const size_t rk = ((size_t)b * L + s) * K;
        if (cg == 0) {
          int id = a.ids[rk + k];
          if (id < 0 || id >= a.V) {                // an id outside the vocabulary: flag, read row 0
            set_status(a.status, LILICORR_ERR_ARG);
            id = 0;
          }
          s_ids[r] = id;
        }
        const float lp = a.logp[rk + k], lp0 = a.logp[rk];
        f[0] = lp;
        f[1] = expf(lp);
        f[2] = lp0 - lp;
        f[3] = K > 1 ? (float)k / (float)(K - 1) : 0.f;
        f[4] = k == 0 ? 1.f : 0.f;
      }
      // slice rows of the drafter state, slot and rank tables (HF chunks 2-3, 256-byte rows whose
      // 16-byte pieces are XOR-swizzled by row) and of the folded embedding (HF)
      float* fold_s = reinterpret_cast<float*>(sm + OFF_HF);
      auto fold_at = [&](int row, int c) {
        return fold_s + (size_t)row * NC_SL + ((((c >> 2) ^ (row & 7))) << 2);
      };
      for (int i = tid; i < L * (NC_SL / 4); i += NC_RW) {
        const int row = i / (NC_SL / 4), c = (i % (NC_SL / 4)) * 4;
        cp_async16(tab_at(sm, row, c), a.hproj + ((size_t)b * L + row) * NC_D + c0s + c);
      }
      rw_bar();                                      // s_ids complete
      for (int i = tid; i < LK * (NC_SL / 4); i += NC_RW) {
        const int n = i / (NC_SL / 4), c = (i % (NC_SL / 4)) * 4;
        cp_async16(fold_at(n, c), a.fold + (size_t)s_ids[n] * NC_D + c0s + c);
      }
      cp_async_wait_all();
      rw_bar();
      for (int i = tid; i < L * (NC_SL / 4); i += NC_RW) {   // S[s] = hproj + slot + b_c2
        const int row = i / (NC_SL / 4), c = (i % (NC_SL / 4)) * 4;
        float4 x = *reinterpret_cast<float4*>(tab_at(sm, row, c));
        const float4 y = *reinterpret_cast<const float4*>(tab_at(sm, L + row, c));
        const float4 z = *reinterpret_cast<const float4*>(vec + V_C2B + c);
        x.x += y.x + z.x; x.y += y.y + z.y; x.z += y.z + z.z; x.w += y.w + z.w;
        *reinterpret_cast<float4*>(tab_at(sm, row, c)) = x;
      }
      rw_bar();
      {
        const int srow = ok ? r / K : 0, rrow = 2 * L + (ok ? r % K : 0);
        float v[16];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int c = 16 * cg + 4 * u;
          const float4 x = *reinterpret_cast<const float4*>(fold_at(ok ? r : 0, c));
          const float4 y = *reinterpret_cast<const float4*>(tab_at(sm, srow, c));
          const float4 z = *reinterpret_cast<const float4*>(tab_at(sm, rrow, c));
          v[4 * u] = ok ? x.x + y.x + z.x : 0.f;
          v[4 * u + 1] = ok ? x.y + y.y + z.y : 0.f;
          v[4 * u + 2] = ok ? x.z + y.z + z.z : 0.f;
          v[4 * u + 3] = ok ? x.w + y.w + z.w : 0.f;
        }
        st16f(tx + 16 * cg, v);
      }
      // c1 for this CTA's 64 columns (16 per thread) into chunk me of ACT, then to the
      // peers (the W_c2 operand needs all 256)
      {
        const int c0 = NC_SL * me + 16 * cg;
        float c1[16];
#pragma unroll
        for (int e = 0; e < 16; e += 4) {
          float4 z = *reinterpret_cast<const float4*>(vec + V_C1B + c0 + e);
#pragma unroll
          for (int i = 0; i < LILICORR_N_CONF; ++i) {
            const float4 w = *reinterpret_cast<const float4*>(vec + V_C1W + i * NC_D + c0 + e);
            z.x = fmaf(w.x, f[i], z.x);
            z.y = fmaf(w.y, f[i], z.y);
            z.z = fmaf(w.z, f[i], z.z);
            z.w = fmaf(w.w, f[i], z.w);
          }
          silu2(z.x, z.y);
          silu2(z.z, z.w);
          c1[e] = ok ? z.x : 0.f;
          c1[e + 1] = ok ? z.y : 0.f;
          c1[e + 2] = ok ? z.z : 0.f;
          c1[e + 3] = ok ? z.w : 0.f;
        }
        put16(sm + OFF_ACT, me, r, cg, c1);
        send_all(sm + OFF_ACT + (size_t)me * CHUNK, CHUNK, &sh.xg[X_C1], tid, pe);
      }
      tmem_wait_st();
      if (cg == 0) s_slot[r] = (uint8_t)min(r / K, L - 1);   // read after the next rw_bar
      rw_signal(&sh.ready[0], lane);
    }

    // ---- Transformer layers
    for (int l = 0; l < nl; ++l) {
      ev_wait(&sh.done[l == 0 ? 0 : D_LAYER(l - 1)], sh.abort);
      tc_fence_after();
      layer_vectors_finish(s_dist, s_same, tid, nd);   // issued a product earlier
      rw_bar();
      // x += b_2 of the previous layer; the row statistics, then (every CTA's W_2 is done)
      // x * g_attn (slice) everywhere
      float rs1;
      {
        float v[16];
        norm_stats(tx, l == 0 ? nullptr : vec + V_B2 + ((l - 1) & 1) * NC_SL, true, cg, r, me,
                   s_ss, s_ssx, &sh.xg[X_SS(l)], pe, v);
        rs1 = norm_recv(r, s_ssx, &sh.xg[X_SS(l)], sh.abort);
        norm_operand(v, vec + V_AN, sm + OFF_ACT, &sh.xg[X_XN(l)], cg, r, me, tid,
                     pe);
      }
      rw_signal(&sh.ready[R_XN(l)], lane);

      // q | k (bf16) and v (fp16) of head 2me+set -> ACT (free once q|k|v ran): the row's
      // RMSNorm factor and the biases applied
      ev_wait(&sh.done[D_QKV(l)], sh.abort);
      tc_fence_after();
      uint8_t* qs = sm + OFF_ACT + set * QKV_SET;
      const int hh = 2 * me + set;
      // the row's 96 values of the head split evenly over the two threads of the set:
      // q and the first half of k, or the second half of k and v
      const int odd = cg & 1;
      {
        const int part = odd ? 2 : 0;
        float v[32];
        ld32f(tscr + 64 * part + 32 * set, v);
        const float* bq = vec + V_BQKV + part * NC_D + hh * NC_HD;
        const bool zero = part == 2 && r >= LK;      // padded values (their keys are masked)
#pragma unroll
        for (int e = 0; e < 32; ++e) v[e] = zero ? 0.f : fmaf(rs1, v[e], bq[e]);
        uint8_t* dst = qs + part * 8192;
#pragma unroll
        for (int p = 0; p < 4; ++p)
          *reinterpret_cast<uint4*>(dst + qkv_off(r, p)) =
              part == 2 ? pack8h(v + 8 * p) : pack8(v + 8 * p);
      }
      {
        float v[16];
        ld16f(tscr + 64 + 32 * set + 16 * odd, v);
        const float* bq = vec + V_BQKV + NC_D + hh * NC_HD + 16 * odd;
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = fmaf(rs1, v[e], bq[e]);
#pragma unroll
        for (int p = 0; p < 2; ++p)
          *reinterpret_cast<uint4*>(qs + 8192 + qkv_off(r, 2 * odd + p)) = pack8(v + 8 * p);
      }
      set_bar(set);
      {
        const int q0 = 16 * wi;
        const int i0 = q0 + (lane >> 2), i1 = i0 + 8, t4 = lane & 3;
        float o[4][4], inv0, inv1;
        head_attention(smem_u32(qs), LK, K, s_slot, s_dist + hh * nd + (L - 1), s_same[hh], q0,
                       lane, o, inv0, inv1);
        // the pair's 64 attention-output columns: chunk me of HF, here and in the peers
        uint8_t* att = sm + OFF_HF + (size_t)me * CHUNK;
#pragma unroll
        for (int nb = 0; nb < 4; ++nb) {
          const int piece = 4 * set + nb;
          *reinterpret_cast<uint32_t*>(att + swz(i0, piece) + 4 * t4) =
              pack_bf16x2(o[nb][0] * inv0, o[nb][1] * inv0);
          *reinterpret_cast<uint32_t*>(att + swz(i1, piece) + 4 * t4) =
              pack_bf16x2(o[nb][2] * inv1, o[nb][3] * inv1);
        }
        send_all(att, CHUNK, &sh.xg[X_ATT(l)], tid, pe);
      }
      rw_signal(&sh.ready[R_ATT(l)], lane);

      // x += b_o; x * g_ffn (slice) everywhere, the row statistics
      ev_wait(&sh.done[D_WO(l)], sh.abort);
      tc_fence_after();
      {
        float v[16];
        norm_stats(tx, vec + V_BO, true, cg, r, me, s_ss, s_ssx + NC_CC * NC_M, &sh.xg[X_SS2(l)],
                   pe, v);
        norm_operand(v, vec + V_FN, sm + OFF_ACT, &sh.xg[X_XN2(l)], cg, r, me,
                     tid, pe);
      }
      rw_signal(&sh.ready[R_XN2(l)], lane);
      const float rs2 = norm_recv(r, s_ssx + NC_CC * NC_M, &sh.xg[X_SS2(l)], sh.abort);
      // FFN hidden units 128me..128me+127: SiLU(rs2 * acc + b_1) -> bf16, gathered into
      // the W_2 operand (units 0-255 in HF, 256-511 in ACT) here and in every peer. ACT
      // still holds the W_1 operand until each CTA's W_1 product is done: CTAs that write
      // there wait for the three peers' word (the W_1 products' completion, signalled as
      // soon as this CTA sees its own).
      ev_wait(&sh.done[D_W1(l)], sh.abort);
      tc_fence_after();
      if (tid == 0) {
        uint64_t* wf = &sh.w1f[l];
#pragma unroll
        for (int qq = 1; qq < NC_CC; ++qq) mbar_arrive_peer(pe.at(qq, wf));
      }
      {
        uint8_t* hbuf = me < 2 ? sm + OFF_HF : sm + OFF_ACT;
        const int ch0 = 2 * (me & 1);              // the two chunks of this CTA's units
        float v[32];
        ld32f(tscr + 32 * cg, v);
        const float* b1 = vec + V_B1 + 128 * me + 32 * cg;
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          v[e] = fmaf(rs2, v[e], b1[e]);
          v[e + 1] = fmaf(rs2, v[e + 1], b1[e + 1]);
          silu2(v[e], v[e + 1]);
        }
        // columns 32cg..32cg+31 of the 128: chunk ch0 + (cg >> 1), pieces 4(cg & 1)..+3
        uint8_t* ch = hbuf + (size_t)(ch0 + (cg >> 1)) * CHUNK;
#pragma unroll
        for (int p = 0; p < 4; ++p)
          *reinterpret_cast<uint4*>(ch + swz(r, 4 * (cg & 1) + p)) = pack8(v + 8 * p);
        fence_async_shared();
        rw_bar();
        if (tid == 0) {
          if (me >= 2) xg_wait(&sh.w1f[l], sh.abort);   // the peers' ACT is free
          uint8_t* src = hbuf + (size_t)ch0 * CHUNK;
#pragma unroll
          for (int qq = 1; qq < NC_CC; ++qq)
            bulk_to_peer(pe.at(qq, src), src, 2 * CHUNK, pe.at(qq, &sh.xg[X_H(l)]));
          bulk_wait_read();
        }
        // every reader of this layer's vectors is past the barrier: the next layer's
        // vectors load while W_2 runs
        if (l + 1 < nl) layer_vectors_issue(a, l + 1, vec, s_dist, s_same, tid, c0s, nd);
      }
      rw_signal(&sh.ready[R_H(l)], lane);
    }

    // ---- fusion: xf = RMSNorm(x + b_2) -> ACT, xf * t -> HF (slices everywhere);
    //      u = SiLU(. + cb) -> ACT
    ev_wait(&sh.done[D_LAYER(nl - 1)], sh.abort);
    tc_fence_after();
    float rsf;
    {
      float v[16];
      norm_stats(tx, vec + V_B2 + ((nl - 1) & 1) * NC_SL, false, cg, r, me, s_ss, s_ssx,
                 &sh.xg[xb(nl)], pe, v);
      rsf = norm_recv(r, s_ssx, &sh.xg[xb(nl)], sh.abort);
      // xf here and in the peers (ACT); xf * t of this CTA's slice into HF here
      float vt[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) vt[e] = v[e] * vec[V_FIN + 16 * cg + e] * vec[V_T + 16 * cg + e];
      put16(sm + OFF_HF, me, r, cg, vt);
      norm_operand(v, vec + V_FIN, sm + OFF_ACT, &sh.xg[xb(nl) + 1], cg, r, me,
                   tid, pe);
    }
    // xf * t of the peers' slices from their xf, once it is here (one exchange instead of
    // two): 16 columns of each peer chunk per thread
    xg_wait(&sh.xg[xb(nl) + 1], sh.abort);
#pragma unroll 1
    for (int qq = 1; qq < NC_CC; ++qq) {
      const int q = (me + qq) % NC_CC;
#pragma unroll
      for (int p = 0; p < 2; ++p) {
        const uint32_t off = (uint32_t)q * CHUNK + swz(r, 2 * cg + p);
        const uint4 w = *reinterpret_cast<const uint4*>(sm + OFF_ACT + off);
        const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
        const float* tq = vec + V_TF + NC_SL * q + 16 * cg + 8 * p;
        float x8[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          x8[2 * e] = __uint_as_float(wv[e] << 16) * tq[2 * e];
          x8[2 * e + 1] = __uint_as_float(wv[e] & 0xFFFF0000u) * tq[2 * e + 1];
        }
        *reinterpret_cast<uint4*>(sm + OFF_HF + off) = pack8(x8);
      }
    }
    rw_signal(&sh.ready[lb(nl)], lane);
    ev_wait(&sh.done[lb(nl)], sh.abort);
    tc_fence_after();
    drain_silu(sm + OFF_ACT, tscr, vec + V_CB, rsf, cg, r);
    rw_signal(&sh.ready[lb(nl) + 1], lane);
    // ---- out / in heads: this CTA's 64 columns of the out and of the in vectors -> oi
    //      (fp32, not yet unit) through a staging buffer (row r: 64 out then 64 in values,
    //      16-byte pieces swizzled by row) for row-contiguous stores
    ev_wait(&sh.done[lb(nl) + 1], sh.abort);
    tc_fence_after();
    {
      uint8_t* stg = sm + OFF_HF;
      auto stg_at = [&](int row, int piece) {
        return reinterpret_cast<float4*>(stg + row * 512 + ((piece ^ (row & 7)) << 4));
      };
      float ss = 0.f;
#pragma unroll 1
      for (int j = 0; j < 2; ++j) {
        const int cl = 32 * cg + 16 * j;            // column of the 128 staged
        float v[16];
        ld16f(tscr + cl, v);
        const float* bo = vec + V_BOI + cl;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float4 w = make_float4(v[4 * u] + bo[4 * u], v[4 * u + 1] + bo[4 * u + 1],
                                       v[4 * u + 2] + bo[4 * u + 2], v[4 * u + 3] + bo[4 * u + 3]);
          ss = fmaf(w.x, w.x, fmaf(w.y, w.y, fmaf(w.z, w.z, fmaf(w.w, w.w, ss))));
          *stg_at(r, (cl >> 2) + u) = w;
        }
      }
      s_ss[cg * NC_M + r] = ss;                    // 32 columns' part of |o|^2 (cg < 2) or |i|^2
      rw_bar();
      const int dh = a.d2 / 2;
      for (int row = wr; row < LK; row += NC_RW / 32)
        *reinterpret_cast<float4*>(a.oi + ((size_t)b * LK + row) * a.d2 + (lane < 16 ? 0 : dh) + c0s +
                                   4 * (lane & 15)) = *stg_at(row, lane);
      if (a.tail) {
        // Steps (3), (4): the scores are cosines over all d columns (Eq. "pair"), so each
        // CTA sums its 64 columns' part of every dot product and squared norm into a record
        // in its (now idle) weight ring: pair dots [(L-1)][K][K] (out of slot s, in of
        // slot s+1), anchor dots [K], |o|^2 [LK], |i|^2 [LK], |anchor|^2. The first CTA
        // adds the peers' records (in rank order), forms the cosines and walks.
        float* pr = reinterpret_cast<float*>(sm + OFF_RING);
        const int npair = (L - 1) * K * K, o_ad = npair, o_on = o_ad + K, o_in = o_on + LK,
                  o_an = o_in + LK, npr = o_an + 1;
        for (int idx = tid; idx < npair; idx += NC_RW) {
          const int s = idx / (K * K), j = (idx / K) % K, k = idx % K;
          const int n1 = s * K + j, n2 = (s + 1) * K + k;
          float dot = 0.f;
#pragma unroll 4
          for (int p = 0; p < 16; ++p) {
            const float4 o = *stg_at(n1, p), i = *stg_at(n2, 16 + p);
            dot = fmaf(o.x, i.x, fmaf(o.y, i.y, fmaf(o.z, i.z, fmaf(o.w, i.w, dot))));
          }
          pr[idx] = dot;
        }
        for (int k = tid; k < K; k += NC_RW) {
          const float* an = vec + V_ANC;
          float dot = 0.f;
          for (int p = 0; p < 16; ++p) {
            const float4 i = *stg_at(k, 16 + p);
            dot = fmaf(an[4 * p], i.x, fmaf(an[4 * p + 1], i.y, fmaf(an[4 * p + 2], i.z, fmaf(an[4 * p + 3], i.w, dot))));
          }
          pr[o_ad + k] = dot;
        }
        if (cg == 0 && r < LK) {
          pr[o_on + r] = s_ss[r] + s_ss[NC_M + r];
          pr[o_in + r] = s_ss[2 * NC_M + r] + s_ss[3 * NC_M + r];
        }
        if (wr == 0) {
          float q = 0.f;
          for (int c = lane; c < NC_SL; c += 32) q = fmaf(vec[V_ANC + c], vec[V_ANC + c], q);
          q = warp_sum(q);
          if (lane == 0) pr[o_an] = q;
        }
        rw_bar();
        if (me != 0) {
          if (tid == 0) mbar_arrive_peer(pe.at(NC_CC - me, sh.prb));   // to rank 0
        } else if (xg_wait(sh.prb, sh.abort)) {
          for (int i = tid; i < npr; i += NC_RW) {
            float v = pr[i];
#pragma unroll
            for (int q = 1; q < NC_CC; ++q) v += ld_peer_f32(pe.at(q, pr + i));
            pr[i] = v;
          }
          rw_bar();
          const float an = fmaxf(sqrtf(pr[o_an]), 1e-12f);
          float* gP = a.tl.P + (size_t)b * npair;
          for (int idx = tid; idx < npair; idx += NC_RW) {
            const int s = idx / (K * K), j = (idx / K) % K, k = idx % K;
            const float v = pr[idx] / (fmaxf(sqrtf(pr[o_on + s * K + j]), 1e-12f) *
                                       fmaxf(sqrtf(pr[o_in + (s + 1) * K + k]), 1e-12f));
            pr[idx] = v;
            gP[idx] = v;
          }
          for (int k = tid; k < K; k += NC_RW) {
            const float v = pr[o_ad + k] / (an * fmaxf(sqrtf(pr[o_in + k]), 1e-12f));
            pr[o_ad + k] = v;
            a.tl.A[(size_t)b * K + k] = v;
          }
          rw_bar();
          if (wr == 0) {
            walk::walk_sequence(pr + o_ad, pr, b, L, K, nullptr, s_slot);
            __syncwarp();
            for (int s = lane; s < L; s += 32) {
              const size_t o = (size_t)b * L + s;
              const int c = s_slot[s];
              a.tl.choice[o] = c;
              a.tl.tokens[o] = a.ids[o * K + c];
            }
          }
        }
      }
    }
  }

  // ---- teardown: no CTA leaves while a peer may still address its shared memory
  tc_fence_before();
  __syncthreads();
  if (abort_flag) {
    if (threadIdx.x == 0) {
      set_status(a.status, LILICORR_ERR_TIMEOUT);
      const long long t0 = clock64();            // let copies and products in flight land
      while (clock64() - t0 < NC_WAIT / 10) {
      }
    }
    __syncthreads();
  }
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, NC_TMEM);
  }
}

// W [rows, cols] bf16 row-major as (64, rows, cols / 64): box (64, box_rows, 1) is one K
// chunk of box_rows rows, 128-byte swizzled.
bool nc_chunk_map(CUtensorMap* m, const void* W, int rows, int cols, int box_rows) {
  const uint64_t dims[3] = {64, (uint64_t)rows, (uint64_t)(cols / 64)};
  const uint64_t strides[3] = {2, (uint64_t)cols * 2, 128};
  const uint32_t box[3] = {64, (uint32_t)box_rows, 1};
  return make_map_nd(m, W, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, dims, strides, box);
}
// W_qkv [3D, D] as (64 k, 64 rows, 4 head pairs, 3 parts q/k/v, D / 64 chunks): box
// (64, 64, 1, 3, 1) brings the q, k and v rows of one head pair for one K chunk.
bool nc_qkv_map(CUtensorMap* m, const void* W) {
  const uint64_t dims[5] = {64, 64, NC_D / 64, 3, NC_D / 64};
  const uint64_t strides[5] = {2, NC_D * 2, 64ull * NC_D * 2, (uint64_t)NC_D * NC_D * 2, 128};
  const uint32_t box[5] = {64, 64, 1, 3, 1};
  return make_map_nd(m, W, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, dims, strides, box);
}

}  // namespace

bool net_cluster_supported(const lilicorr_head_desc& d) {
  return d.dtype == LILICORR_BF16 && d.D == NC_D && d.ffn == NC_F && d.n_heads == NC_NH &&
         d.n_layers >= 1 && d.n_layers <= NC_MAX_LAYERS && d.L >= 1 && d.L <= NC_MAX_L &&
         d.K >= 1 && d.L * d.K <= NC_M && (2 * d.L + d.K) * NC_SL * 4 <= 2 * (int)CHUNK &&
         2 * d.d == NC_CC * 128 && encode_fn() != nullptr;
}

void* net_cluster_maps_create(const lilicorr_head* h) {
  const lilicorr_head_desc& d = h->desc;
  if (!net_cluster_supported(d)) return nullptr;
  ClusterMaps* m = new (std::nothrow) ClusterMaps;
  if (!m) return nullptr;
  memset(m, 0, sizeof(*m));
  bool ok = nc_chunk_map(&m->conf2, h->conf2_w, NC_D, NC_D, NC_SL) &&
            nc_chunk_map(&m->fuse, h->fuse_x, NC_D, 2 * NC_D, 256) &&
            nc_chunk_map(&m->woi, h->woi, 2 * d.d, NC_D, NC_SL);
  for (int l = 0; l < d.n_layers && ok; ++l) {
    const HeadW& w = h->layer[l];
    ok = nc_qkv_map(&m->wqkv[l], w.wqkv) && nc_chunk_map(&m->wo[l], w.wo, NC_D, NC_D, NC_SL) &&
         nc_chunk_map(&m->w1[l], w.w1, NC_F, NC_D, 128) &&
         nc_chunk_map(&m->w2[l], w.w2, NC_D, NC_F, NC_SL);
  }
  for (int l = d.n_layers; l < NC_MAX_LAYERS && ok; ++l) {   // unused slots: valid maps
    m->wqkv[l] = m->wqkv[0];
    m->wo[l] = m->wo[0];
    m->w1[l] = m->w1[0];
    m->w2[l] = m->w2[0];
  }
  if (!ok) {
    delete m;
    return nullptr;
  }
  return m;
}

void net_cluster_maps_free(void* p) { delete static_cast<ClusterMaps*>(p); }

// Clusters of this kernel that fit on the current device at once (0 if it cannot run).
int net_cluster_capacity() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    (void)cudaGetLastError();
    return 0;
  }
  if (cache[dev]) return cache[dev] > 0 ? cache[dev] : 0;
  static bool configured[64] = {false};
  int n = 0;
  if (allow_max_dynamic_smem(net_cluster_kernel, configured) == LILICORR_OK) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(NC_CC * 64);
    cfg.blockDim = dim3(NC_THREADS);
    cfg.dynamicSmemBytes = NC_SMEM;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = NC_CC;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, net_cluster_kernel, &cfg) != cudaSuccess) n = 0;
  }
  (void)cudaGetLastError();
  cache[dev] = n > 0 ? n : -1;
  return n > 0 ? n : 0;
}

lilicorr_status_t launch_net_cluster(const lilicorr_head* h, int B, const int32_t* ids,
                                     const float* logp, const float* hproj, const float* t,
                                     const float* cb, float* oi, uint32_t* status, cudaStream_t st,
                                     const ClusterTail* tail) {
  if (B == 0) return LILICORR_OK;
  const ClusterMaps* m = static_cast<const ClusterMaps*>(h->cluster_maps);
  if (!m) return LILICORR_ERR_SHAPE;
  const lilicorr_head_desc& d = h->desc;
  ClusterArgs a;
  memset(&a, 0, sizeof(a));
  a.B = B; a.L = d.L; a.K = d.K; a.LK = d.L * d.K; a.V = d.V; a.n_layers = d.n_layers;
  a.d2 = 2 * d.d;
  a.ids = ids; a.logp = logp; a.hproj = hproj; a.t = t; a.cb = cb;
  a.fold = static_cast<const float*>(h->fold);
  a.slot = h->slot; a.rank = h->rank;
  a.conf1_w = h->conf1_w; a.conf1_b = h->conf1_b; a.conf2_b = h->conf2_b;
  for (int l = 0; l < d.n_layers; ++l) {
    const HeadW& w = h->layer[l];
    a.bqkv[l] = w.bqkv; a.bo[l] = w.bo; a.b1[l] = w.b1; a.b2[l] = w.b2;
    a.an[l] = w.an; a.fn[l] = w.fn; a.dist[l] = w.dist; a.same[l] = w.same;
  }
  a.final_norm = h->final_norm;
  a.boi = h->boi;
  a.oi = oi;
  a.status = status;
  if (tail) {
    a.tail = 1;
    a.tl = *tail;
  }
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(net_cluster_kernel, configured));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(NC_CC * B);
  cfg.blockDim = dim3(NC_THREADS);
  cfg.dynamicSmemBytes = NC_SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = NC_CC;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  count_launch();
  LL_CUDA_TRY(cudaLaunchKernelEx(&cfg, net_cluster_kernel, *m, a));
  return LILICORR_OK;
}

}  // namespace lilicorr
