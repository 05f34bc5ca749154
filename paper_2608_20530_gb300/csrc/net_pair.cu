// Step (2), candidate-dependent part, for sequences of 129-256 nodes: the node features, the
// two-layer scoring Transformer, the fusion layer and the out / in heads (Sec. 3.2; App. A)
// on the bf16 head with D = 256, 8 heads, FFN 2D, on a cluster of two CTAs per sequence.
//
// The L*K nodes are two 128-row tensor-core tiles; CTA rank p of the cluster owns nodes
// 128p .. 128p+127 and runs, for its tile, exactly the one-CTA kernel of net_fused.cu: the
// residual stream x[128, 256] in tensor memory (columns 0-255), every matrix product on its
// own rows with the weights streamed by TMA, the RMSNorms, the fusion layer and the heads.
// Only the attention reaches across the tiles (every node attends to all L*K nodes): per
// head, each CTA drains its rows' q, k, v from the scratch accumulator into shared memory
// and writes its k and v rows into the peer's copy as well (distributed shared memory), so
// both CTAs hold k and v of all 256 nodes. Two barriers per head and direction (16 warp
// arrivals each, release / acquire at cluster scope): one opens a CTA's buffer to the
// peer's rows once every warp of the CTA is done with what the buffer held before (the
// previous head, or the FFN and output staging that share it), the other says the peer's
// rows have landed. Each CTA opens its own buffer before it waits on the peer's, so the
// two never wait on each other in a cycle. The 16
// row-worker warps then take 16 queries each over one half of the keys (warp w: queries
// 16(w % 8).., keys 128(w / 8)..), and the two halves' online-softmax states (maxima,
// sums, unnormalised outputs) merge through shared memory: once every warp is done with the
// head's q, k and v, the buffer opens to the peer's rows of the next head, and the second-half
// warp parks its state (outputs as fp16) in the q rows and the 8 KB after v, where the
// first-half warp of the same queries combines it and writes the head's output. (A hand-off
// of the same state through tensor-memory columns, second-half warp storing and first-half
// warp loading the same lanes after tcgen05.wait::st, the thread-sync fences and a named
// barrier, gave run-to-run differences, so it is not used.) The two heads of a pair run one after the other,
// which keeps one head's q, k, v (40 KB) in the buffer that held both heads' before.
#include <new>

#include "net_common.cuh"

namespace lilicorr {

namespace {
using namespace tc;
using namespace net;

constexpr int NF_D = 256;                 // node width
constexpr int NF_F = 512;                 // FFN width
constexpr int NF_NH = 8;                  // heads
constexpr int NF_HD = 32;                 // head width
constexpr int NF_M = 128;                 // node rows per CTA
constexpr int NP_NODES = 2 * NF_M;         // nodes per sequence (two CTAs)
constexpr int NF_STAGES = 2;              // weight ring depth
constexpr int NF_MAX_LAYERS = 4;
constexpr int NF_MAX_L = 64;
constexpr int NF_RW = 512;                // row-worker threads (16 warps)
constexpr int NF_CG = 4;                  // a row's 256 columns split over 4 threads
constexpr int NF_CW = NF_D / NF_CG;       // 64 columns per thread
constexpr int NF_THREADS = 64 + NF_RW;
constexpr uint32_t STAGE_BYTES = 256 * 64 * 2;   // one K chunk of 256 weight rows
constexpr uint32_t CHUNK = 128 * 128;     // 128 rows x 64 bf16, one swizzled K chunk
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t X_COL = 0, SCR_COL = 256;
constexpr long long WAIT_LIMIT = 4000000000ll;   // about 2 s of SM cycles
constexpr float LOG2E = 1.4426950408889634f;
constexpr float NF_RMS_EPS = 1e-6f;

// shared-memory layout (offsets from the 1024-aligned base)
constexpr uint32_t OFF_RING = 0;
constexpr uint32_t OFF_ACT = OFF_RING + NF_STAGES * STAGE_BYTES;   // 64 KB: 4 chunks
constexpr uint32_t OFF_HF = OFF_ACT + 4 * CHUNK;                   // 64 KB: 4 chunks
constexpr uint32_t OFF_ATT = OFF_HF + 3 * CHUNK;                   // attention output chunk
constexpr uint32_t Q_OFF = 0, K_OFF = 8192, V_OFF = 8192 + 16384;  // one head in HF (40 KB)
constexpr uint32_t OFF_VEC = OFF_HF + 4 * CHUNK;                   // staged vectors (floats)
// float offsets inside the vector area
constexpr int V_AN = 0, V_FN = 256, V_BO = 512, V_B1 = 768, V_BQKV = 1280, V_B2 = 2048,
              V_C1W = 2560, V_C1B = 3840, V_C2B = 4096, V_FIN = 4352, V_BOI = 4608, V_T = 5120,
              V_CB = 5376, V_END = 5632;
constexpr uint32_t OFF_SS = OFF_VEC + V_END * 4;                   // [4][128] float
constexpr uint32_t OFF_DIST = OFF_SS + NF_CG * NF_M * 4;           // [8][127] float
constexpr uint32_t OFF_SAME = OFF_DIST + NF_NH * (2 * NF_MAX_L - 1) * 4;
constexpr uint32_t OFF_SLOT = OFF_SAME + NF_NH * 4;                // [256] slot of each node
constexpr uint32_t OFF_IDS = OFF_SLOT + NP_NODES;                  // [128] token id of each node
constexpr uint32_t OFF_BAR = (OFF_IDS + NF_M * 4 + 63) & ~63u;
constexpr int N_EV = 52;                                           // per direction
constexpr int N_KV = NF_MAX_LAYERS * NF_NH;                        // heads of a sequence
constexpr uint32_t NF_SMEM_USED = OFF_BAR + (2 * NF_STAGES + 2 * N_EV + 2 * N_KV) * 8;
constexpr size_t NF_SMEM = 1024 + NF_SMEM_USED;
static_assert(NF_SMEM <= 227 * 1024, "shared memory of the pair network kernel");
static_assert(OFF_ACT % 1024 == 0 && OFF_HF % 1024 == 0 && OFF_ATT % 1024 == 0, "swizzle atoms");

enum { G_CONF2, G_QKV, G_WO, G_W1, G_W2, G_FUSE, G_WOI };

// event ids: MMA -> row workers (commits) and row workers -> MMA (8 warp arrivals)
__device__ __forceinline__ int lb(int l) { return 1 + 11 * l; }
__device__ __forceinline__ int done_id(int kind, int l, int g, int nl) {
  switch (kind) {
    case G_CONF2: return 0;
    case G_QKV: return lb(l) + g;
    case G_WO: return lb(l) + 4 + g;
    case G_W1: return lb(l) + 8 + g;
    case G_W2: return g == 1 ? lb(l) + 10 : -1;
    case G_FUSE: return lb(nl);
    default: return lb(nl) + 1 + g;
  }
}
__device__ __forceinline__ int ready_id(int kind, int l, int g, int nl) {
  switch (kind) {
    case G_CONF2: return 0;
    case G_QKV: return g == 0 ? lb(l) : lb(l) + g;        // xn, then "q|k|v of pair g-1 drained"
    case G_WO: return lb(l) + 4 + g;                     // attention output of pair g
    case G_W1: return lb(l) + 8 + g;                     // xn2; then h_a drained into HF
    case G_W2: return g == 1 ? lb(l) + 10 : -1;          // h_b in ACT
    case G_FUSE: return lb(nl);
    default: return lb(nl) + 1 + g;                      // u; then head half g-1 drained
  }
}
// ids the row workers use
__device__ __forceinline__ int D_QKV(int l, int g) { return lb(l) + g; }
__device__ __forceinline__ int D_WO(int l, int g) { return lb(l) + 4 + g; }
__device__ __forceinline__ int D_FFN(int l, int h) { return lb(l) + 8 + h; }
__device__ __forceinline__ int D_LAYER(int l) { return lb(l) + 10; }
__device__ __forceinline__ int R_XN(int l) { return lb(l); }
__device__ __forceinline__ int R_QKV_DRAINED(int l, int g) { return lb(l) + 1 + g; }
__device__ __forceinline__ int R_ATT(int l, int g) { return lb(l) + 4 + g; }
__device__ __forceinline__ int R_XN2(int l) { return lb(l) + 8; }
__device__ __forceinline__ int R_HFA(int l) { return lb(l) + 9; }
__device__ __forceinline__ int R_HFB(int l) { return lb(l) + 10; }

struct NetMaps {
  CUtensorMap conf2, fuse, woi;
  CUtensorMap wqkv[NF_MAX_LAYERS], wo[NF_MAX_LAYERS], w1[NF_MAX_LAYERS], w2[NF_MAX_LAYERS];
};

struct NetArgs {
  int B, L, K, LK, V, n_layers, d2;
  const int32_t* ids;
  const float* logp;
  const float* hproj;       // [B*L, D]
  const float* t;           // [B, D]
  const float* cb;          // [B, D]: t block of the fusion layer plus its bias
  const float* fold;        // [V, D]
  const float *slot, *rank, *conf1_w, *conf1_b, *conf2_b;
  const float* bqkv[NF_MAX_LAYERS];
  const float* bo[NF_MAX_LAYERS];
  const float* b1[NF_MAX_LAYERS];
  const float* b2[NF_MAX_LAYERS];
  const float* an[NF_MAX_LAYERS];
  const float* fn[NF_MAX_LAYERS];
  const float* dist[NF_MAX_LAYERS];
  const float* same[NF_MAX_LAYERS];
  const float* final_norm;
  const float* boi;
  float* oi;                // [B*LK, d2]
  uint32_t* status;
};

// K chunks of a product and the rows (output columns) of each chunk's weight tile
__device__ __forceinline__ int n_chunks(int kind) {
  switch (kind) {
    case G_WO: return 1;
    case G_FUSE: return 8;
    default: return 4;
  }
}
__device__ __forceinline__ int tile_rows(int kind) { return kind == G_QKV ? 192 : 256; }

// Copy K chunk kc of product (kind, l, g)'s weights into a ring stage.
__device__ __forceinline__ void load_chunk(const NetMaps& m, int kind, int l, int g, int kc,
                                           void* dst, uint64_t* bar) {
  switch (kind) {
    case G_CONF2: tma_load_3d(dst, &m.conf2, bar, 0, 0, kc); break;
    // q, k, v rows of head pair g, gathered from [3D, D] by a 5-D view
    case G_QKV: tma_load_5d(dst, &m.wqkv[l], bar, 0, 0, g, 0, kc); break;
    case G_WO: tma_load_3d(dst, &m.wo[l], bar, 0, 0, g); break;
    case G_W1: tma_load_3d(dst, &m.w1[l], bar, 0, 256 * g, kc); break;
    case G_W2: tma_load_3d(dst, &m.w2[l], bar, 0, 0, 4 * g + kc); break;
    case G_FUSE: tma_load_3d(dst, &m.fuse, bar, 0, 0, kc); break;
    default: tma_load_3d(dst, &m.woi, bar, 0, 256 * g, kc); break;
  }
}

// The product sequence of one sequence, shared by the producer and the MMA issuer.
template <class Op>
__device__ __forceinline__ void schedule(const NetArgs& a, Op& op) {
  op.gemm(G_CONF2, 0, 0);
  for (int l = 0; l < a.n_layers; ++l) {
    op.gemm(G_QKV, l, 0);
    for (int g = 0; g < 4; ++g) {
      if (g + 1 < 4) op.gemm(G_QKV, l, g + 1);
      op.gemm(G_WO, l, g);
    }
    op.gemm(G_W1, l, 0);
    op.gemm(G_W1, l, 1);
    op.gemm(G_W2, l, 0);
    op.gemm(G_W2, l, 1);
  }
  op.gemm(G_FUSE, 0, 0);
  for (int h = 0; h * 256 < a.d2; ++h) op.gemm(G_WOI, 0, h);
}

struct Shared {
  uint8_t* base;
  uint64_t *full, *empty, *done, *ready;
  volatile int* abort;
};

__device__ __forceinline__ bool ev_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  if (*abort) return false;
  if (!mbar_wait(bar, parity, WAIT_LIMIT)) {
    *abort = 1;
    return false;
  }
  return true;
}

// wait for a phase that CTAs of the cluster complete (acquire at cluster scope), bounded
__device__ __forceinline__ bool ev_wait_cluster(uint64_t* bar, uint32_t parity, volatile int* abort) {
  if (*abort) return false;
  if (!mbar_wait_cluster_sleep(bar, parity, WAIT_LIMIT)) {
    *abort = 1;
    return false;
  }
  return true;
}
__device__ __forceinline__ void fence_cluster() {
  asm volatile("fence.acq_rel.cluster;" ::: "memory");
}

struct Producer {
  const NetMaps* m;
  const NetArgs* a;
  Shared sh;
  uint32_t n;                              // chunks issued so far
  __device__ void gemm(int kind, int l, int g) {
    const int nk = n_chunks(kind);
    const uint32_t bytes = (uint32_t)tile_rows(kind) * 128u;
    for (int kc = 0; kc < nk; ++kc, ++n) {
      const int s = (int)(n % NF_STAGES);
      const uint32_t ph = (n / NF_STAGES) & 1u;
      if (!ev_wait(&sh.empty[s], ph ^ 1u, sh.abort)) continue;
      mbar_expect_tx(&sh.full[s], bytes);
      load_chunk(*m, kind, l, g, kc, sh.base + OFF_RING + (size_t)s * STAGE_BYTES, &sh.full[s]);
    }
  }
};

struct Issuer {
  const NetArgs* a;
  Shared sh;
  uint32_t n, tmem, parity;
  __device__ void gemm(int kind, int l, int g) {
    const int nl = a->n_layers;
    const int rd = ready_id(kind, l, g, nl);
    if (rd >= 0) {
      ev_wait(&sh.ready[rd], parity, sh.abort);
      tc_fence_after();
    }
    const int nk = n_chunks(kind);
    const bool onto_x = kind == G_CONF2 || kind == G_WO || kind == G_W2;
    const uint32_t d = tmem + (onto_x ? X_COL : SCR_COL);
    const uint32_t idesc = kind == G_QKV ? instr_desc(128, 192) : instr_desc(128, 256);
    for (int kc = 0; kc < nk; ++kc, ++n) {
      uint32_t a_off;
      switch (kind) {
        case G_WO: a_off = OFF_ATT; break;
        case G_W2: a_off = (g == 0 ? OFF_HF : OFF_ACT) + kc * CHUNK; break;
        case G_FUSE: a_off = kc < 4 ? OFF_ACT + kc * CHUNK : OFF_HF + (kc - 4) * CHUNK; break;
        default: a_off = OFF_ACT + kc * CHUNK; break;
      }
      const int s = (int)(n % NF_STAGES);
      const uint32_t ph = (n / NF_STAGES) & 1u;
      if (!ev_wait(&sh.full[s], ph, sh.abort)) continue;
      tc_fence_after();
      const uint64_t ad = smem_desc(sh.base + a_off);
      const uint64_t bd = smem_desc(sh.base + OFF_RING + (size_t)s * STAGE_BYTES);
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_bf16(d, ad + 2ull * k, bd + 2ull * k, idesc, (onto_x || kc > 0 || k > 0) ? 1u : 0u);
      mma_commit(&sh.empty[s]);
    }
    const int dn = done_id(kind, l, g, nl);
    if (dn >= 0 && !*sh.abort) mma_commit(&sh.done[dn]);
  }
};

// ---------------------------------------------------------------- row-worker helpers
__device__ __forceinline__ uint32_t swz(int r, int j) {     // 16-byte piece j of row r
  return (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4));
}
__device__ __forceinline__ void rw_bar() { named_bar(1, NF_RW); }
// One warp's arrival on a row-worker -> MMA event, after its shared-memory writes
// (generic proxy, read by the tensor cores through the async proxy) and tensor-memory
// stores.
__device__ __forceinline__ void rw_signal(uint64_t* bar, int lane) {
  fence_async_shared();
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(bar);
}

// RMSNorm statistics of row r over the 256 columns of x (4 threads, 64 columns each):
// adds `bias` (shared memory) into x first, and writes x back to tensor memory when
// write_back. Returns 1 / rms.
__device__ float row_rstd(uint32_t tx, const float* bias, bool write_back, int cg, int r,
                          float* s_ss) {
  float ss = 0.f;
#pragma unroll 1
  for (int j = 0; j < 2; ++j) {
    const int c0 = NF_CW * cg + 32 * j;
    float v[32];
    ld32f(tx + c0, v);
    if (bias) {
#pragma unroll
      for (int e = 0; e < 32; ++e) v[e] += bias[c0 + e];
      if (write_back) st32f(tx + c0, v);
    }
#pragma unroll
    for (int e = 0; e < 32; ++e) ss = fmaf(v[e], v[e], ss);
  }
  if (bias && write_back) tmem_wait_st();
  s_ss[cg * NF_M + r] = ss;
  rw_bar();
  const float tot = (s_ss[r] + s_ss[NF_M + r]) + (s_ss[2 * NF_M + r] + s_ss[3 * NF_M + r]);
  rw_bar();                                  // s_ss free for the next statistics
  return rsqrtf(tot / (float)NF_D + NF_RMS_EPS);
}

// xn = (x + bias) * rstd * gain -> bf16 into ACT; with t, also xn * t -> HF
__device__ void row_normed(uint8_t* sm, uint32_t tx, const float* bias, float rstd,
                           const float* gain, const float* t, int cg, int r) {
#pragma unroll 1
  for (int j = 0; j < 2; ++j) {
    const int c0 = NF_CW * cg + 32 * j;
    float v[32];
    ld32f(tx + c0, v);
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      const float b = bias ? bias[c0 + e] : 0.f;
      v[e] = (v[e] + b) * rstd * gain[c0 + e];
    }
    put32(sm + OFF_ACT, r, c0, v);
    if (t) {
#pragma unroll
      for (int e = 0; e < 32; ++e) v[e] *= t[c0 + e];
      put32(sm + OFF_HF, r, c0, v);
    }
  }
}

// Drain this thread's 64 of 256 scratch columns: v + bias, SiLU -> bf16 into buf.
__device__ void drain_silu(uint8_t* buf, uint32_t tscr, const float* bias, int cg, int r) {
#pragma unroll 1
  for (int j = 0; j < 2; ++j) {
    const int c0 = NF_CW * cg + 32 * j;
    float v[32];
    ld32f(tscr + c0, v);
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
      v[e] += bias[c0 + e];
      v[e + 1] += bias[c0 + e + 1];
      silu2(v[e], v[e + 1]);
    }
    put32(buf, r, c0, v);
  }
}

// ---------------------------------------------------------------- the kernel
__global__ void __launch_bounds__(NF_THREADS, 1)
    net_pair_kernel(const __grid_constant__ NetMaps maps, const __grid_constant__ NetArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint32_t tmem_base;
  __shared__ volatile int abort_flag;
  Shared sh;
  sh.base = sm;
  sh.full = reinterpret_cast<uint64_t*>(sm + OFF_BAR);
  sh.empty = sh.full + NF_STAGES;
  sh.done = sh.empty + NF_STAGES;
  sh.ready = sh.done + N_EV;
  sh.abort = &abort_flag;
  float* s_ss = reinterpret_cast<float*>(sm + OFF_SS);
  float* s_dist = reinterpret_cast<float*>(sm + OFF_DIST);
  float* s_same = reinterpret_cast<float*>(sm + OFF_SAME);
  uint8_t* s_slot = sm + OFF_SLOT;
  int32_t* s_ids = reinterpret_cast<int32_t*>(sm + OFF_IDS);
  float* vec = reinterpret_cast<float*>(sm + OFF_VEC);
  uint64_t* kv_full = sh.ready + N_EV;      // per head: the peer's k, v rows have landed here
  uint64_t* kv_open = kv_full + N_KV;       // per head: the peer's buffer may take this CTA's rows
  const uint32_t rank = cluster_rank(), peer = rank ^ 1u;
  const int cid = blockIdx.x >> 1, ncl = gridDim.x >> 1;   // this cluster, clusters in the grid

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < NF_STAGES; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], 1);
    }
    for (int e = 0; e < N_EV; ++e) {
      mbar_init(&sh.done[e], 1);
      mbar_init(&sh.ready[e], NF_RW / 32);
    }
    for (int e = 0; e < N_KV; ++e) {        // one arrival per row-worker warp of the peer
      mbar_init(&kv_full[e], NF_RW / 32);
      mbar_init(&kv_open[e], NF_RW / 32);
    }
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(&tmem_base, TMEM_COLS);
  tc_fence_before();
  cluster_sync();                  // both CTAs' barriers exist before either signals the other
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  if (warp == 0 && lane == 0)      // the weight stream needs nothing from earlier launches
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  else
    pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      for (int i = 0; i < 19; ++i)
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(
                         reinterpret_cast<const CUtensorMap*>(&maps) + i))
                     : "memory");
      Producer p{&maps, &a, sh, 0u};
      for (int b = cid; b < a.B; b += ncl) schedule(a, p);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      Issuer is{&a, sh, 0u, tmem, 0u};
      for (int b = cid; b < a.B; b += ncl, is.parity ^= 1u) schedule(a, is);
    }
  } else {
    // ------------------------------------------------------------ row workers
    const int cg = (warp - 2) >> 2;                  // column group: columns 64cg .. 64cg+63
    const int q = warp & 3;                          // tensor-memory lane quarter
    const int r = q * 32 + lane;                     // node row of the tile
    const int nbase = NF_M * (int)rank;              // the tile's first node
    const int rg = nbase + r;                        // node index in the sequence
    const int wr = warp - 2;                         // row-worker warp index 0..15
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const uint32_t tx = tmem + lane_off + X_COL, tscr = tmem + lane_off + SCR_COL;
    const int L = a.L, K = a.K, LK = a.LK, nl = a.n_layers;
    const int nd = 2 * L - 1;
    const int tid = threadIdx.x - 64;
    // vectors used by every sequence: confidence-network weights (transposed to [5][D]),
    // b_c2, the final RMSNorm gain, the out / in head biases
    for (int i = tid; i < NF_D; i += NF_RW) {
#pragma unroll
      for (int j = 0; j < LILICORR_N_CONF; ++j)
        vec[V_C1W + j * NF_D + i] = a.conf1_w[i * LILICORR_N_CONF + j];
      vec[V_C1B + i] = a.conf1_b[i];
      vec[V_C2B + i] = a.conf2_b[i];
      vec[V_FIN + i] = a.final_norm[i];
    }
    for (int i = tid; i < a.d2; i += NF_RW) vec[V_BOI + i] = a.boi[i];
    for (int i = tid; i < NP_NODES; i += NF_RW) s_slot[i] = (uint8_t)min(i / K, L - 1);
    uint32_t par = 0;
    for (int b = cid; b < a.B; b += ncl, par ^= 1u) {
      for (int i = tid; i < NF_D; i += NF_RW) {           // this sequence's t and t block
        vec[V_T + i] = a.t[(size_t)b * NF_D + i];
        vec[V_CB + i] = a.cb[(size_t)b * NF_D + i];
      }
      rw_bar();
      // ---- nodes: x = fold[id] + W_h h_s + b_h + slot[s] + rank[k] + b_c2, c1 = SiLU(W_c1 f + b_c1)
      {
        const bool ok = rg < LK;
        float f[LILICORR_N_CONF] = {0.f, 0.f, 0.f, 0.f, 0.f};
        if (ok) {
          const int s = rg / K, k = rg % K;
          const size_t rk = ((size_t)b * L + s) * K;
          if (cg == 0) {                            // the node's token, read once per row
            int id = a.ids[rk + k];
            if (id < 0 || id >= a.V) {              // an id outside the vocabulary: flag, read row 0
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
        // node base rows. cp.async brings, all at once, the drafter-state rows W_h h_s + b_h,
        // the slot and rank tables (into ACT, which c1 fills afterwards) and the folded
        // embedding rows of 64 nodes at a time (into HF, 16-byte pieces XOR-swizzled by row);
        // the threads owning a row then sum it from shared memory into tensor memory.
        // rows: hproj+slot+b_c2 [L], rank [K]; the 16-byte pieces of row i XOR-swizzled by
        // i & 7, so rows read side by side (a warp's slots, its ranks) hit distinct banks
        float* tab = reinterpret_cast<float*>(sm + OFF_ACT);
        auto tab_at = [&](int row, int c) {         // c: a multiple of 4
          return tab + (size_t)row * NF_D + (((c >> 2) ^ (row & 7)) << 2);
        };
        uint8_t* stg = sm + OFF_HF;
        for (int i = tid; i < (2 * L + K) * (NF_D / 4); i += NF_RW) {
          const int row = i / (NF_D / 4), c = (i % (NF_D / 4)) * 4;
          const float* src = row < L ? a.hproj + ((size_t)b * L + row) * NF_D + c
                           : row < 2 * L ? a.slot + (size_t)(row - L) * NF_D + c
                                         : a.rank + (size_t)(row - 2 * L) * NF_D + c;
          cp_async16(tab_at(row, c), src);
        }
        rw_bar();                                   // s_ids complete
        auto fetch_fold = [&](int p) {
          for (int nloc = wr; nloc < 64; nloc += NF_RW / 32) {
            const int n = 64 * p + nloc;
            if (nbase + n >= LK) break;
            const float* src = a.fold + (size_t)s_ids[n] * NF_D + 8 * lane;
            uint8_t* row = stg + nloc * 1024;
            cp_async16(row + (((2 * lane) ^ (nloc & 7)) << 4), src);
            cp_async16(row + (((2 * lane + 1) ^ (nloc & 7)) << 4), src + 4);
          }
        };
        fetch_fold(0);
        cp_async_wait_all();
        rw_bar();
        for (int i = tid; i < L * (NF_D / 4); i += NF_RW) {   // S[s] = hproj + slot + b_c2
          const int row = i / (NF_D / 4), c = (i % (NF_D / 4)) * 4;
          float4 x = *reinterpret_cast<float4*>(tab_at(row, c));
          const float4 y = *reinterpret_cast<const float4*>(tab_at(L + row, c));
          const float4 z = *reinterpret_cast<const float4*>(vec + V_C2B + c);
          x.x += y.x + z.x; x.y += y.y + z.y; x.z += y.z + z.z; x.w += y.w + z.w;
          *reinterpret_cast<float4*>(tab_at(row, c)) = x;
        }
        rw_bar();
#pragma unroll 1
        for (int p = 0; p < 2; ++p) {
          if ((q >> 1) == p) {                      // rows 64p .. 64p+63 belong to quarters 2p, 2p+1
            const int nr = r - 64 * p;
            const uint8_t* row = stg + nr * 1024;
            const int srow = ok ? rg / K : 0, rrow = 2 * L + (ok ? rg % K : 0);
#pragma unroll 1
            for (int j = 0; j < 2; ++j) {
              const int c0 = NF_CW * cg + 32 * j;
              float v[32];
#pragma unroll
              for (int u = 0; u < 8; ++u) {
                const float4 x =
                    *reinterpret_cast<const float4*>(row + ((((c0 >> 2) + u) ^ (nr & 7)) << 4));
                const float4 y = *reinterpret_cast<const float4*>(tab_at(srow, c0 + 4 * u));
                const float4 z = *reinterpret_cast<const float4*>(tab_at(rrow, c0 + 4 * u));
                v[4 * u] = ok ? x.x + y.x + z.x : 0.f;
                v[4 * u + 1] = ok ? x.y + y.y + z.y : 0.f;
                v[4 * u + 2] = ok ? x.z + y.z + z.z : 0.f;
                v[4 * u + 3] = ok ? x.w + y.w + z.w : 0.f;
              }
              st32f(tx + c0, v);
            }
          }
          rw_bar();                                 // staging free for the next 64 nodes
          if (p == 0 && LK - nbase > 64) {
            fetch_fold(1);
            cp_async_wait_all();
            rw_bar();
          }
        }
        // c1 of this thread's row and 64 columns, 4 columns per step (ACT is free again)
#pragma unroll 1
        for (int j = 0; j < 2; ++j) {
          const int c0 = NF_CW * cg + 32 * j;
          float c1[32];
#pragma unroll
          for (int e = 0; e < 32; e += 4) {
            float4 z = *reinterpret_cast<const float4*>(vec + V_C1B + c0 + e);
#pragma unroll
            for (int i = 0; i < LILICORR_N_CONF; ++i) {
              const float4 w = *reinterpret_cast<const float4*>(vec + V_C1W + i * NF_D + c0 + e);
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
          put32(sm + OFF_ACT, r, c0, c1);
        }
        tmem_wait_st();
        rw_signal(&sh.ready[0], lane);
      }
      // ---- Transformer layers
      for (int l = 0; l < nl; ++l) {
        ev_wait(&sh.done[l == 0 ? 0 : D_LAYER(l - 1)], par, sh.abort);
        tc_fence_after();
        // this layer's vectors (the previous layer's readers are past this barrier)
        rw_bar();
        for (int i = tid; i < NF_D; i += NF_RW) {
          vec[V_AN + i] = a.an[l][i];
          vec[V_FN + i] = a.fn[l][i];
          vec[V_BO + i] = a.bo[l][i];
          vec[V_B2 + (l & 1) * NF_D + i] = a.b2[l][i];
        }
        for (int i = tid; i < NF_F; i += NF_RW) vec[V_B1 + i] = a.b1[l][i];
        for (int i = tid; i < 3 * NF_D; i += NF_RW) vec[V_BQKV + i] = a.bqkv[l][i];
        for (int i = tid; i < NF_NH * nd; i += NF_RW) s_dist[i] = a.dist[l][i] * LOG2E;
        if (tid < NF_NH) s_same[tid] = a.same[l][tid] * LOG2E;
        // x += b_2 of the previous layer (staged then), RMSNorm statistics
        const float* b2p = l == 0 ? nullptr : vec + V_B2 + ((l - 1) & 1) * NF_D;
        float rstd = row_rstd(tx, b2p, true, cg, r, s_ss);
        row_normed(sm, tx, nullptr, rstd, vec + V_AN, nullptr, cg, r);
        rw_signal(&sh.ready[R_XN(l)], lane);

        const int wr16 = wr & 7, kh = wr >> 3;           // queries 16 wr16 .., key half kh
        uint8_t* hq = sm + OFF_HF;
        for (int g = 0; g < 4; ++g) {
          ev_wait(&sh.done[D_QKV(l, g)], par, sh.abort);
          tc_fence_after();
#pragma unroll 1
          for (int e = 0; e < 2; ++e) {
            const int hh = 2 * g + e, hn = l * NF_NH + hh;   // head, and its number in the sequence
            // every warp of this CTA is done with the previous head's q, k, v (and, for the
            // first head of a layer, with the FFN's use of the buffer): the peer may now write
            // its rows of head hn here
            rw_bar();
            if (hh == 0 && lane == 0) mbar_arrive_peer(peer_addr(smem_u32(&kv_open[hn]), peer));
            // q (columns of part 0), k (part 1, bf16) and v (part 2, fp16) of head hh, biases
            // added, by column groups 0, 1, 2; the k and v rows go to the peer as well, once
            // the peer's buffer is open for this head
            const bool open = ev_wait_cluster(&kv_open[hn], par, sh.abort);
            if (cg < 3) {
              float v[32];
              ld32f(tscr + 64 * cg + 32 * e, v);
              const float* bq = vec + V_BQKV + cg * NF_D + hh * NF_HD;
              const bool zero = cg > 0 && rg >= LK;    // padded nodes (their keys are masked)
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = zero ? 0.f : v[i] + bq[i];
              uint8_t* dst = hq + (cg == 0 ? Q_OFF : cg == 1 ? K_OFF : V_OFF);
              const int row = cg == 0 ? r : rg;
#pragma unroll
              for (int p = 0; p < 4; ++p) {
                const uint4 w = cg == 2 ? pack8h(v + 8 * p) : pack8(v + 8 * p);
                uint8_t* at = dst + qkv_off(row, p);
                *reinterpret_cast<uint4*>(at) = w;
                if (cg > 0 && open) st_peer_v4(peer_addr(smem_u32(at), peer), w);
              }
            }
            // both heads of the pair drained: the scratch accumulator may take the next pair
            if (e == 1 && g < 3) rw_signal(&sh.ready[R_QKV_DRAINED(l, g)], lane);
            // publish this warp's rows to the peer, then wait for the peer's rows
            fence_cluster();
            __syncwarp();
            if (lane == 0) mbar_arrive_peer(peer_addr(smem_u32(&kv_full[hn]), peer));
            ev_wait_cluster(&kv_full[hn], par, sh.abort);
            rw_bar();
            // this warp's 16 queries over its half of the keys
            float o[4][4], m0, m1, l0, l1;
            head_attention_part(smem_u32(hq + Q_OFF), smem_u32(hq + K_OFF), smem_u32(hq + V_OFF),
                                NF_M * kh, NF_M, LK, K, s_slot, s_dist + hh * nd + (L - 1),
                                s_same[hh], 16 * wr16, nbase, lane, o, m0, m1, l0, l1);
            // every warp is done with q, k and v of head hh: k and v may take the peer's rows
            // of the next head of the layer while the two key halves merge. The second-half
            // warp parks its state (outputs as fp16 pairs: |o| <= the sum of the half's
            // weights times max |v|, far inside fp16's range; then its maxima and sums) in the
            // q rows and the free 8 KB after v: word j of thread (pair wr16, lane) at
            // park[j][32 wr16 + lane]; the first-half warp of the same queries combines.
            rw_bar();
            if (hh < NF_NH - 1 && lane == 0)
              mbar_arrive_peer(peer_addr(smem_u32(&kv_open[hn + 1]), peer));
            uint32_t* park_o = reinterpret_cast<uint32_t*>(hq + Q_OFF);           // 8 words
            float* park_s = reinterpret_cast<float*>(hq + V_OFF + 16384);         // 4 words
            const int slot_ = 32 * wr16 + lane;
            if (kh == 1) {
#pragma unroll
              for (int nb = 0; nb < 4; ++nb) {
                park_o[(2 * nb) * 256 + slot_] = pack_h2(o[nb][0], o[nb][1]);
                park_o[(2 * nb + 1) * 256 + slot_] = pack_h2(o[nb][2], o[nb][3]);
              }
              park_s[0 * 256 + slot_] = m0;
              park_s[1 * 256 + slot_] = m1;
              park_s[2 * 256 + slot_] = l0;
              park_s[3 * 256 + slot_] = l1;
            }
            rw_bar();
            if (kh == 0) {
              float ot[16], mt[4];
#pragma unroll
              for (int nb = 0; nb < 4; ++nb) {
                const float2 a01 = h2_to_f2(park_o[(2 * nb) * 256 + slot_]);
                const float2 a23 = h2_to_f2(park_o[(2 * nb + 1) * 256 + slot_]);
                ot[4 * nb + 0] = a01.x; ot[4 * nb + 1] = a01.y;
                ot[4 * nb + 2] = a23.x; ot[4 * nb + 3] = a23.y;
              }
#pragma unroll
              for (int j = 0; j < 4; ++j) mt[j] = park_s[j * 256 + slot_];
              const float M0 = fmaxf(m0, mt[0]), M1 = fmaxf(m1, mt[1]);
              const float a0 = ex2f(m0 - M0), b0 = ex2f(mt[0] - M0);
              const float a1 = ex2f(m1 - M1), b1 = ex2f(mt[1] - M1);
              const float inv0 = 1.0f / (l0 * a0 + mt[2] * b0);
              const float inv1 = 1.0f / (l1 * a1 + mt[3] * b1);
              // the attention-output buffer is free once the previous pair's W_o product ran
              if (g > 0 && e == 0) ev_wait(&sh.done[D_WO(l, g - 1)], par, sh.abort);
              uint8_t* att = sm + OFF_ATT;
              const int i0 = 16 * wr16 + (lane >> 2), i1 = i0 + 8, t4 = lane & 3;
#pragma unroll
              for (int nb = 0; nb < 4; ++nb) {
                const int piece = 4 * e + nb;
                const float y0 = (o[nb][0] * a0 + ot[4 * nb + 0] * b0) * inv0;
                const float y1 = (o[nb][1] * a0 + ot[4 * nb + 1] * b0) * inv0;
                const float y2 = (o[nb][2] * a1 + ot[4 * nb + 2] * b1) * inv1;
                const float y3 = (o[nb][3] * a1 + ot[4 * nb + 3] * b1) * inv1;
                *reinterpret_cast<uint32_t*>(att + swz(i0, piece) + 4 * t4) = pack_bf16x2(y0, y1);
                *reinterpret_cast<uint32_t*>(att + swz(i1, piece) + 4 * t4) = pack_bf16x2(y2, y3);
              }
            }
          }
          rw_signal(&sh.ready[R_ATT(l, g)], lane);
        }
        // ---- FFN: x += b_o, xn2 = RMSNorm(x)
        ev_wait(&sh.done[D_WO(l, 3)], par, sh.abort);
        tc_fence_after();
        rstd = row_rstd(tx, vec + V_BO, true, cg, r, s_ss);
        row_normed(sm, tx, nullptr, rstd, vec + V_FN, nullptr, cg, r);
        rw_signal(&sh.ready[R_XN2(l)], lane);
        ev_wait(&sh.done[D_FFN(l, 0)], par, sh.abort);
        tc_fence_after();
        drain_silu(sm + OFF_HF, tscr, vec + V_B1, cg, r);
        rw_signal(&sh.ready[R_HFA(l)], lane);
        ev_wait(&sh.done[D_FFN(l, 1)], par, sh.abort);
        tc_fence_after();
        drain_silu(sm + OFF_ACT, tscr, vec + V_B1 + 256, cg, r);
        rw_signal(&sh.ready[R_HFB(l)], lane);
      }
      // ---- fusion: xf = RMSNorm(x + b_2) -> ACT, xf * t -> HF; u = SiLU(. + cb) -> ACT
      ev_wait(&sh.done[D_LAYER(nl - 1)], par, sh.abort);
      tc_fence_after();
      {
        const float* b2l = vec + V_B2 + ((nl - 1) & 1) * NF_D;
        const float rstd = row_rstd(tx, b2l, false, cg, r, s_ss);
        row_normed(sm, tx, b2l, rstd, vec + V_FIN, vec + V_T, cg, r);
      }
      rw_signal(&sh.ready[lb(nl)], lane);
      ev_wait(&sh.done[lb(nl)], par, sh.abort);
      tc_fence_after();
      drain_silu(sm + OFF_ACT, tscr, vec + V_CB, cg, r);
      rw_signal(&sh.ready[lb(nl) + 1], lane);
      // ---- out / in heads: 256 columns of [o | i] at a time -> oi (fp32, not yet unit).
      // Each 128-column half goes through a staging buffer (128 rows x 128 floats, pieces
      // swizzled by row) so that the global stores are row-contiguous.
      for (int h = 0; h * 256 < a.d2; ++h) {
        ev_wait(&sh.done[lb(nl) + 1 + h], par, sh.abort);
        tc_fence_after();
        uint8_t* stg = sm + OFF_HF;
#pragma unroll 1
        for (int hs = 0; hs < 2; ++hs) {
          if ((cg >> 1) == hs) {
#pragma unroll 1
            for (int j = 0; j < 2; ++j) {
              const int cl = 64 * (cg & 1) + 32 * j;          // column inside the 128 staged
              float v[32];
              ld32f(tscr + 128 * hs + cl, v);
              const float* bo = vec + V_BOI + 256 * h + 128 * hs + cl;
#pragma unroll
              for (int u = 0; u < 8; ++u)
                *reinterpret_cast<float4*>(stg + r * 512 + ((((cl >> 2) + u) ^ (r & 7)) << 4)) =
                    make_float4(v[4 * u] + bo[4 * u], v[4 * u + 1] + bo[4 * u + 1],
                                v[4 * u + 2] + bo[4 * u + 2], v[4 * u + 3] + bo[4 * u + 3]);
            }
          }
          rw_bar();
          for (int row = wr; row < min(NF_M, LK - nbase); row += NF_RW / 32)
            *reinterpret_cast<float4*>(a.oi + ((size_t)b * LK + nbase + row) * a.d2 + 256 * h +
                                       128 * hs + 4 * lane) =
                *reinterpret_cast<const float4*>(stg + row * 512 + ((lane ^ (row & 7)) << 4));
          rw_bar();
        }
        if ((h + 1) * 256 < a.d2) rw_signal(&sh.ready[lb(nl) + 2 + h], lane);
      }
      tc_fence_before();
      rw_bar();                                      // s_dist / s_ss / vectors reuse by the next sequence
    }
  }

  // ---- teardown (no CTA leaves while its peer may still write to or signal it)
  tc_fence_before();
  cluster_sync();
  if (abort_flag) {
    if (threadIdx.x == 0) {
      set_status(a.status, LILICORR_ERR_TIMEOUT);
      const long long t0 = clock64();            // let copies and products in flight land
      while (clock64() - t0 < WAIT_LIMIT / 10) {
      }
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

}  // namespace

// ----------------------------------------------------------------------------- host side
struct NetPairMaps {
  NetMaps m;
};

bool net_pair_supported(const lilicorr_head_desc& d) {
  return d.dtype == LILICORR_BF16 && d.D == NF_D && d.ffn == NF_F && d.n_heads == NF_NH &&
         d.n_layers >= 1 && d.n_layers <= NF_MAX_LAYERS && d.L >= 1 && d.L <= NF_MAX_L &&
         d.K >= 1 && d.L * d.K > NF_M && d.L * d.K <= NP_NODES &&
         2 * d.L + d.K <= 64 &&                     // node tables fit in ACT
         (2 * d.d) % 256 == 0 && 2 * d.d <= 512 &&
         encode_fn() != nullptr;
}

namespace {
// W [rows, cols] bf16 row-major as (64, rows, cols / 64): box (64, box_rows, 1) is one K chunk
// of box_rows rows, 128-byte swizzled.
bool chunk_map(CUtensorMap* m, const void* W, int rows, int cols, int box_rows) {
  const uint64_t dims[3] = {64, (uint64_t)rows, (uint64_t)(cols / 64)};
  const uint64_t strides[3] = {2, (uint64_t)cols * 2, 128};
  const uint32_t box[3] = {64, (uint32_t)box_rows, 1};
  return make_map_nd(m, W, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, dims, strides, box);
}
// W_qkv [3D, D] as (64 k, 64 rows, 4 head pairs, 3 parts q/k/v, D / 64 chunks): box
// (64, 64, 1, 3, 1) brings the q, k and v rows of one head pair for one K chunk.
bool qkv_map(CUtensorMap* m, const void* W) {
  const uint64_t dims[5] = {64, 64, NF_D / 64, 3, NF_D / 64};
  const uint64_t strides[5] = {2, NF_D * 2, 64ull * NF_D * 2, (uint64_t)NF_D * NF_D * 2, 128};
  const uint32_t box[5] = {64, 64, 1, 3, 1};
  return make_map_nd(m, W, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, dims, strides, box);
}

cudaLaunchConfig_t pair_config(int clusters, cudaStream_t st, cudaLaunchAttribute (&attr)[2]) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * clusters);
  cfg.blockDim = dim3(NF_THREADS);
  cfg.dynamicSmemBytes = NF_SMEM;
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cfg;
}
}  // namespace

void* net_pair_maps_create(const lilicorr_head* h) {
  const lilicorr_head_desc& d = h->desc;
  if (!net_pair_supported(d)) return nullptr;
  NetPairMaps* nm = new (std::nothrow) NetPairMaps;
  if (!nm) return nullptr;
  memset(nm, 0, sizeof(*nm));
  bool ok = chunk_map(&nm->m.conf2, h->conf2_w, NF_D, NF_D, 256) &&
            chunk_map(&nm->m.fuse, h->fuse_x, NF_D, 2 * NF_D, 256) &&
            chunk_map(&nm->m.woi, h->woi, 2 * d.d, NF_D, 256);
  for (int l = 0; l < d.n_layers && ok; ++l) {
    const HeadW& w = h->layer[l];
    ok = qkv_map(&nm->m.wqkv[l], w.wqkv) && chunk_map(&nm->m.wo[l], w.wo, NF_D, NF_D, 256) &&
         chunk_map(&nm->m.w1[l], w.w1, NF_F, NF_D, 256) &&
         chunk_map(&nm->m.w2[l], w.w2, NF_D, NF_F, 256);
  }
  for (int l = d.n_layers; l < NF_MAX_LAYERS && ok; ++l) {   // unused slots: valid maps
    nm->m.wqkv[l] = nm->m.wqkv[0];
    nm->m.wo[l] = nm->m.wo[0];
    nm->m.w1[l] = nm->m.w1[0];
    nm->m.w2[l] = nm->m.w2[0];
  }
  if (!ok) {
    delete nm;
    return nullptr;
  }
  return nm;
}

void net_pair_maps_free(void* p) { delete static_cast<NetPairMaps*>(p); }

// Clusters of this kernel that fit on the current device at once (0 if it cannot run).
int net_pair_capacity() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    (void)cudaGetLastError();
    return 0;
  }
  if (cache[dev]) return cache[dev] > 0 ? cache[dev] : 0;
  static bool configured[64] = {false};
  int n = 0;
  if (allow_max_dynamic_smem(net_pair_kernel, configured) == LILICORR_OK) {
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = pair_config(64, nullptr, attr);
    cfg.numAttrs = 1;                                   // the cluster shape only
    if (cudaOccupancyMaxActiveClusters(&n, net_pair_kernel, &cfg) != cudaSuccess) n = 0;
  }
  (void)cudaGetLastError();
  cache[dev] = n > 0 ? n : -1;
  return n > 0 ? n : 0;
}

lilicorr_status_t launch_net_pair(const lilicorr_head* h, int B, const int32_t* ids,
                                  const float* logp, const float* hproj, const float* t,
                                  const float* cb, float* oi, uint32_t* status, cudaStream_t st) {
  if (B == 0) return LILICORR_OK;
  const NetPairMaps* nm = static_cast<const NetPairMaps*>(h->pair_maps);
  if (!nm) return LILICORR_ERR_SHAPE;
  const int cap = net_pair_capacity();
  if (cap <= 0) return LILICORR_ERR_CUDA;
  const lilicorr_head_desc& d = h->desc;
  NetArgs a;
  memset(&a, 0, sizeof(a));
  a.B = B; a.L = d.L; a.K = d.K; a.LK = d.L * d.K; a.V = d.V; a.n_layers = d.n_layers;
  a.d2 = 2 * d.d;
  a.ids = ids; a.logp = logp; a.hproj = hproj; a.t = t; a.cb = cb;
  a.fold = static_cast<const float*>(h->fold);
  a.slot = h->slot; a.rank = h->rank;
  a.conf1_w = h->conf1_w; a.conf1_b = h->conf1_b; a.conf2_b = h->conf2_b;
  for (int l = 0; l < NF_MAX_LAYERS; ++l) {
    const HeadW& w = h->layer[l < d.n_layers ? l : 0];
    a.bqkv[l] = w.bqkv; a.bo[l] = w.bo; a.b1[l] = w.b1; a.b2[l] = w.b2;
    a.an[l] = w.an; a.fn[l] = w.fn; a.dist[l] = w.dist; a.same[l] = w.same;
  }
  a.final_norm = h->final_norm;
  a.boi = h->boi;
  a.oi = oi;
  a.status = status;
  static bool configured[64] = {false};
  LL_TRY(allow_max_dynamic_smem(net_pair_kernel, configured));
  cudaLaunchAttribute attr[2];
  const cudaLaunchConfig_t cfg = pair_config(B < cap ? B : cap, st, attr);
  count_launch();
  LL_CUDA_TRY(cudaLaunchKernelEx(&cfg, net_pair_kernel, nm->m, a));
  return LILICORR_OK;
}

}  // namespace lilicorr
