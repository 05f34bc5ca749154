// C ABI of the selection path: argument checks, the head's device layout, the
// workspace layout and the launch sequence of each entry point.
#include <stdlib.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "internal.cuh"
#include "lilicorr_testing.h"

namespace lilicorr {

size_t attention_smem_bytes(int LK, int hd, int warps);
size_t pair_walk_smem_bytes(int L, int K, int d);

static std::atomic<uint64_t> g_launches{0};
int g_fused_enabled = 1;
// The chain's attention core: 0 the mma.sync kernel, 1 the tcgen05 kernel wherever it
// applies, 2 (the default) the tcgen05 kernel on full 256-node tiles with slots in 8-node
// groups (where it was measured faster: 104 against 179 us per launch at 256 sequences x
// 8 heads of 64), the mma.sync kernel elsewhere.
int g_attn_umma = 2;
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int num_sms() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev >= 0 && dev < 64 && cache[dev]) return cache[dev];
  int n = 148;
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  if (dev >= 0 && dev < 64) cache[dev] = n;
  return n;
}

namespace {

size_t esize(lilicorr_dtype_t t) { return t == LILICORR_BF16 ? 2 : 4; }

bool desc_ok(const lilicorr_head_desc* d) {
  if (!d) return false;
  if (d->dtype != LILICORR_F32 && d->dtype != LILICORR_BF16) return false;
  if (d->H <= 0 || d->D <= 0 || d->d <= 0 || d->n_heads <= 0 || d->ffn <= 0) return false;
  if (d->n_layers <= 0 || d->n_layers > 8 || d->n_tgt <= 0) return false;
  if (d->L <= 0 || d->L > LILICORR_MAX_L || d->K <= 0 || d->K > LILICORR_MAX_K) return false;
  if (d->K > d->V || d->L * d->K > LILICORR_MAX_NODES) return false;
  if (d->D % d->n_heads != 0 || d->D / d->n_heads > 128 || (d->D / d->n_heads) % 4 != 0)
    return false;
  // every row handed to a linear layer or a TMA copy stays 16-byte aligned
  if (d->H % 8 != 0 || d->D % 8 != 0 || d->d % 8 != 0 || d->ffn % 8 != 0) return false;
  if (attention_smem_bytes(d->L * d->K, d->D / d->n_heads, 8) > 200 * 1024) return false;
  if (pair_walk_smem_bytes(d->L, d->K, d->d) > 200 * 1024) return false;
  return true;
}

// Element offsets of each tensor in the weight blob (the order documented in lilicorr.h).
struct BlobIndex {
  size_t emb_w, emb_b, hid_w, hid_b, conf1_w, conf1_b, conf2_w, conf2_b, slot, rank;
  size_t tgt_norm, tgt_w, tgt_b;
  struct Layer {
    size_t an, wq, bq, wk, bk, wv, bv, wo, bo, dist, same, fn, w1, b1, w2, b2;
  } layer[8];
  size_t final_norm, fuse_w, fuse_b, out_w, out_b, in_w, in_b, anc_w, anc_b;
  size_t total;
};

BlobIndex blob_index(const lilicorr_head_desc& d) {
  BlobIndex b;
  size_t o = 0;
  auto take = [&](size_t n) { size_t r = o; o += n; return r; };
  const size_t D = d.D, H = d.H, F = d.ffn, dd = d.d;
  b.emb_w = take(D * H); b.emb_b = take(D);
  b.hid_w = take(D * H); b.hid_b = take(D);
  b.conf1_w = take(D * LILICORR_N_CONF); b.conf1_b = take(D);
  b.conf2_w = take(D * D); b.conf2_b = take(D);
  b.slot = take((size_t)d.L * D); b.rank = take((size_t)d.K * D);
  b.tgt_norm = take(H); b.tgt_w = take(D * H); b.tgt_b = take(D);
  for (int i = 0; i < d.n_layers; ++i) {
    BlobIndex::Layer& l = b.layer[i];
    l.an = take(D);
    l.wq = take(D * D); l.bq = take(D); l.wk = take(D * D); l.bk = take(D);
    l.wv = take(D * D); l.bv = take(D); l.wo = take(D * D); l.bo = take(D);
    l.dist = take((size_t)d.n_heads * (2 * d.L - 1)); l.same = take(d.n_heads);
    l.fn = take(D);
    l.w1 = take(F * D); l.b1 = take(F); l.w2 = take(D * F); l.b2 = take(D);
  }
  b.final_norm = take(D);
  b.fuse_w = take(D * 3 * D); b.fuse_b = take(D);
  b.out_w = take(dd * D); b.out_b = take(dd);
  b.in_w = take(dd * D); b.in_b = take(dd);
  b.anc_w = take(dd * D); b.anc_b = take(dd);
  b.total = o;
  return b;
}

// Host staging of the device pool: matrices keep the head dtype, vectors become fp32.
struct Stager {
  lilicorr_dtype_t dt;
  const unsigned char* blob;
  std::vector<unsigned char> host;
  size_t off = 0;
  size_t alloc(size_t bytes) {
    off = align_up(off, 256);
    size_t r = off;
    off += bytes;
    if (host.size() < off) host.resize(off);
    return r;
  }
  float elem_f32(size_t i) const {
    if (dt == LILICORR_F32) { float f; memcpy(&f, blob + 4 * i, 4); return f; }
    uint16_t h; memcpy(&h, blob + 2 * i, 2);
    uint32_t u = (uint32_t)h << 16; float f; memcpy(&f, &u, 4); return f;
  }
  // copy rows [r0, r0+nr) x cols [c0, c0+nc) of a row-major [*, ld] blob matrix at `src`
  void put_mat(size_t dst, size_t src, size_t ld, size_t r0, size_t nr, size_t c0, size_t nc,
               size_t dst_ld, size_t dst_c0) {
    const size_t es = esize(dt);
    for (size_t r = 0; r < nr; ++r)
      memcpy(&host[dst + (r * dst_ld + dst_c0) * es], blob + (src + (r0 + r) * ld + c0) * es, nc * es);
  }
  size_t mat(size_t src, size_t rows, size_t cols) {
    size_t dst = alloc(rows * cols * esize(dt));
    put_mat(dst, src, cols, 0, rows, 0, cols, cols, 0);
    return dst;
  }
  size_t vec(size_t src, size_t n) {
    size_t dst = alloc(n * 4);
    for (size_t i = 0; i < n; ++i) { float f = elem_f32(src + i); memcpy(&host[dst + 4 * i], &f, 4); }
    return dst;
  }
  size_t vec_cat(std::initializer_list<std::pair<size_t, size_t>> parts) {
    size_t n = 0;
    for (auto& p : parts) n += p.second;
    size_t dst = alloc(n * 4), o = 0;
    for (auto& p : parts)
      for (size_t i = 0; i < p.second; ++i, ++o) {
        float f = elem_f32(p.first + i);
        memcpy(&host[dst + 4 * o], &f, 4);
      }
    return dst;
  }
};

}  // namespace

// ----------------------------------------------------------------------------- workspace
WsLayout ws_layout(const lilicorr_head_desc& d, int B) {
  WsLayout w;
  const size_t R = (size_t)B * d.L, N = R * d.K, Np = align_up(N, 128);
  const TopkPlan p = topk_plan((int)R, d.V, d.K, d.dtype);
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t r = o; o = align_up(o + bytes, 256); return r; };
  w.status = take(256);
  w.counters = take(R * 4);
  w.partials = take(R * p.pieces * p.rec_bytes);
  w.ids = take(N * 4); w.logp = take(N * 4); w.lse = take(R * 4);
  w.hproj = take(R * d.D * 4);
  w.tn = take((size_t)B * d.H * 4);
  w.t = take((size_t)B * d.D * 4);
  w.anc = take((size_t)B * d.d * 4);
  w.cb = take((size_t)B * d.D * 4);
  w.x = take(Np * d.D * 4);
  w.c1 = take(Np * d.D * 4);
  w.xn = take(Np * 2 * d.D * 4);
  w.qkv = take(Np * 3 * d.D * 4);
  w.att = take(Np * d.D * 4);
  w.hf = take(Np * d.ffn * 4);
  w.u = take(Np * d.D * 4);
  w.oi = take(Np * 2 * d.d * 4);
  w.A = take((size_t)B * d.K * 4);
  w.P = take((size_t)B * (d.L > 1 ? d.L - 1 : 0) * d.K * d.K * 4);
  w.choice = take(R * 4);
  w.pw_counters = take((size_t)B * 4);
  w.ss = take(Np * SS_LD * 4);
  w.total = o;
  return w;
}

}  // namespace lilicorr

using namespace lilicorr;

namespace {

template <typename T> T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<unsigned char*>(ws) + off);
}

GemmArgs gemm(const void* A, lilicorr_dtype_t a_dt, int lda, const void* W, lilicorr_dtype_t w_dt,
              int ldw, void* C, lilicorr_dtype_t c_dt, int ldc, int M, int N, int Kd) {
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.A = A; g.a_dt = a_dt; g.lda = lda;
  g.W = W; g.w_dt = w_dt; g.ldw = ldw;
  g.C = C; g.c_dt = c_dt; g.ldc = ldc;
  g.M = M; g.N = N; g.Kd = Kd;
  g.rows_per_bias = 1;
  return g;
}

// Few rows: split-N CUDA-core kernel. bf16 operands: tensor cores. Otherwise the
// tiled fp32 CUDA-core kernel (the fp32 head keeps fp32 arithmetic throughout).
// The persistent tensor-core kernel is the one run_gemm picks for g.
bool takes_gemm_tc(const GemmArgs& g) {
  return !(g.M <= 64 || (g.a_dt == LILICORR_F32 && g.M <= 1024)) && !gemm_small_supported(g) &&
         gemm_tc_supported(g);
}

lilicorr_status_t run_gemm(const GemmArgs& g, cudaStream_t st) {
  // a folded RMSNorm only exists in the persistent tensor-core kernel
  if (g.c2 || g.ss_in) return takes_gemm_tc(g) ? launch_gemm_tc(g, st) : LILICORR_ERR_SHAPE;
  // fp32 activations (the tensor-core kernels take bf16) at per-sequence row counts above
  // 16: 16 x 32 output blocks with the rows staged (256 x 512 x 512: 54 -> ~5 us); few rows
  // otherwise: the split-N kernel spreads the weights over many CTAs
  if (g.a_dt == LILICORR_F32 && g.M > 16 && g.M <= 1024 && gemm_rows_supported(g))
    return launch_gemm_rows(g, st);
  if (g.M <= 64 || (g.a_dt == LILICORR_F32 && g.M <= 1024)) return launch_gemm_skinny(g, st);
  if (gemm_small_supported(g)) return launch_gemm_small(g, st);
  if (gemm_tc_supported(g)) return launch_gemm_tc(g, st);
  return launch_gemm_simt(g, st);
}

// Views of one call's workspace buffers and the per-call kernel choices.
struct HeadCall {
  const lilicorr_head* h;
  const lilicorr_head_desc& d;
  int B, R, N, LK, D, F;
  lilicorr_dtype_t wdt, adt, qkv_dt;     // weights; matrix-product operands; q|k|v buffer
  bool tc_attn;                          // tensor-core attention core
  uint32_t* status;
  lilicorr_dtype_t tn_dt;                // normalised target state (an operand of W_t)
  float *hproj, *t, *anc, *cb, *x, *oi, *ss;
  void *tn, *c1, *xn, *qkv, *att, *hf, *u;

  HeadCall(const lilicorr_head* head, int b, void* ws, const WsLayout& w)
      : h(head), d(head->desc), B(b) {
    R = B * d.L;
    N = R * d.K;
    LK = d.L * d.K;
    D = d.D;
    F = d.ffn;
    wdt = d.dtype;
    adt = d.dtype;                       // bf16 operands on the bf16 head
    const int hd = D / d.n_heads;
    tc_attn = wdt == LILICORR_BF16 && attention_tc_supported(hd) &&
              attention_tc_smem_bytes(LK, hd, d.L) <= 200 * 1024;
    qkv_dt = tc_attn ? LILICORR_BF16 : LILICORR_F32;
    status = at<uint32_t>(ws, w.status);
    hproj = at<float>(ws, w.hproj);
    tn = at<void>(ws, w.tn);
    // rows up to 16384 are normalised in registers; longer ones pass through tn in fp32
    tn_dt = d.H <= 16384 ? wdt : LILICORR_F32;
    t = at<float>(ws, w.t);
    anc = at<float>(ws, w.anc);
    cb = at<float>(ws, w.cb);
    x = at<float>(ws, w.x);
    oi = at<float>(ws, w.oi);
    ss = at<float>(ws, w.ss);
    c1 = at<void>(ws, w.c1);
    xn = at<void>(ws, w.xn);
    qkv = at<void>(ws, w.qkv);
    att = at<void>(ws, w.att);
    hf = at<void>(ws, w.hf);
    u = at<void>(ws, w.u);
  }
  GemmArgs G(const void* A, lilicorr_dtype_t a_dt, int lda, const void* W, int ldw, void* C,
             lilicorr_dtype_t c_dt, int ldc, int M, int Nn, int Kd) const {
    GemmArgs g = gemm(A, a_dt, lda, W, wdt, ldw, C, c_dt, ldc, M, Nn, Kd);
    g.status = status;
    return g;
  }
  // RMSNorm folded around a product (App. A's pre-norm x / rms(x) * gain): the product
  // writing the fp32 state also writes bf16(state * gain) into xn and its row sums of
  // squares; the next product reads xn and scales its rows by 1 / rms.
  void norm_out(GemmArgs& g, const float* gain) const {
    g.c2 = xn; g.ldc2 = D; g.c2_gain = gain; g.ss_out = ss;
  }
  void norm_in(GemmArgs& g) const {
    g.ss_in = ss; g.ss_slots = gemm_tc_ss_slots(N, D); g.ss_dim = D;
  }
  // the final norm into the fusion layer's input [x; x*t] (App. A), both blocks at once:
  // xn [N, 2D] receives bf16(state * gain) and bf16(state * gain * t of the sequence)
  void final_norm_out(GemmArgs& g, const float* gain) const {
    norm_out(g, gain);
    g.C = nullptr;               // nothing reads the last state itself
    g.ldc2 = 2 * D;
    g.c3 = static_cast<__nv_bfloat16*>(xn) + D;
    g.c3_t = t;
    g.c3_rows_per = LK;
  }
};

// Candidate-independent part of the scoring network (Sec. 3.2; App. A), two chains.
// (a) the drafter state projection W_h h_s + b_h, one row per slot.
lilicorr_status_t run_drafter_proj(const HeadCall& c, const void* hidden, cudaStream_t st) {
  const lilicorr_head* h = c.h;
  const lilicorr_head_desc& d = c.d;
  GemmArgs g = c.G(hidden, c.wdt, d.H, h->hid_w, d.H, c.hproj, LILICORR_F32, c.D, c.R, c.D, d.H);
  g.bias = h->hid_b;
  return run_gemm(g, st);
}
// (b) the target state t = W_t RMSNorm(mean of the captured layers) + b_t, then two
// independent products of t: the anchor out vector W_a t + b_a (its consumers normalise
// it) and the fusion layer's t block, constant per sequence: cb = W_f[:, t] t + b_f.
lilicorr_status_t run_target(const HeadCall& c, const void* target, cudaStream_t st) {
  const lilicorr_head* h = c.h;
  const lilicorr_head_desc& d = c.d;
  const lilicorr_dtype_t F32 = LILICORR_F32;
  const int D = c.D;
  LL_TRY(launch_target_norm(target, c.wdt, c.B, d.n_tgt, d.H, h->tgt_norm, c.tn, c.tn_dt, st));
  GemmArgs g = c.G(c.tn, c.tn_dt, d.H, h->tgt_w, d.H, c.t, F32, D, c.B, D, d.H);
  g.bias = h->tgt_b;
  return run_gemm(g, st);
}
lilicorr_status_t run_anchor(const HeadCall& c, cudaStream_t st) {
  GemmArgs g = c.G(c.t, LILICORR_F32, c.D, c.h->anc_w, c.D, c.anc, LILICORR_F32, c.d.d, c.B,
                   c.d.d, c.D);
  g.bias = c.h->anc_b;
  return run_gemm(g, st);
}
lilicorr_status_t run_fusion_t(const HeadCall& c, cudaStream_t st) {
  GemmArgs g = c.G(c.t, LILICORR_F32, c.D, c.h->fuse_t, c.D, c.cb, LILICORR_F32, c.D, c.B, c.D,
                   c.D);
  g.bias = c.h->fuse_b;
  return run_gemm(g, st);
}
// Fork both chains from `st` onto the head's side streams; join_prologue makes `st` wait
// for them. The joins are recorded even when a launch fails, so a capture stays balanced.
lilicorr_status_t fork_prologue(const HeadCall& c, const void* hidden, const void* target,
                                cudaStream_t st) {
  lilicorr_head* hm = const_cast<lilicorr_head*>(c.h);
  LL_CUDA_TRY(cudaEventRecord(hm->ev_fork, st));
  LL_CUDA_TRY(cudaStreamWaitEvent(hm->side, hm->ev_fork, 0));
  LL_CUDA_TRY(cudaStreamWaitEvent(hm->side2, hm->ev_fork, 0));
  // side: drafter-state projection, then (once t exists) the fusion layer's t block;
  // side2: the target state, then the anchor vector
  lilicorr_status_t s1 = run_drafter_proj(c, hidden, hm->side);
  lilicorr_status_t s2 = run_target(c, target, hm->side2);
  LL_CUDA_TRY(cudaEventRecord(hm->ev_t, hm->side2));
  LL_CUDA_TRY(cudaStreamWaitEvent(hm->side, hm->ev_t, 0));
  if (s1 == LILICORR_OK) s1 = run_fusion_t(c, hm->side);
  if (s2 == LILICORR_OK) s2 = run_anchor(c, hm->side2);
  LL_CUDA_TRY(cudaEventRecord(hm->ev_join, hm->side));
  LL_CUDA_TRY(cudaEventRecord(hm->ev_join2, hm->side2));
  return s1 != LILICORR_OK ? s1 : s2;
}
lilicorr_status_t join_prologue(const lilicorr_head* h, cudaStream_t st) {
  LL_CUDA_TRY(cudaStreamWaitEvent(st, h->ev_join, 0));
  LL_CUDA_TRY(cudaStreamWaitEvent(st, h->ev_join2, 0));
  return LILICORR_OK;
}

// Whether every product around the chain's RMSNorms takes the persistent tensor-core
// kernel (the only one that folds a norm): bf16 heads with more node rows than one tile.
bool fold_norms(const HeadCall& c) {
  const lilicorr_head* h = c.h;
  const int D = c.D, F = c.F, N = c.N;
  const lilicorr_dtype_t adt = c.adt, F32 = LILICORR_F32;
  if (c.wdt != LILICORR_BF16) return false;
  GemmArgs p[7] = {c.G(c.c1, adt, D, h->conf2_w, D, c.x, F32, D, N, D, D),
                   c.G(c.xn, adt, D, h->layer[0].wqkv, D, c.qkv, c.qkv_dt, 3 * D, N, 3 * D, D),
                   c.G(c.att, adt, D, h->layer[0].wo, D, c.x, F32, D, N, D, D),
                   c.G(c.xn, adt, D, h->layer[0].w1, D, c.hf, adt, F, N, F, D),
                   c.G(c.hf, adt, F, h->layer[0].w2, F, c.x, F32, D, N, D, F),
                   c.G(c.hf, adt, F, h->layer[0].w2, F, c.x, F32, D, N, D, F),
                   c.G(c.xn, adt, 2 * D, h->fuse_x, 2 * D, c.u, adt, D, N, D, 2 * D)};
  for (int i : {0, 2, 4, 5}) {
    p[i].residual = c.x; p[i].ldr = D;
    c.norm_out(p[i], h->layer[0].an);
  }
  c.final_norm_out(p[5], h->final_norm);
  p[6].bias_rows = c.cb; p[6].rows_per_bias = c.LK; p[6].act = ACT_SILU;
  for (int i : {1, 3, 6}) c.norm_in(p[i]);
  for (const GemmArgs& g : p)
    if (!takes_gemm_tc(g)) return false;
  return true;
}

// Candidate-dependent part, after the prologue: nodes, the Transformer, fusion and the
// out/in heads. Writes oi = [W_o u + b_o | W_i u + b_i] (not yet normalised).
// With `tail`, the cluster kernel also forms the pair scores and walks; *tail_done says
// whether it did (otherwise the caller launches the pair kernel).
lilicorr_status_t run_body(const HeadCall& c, const int32_t* ids, const float* logp,
                           cudaStream_t st, const ClusterTail* tail = nullptr,
                           bool* tail_done = nullptr) {
  if (tail_done) *tail_done = false;
  const lilicorr_head* h = c.h;
  const lilicorr_head_desc& d = c.d;
  const lilicorr_dtype_t F32 = LILICORR_F32, adt = c.adt;
  const int D = c.D, F = c.F, N = c.N;
  // Network kernels: a cluster of four SMs per sequence while every sequence's cluster
  // fits on the GPU at once; beyond that one SM per sequence (fewer waves); the chain of
  // kernels below, each spread over SMs, for heads neither kernel takes.
  const bool cluster = h->cluster_maps &&
                       (g_fused_enabled == 3 ||
                        (g_fused_enabled == 1 && c.B <= net_cluster_capacity()));
  if (cluster) {
    if (tail_done) *tail_done = tail != nullptr;
    return launch_net_cluster(h, c.B, ids, logp, c.hproj, c.t, c.cb, c.oi, c.status, st, tail);
  }
  if (h->net_maps && (g_fused_enabled == 2 || (g_fused_enabled == 1 && c.B >= FUSED_MIN_B)))
    return launch_net_fused(h, c.B, ids, logp, c.hproj, c.t, c.cb, c.oi, c.status, st);
  // 129-256 nodes per sequence: two CTAs per sequence, one 128-node tile each
  if (h->pair_maps && g_fused_enabled != 0)
    return launch_net_pair(h, c.B, ids, logp, c.hproj, c.t, c.cb, c.oi, c.status, st);
  // nodes: x = fold[id] + hproj + slot + rank, then x += W_c2 c1 + b_c2
  LL_TRY(launch_node_build(h, c.B, ids, logp, c.hproj, c.c1, adt, c.x, c.status, st));
  GemmArgs g = c.G(c.c1, adt, D, h->conf2_w, D, c.x, F32, D, N, D, D);
  g.bias = h->conf2_b;
  g.residual = c.x; g.ldr = D;
  // the RMSNorms fold into the products around them when every one of those runs on the
  // persistent tensor-core kernel; otherwise each is a kernel of its own
  const bool fold = fold_norms(c);
  if (fold) c.norm_out(g, h->layer[0].an);
  LL_TRY(run_gemm(g, st));
  // Transformer layers
  for (int i = 0; i < d.n_layers; ++i) {
    const HeadW& l = h->layer[i];
    if (!fold) LL_TRY(launch_rmsnorm(c.x, N, D, l.an, c.xn, adt, st));
    g = c.G(c.xn, adt, D, l.wqkv, D, c.qkv, c.qkv_dt, 3 * D, N, 3 * D, D);
    g.bias = l.bqkv;
    if (fold) c.norm_in(g);
    LL_TRY(run_gemm(g, st));
    if (c.tc_attn && attention_umma_supported(d.L, d.K, D, d.n_heads) &&
        (g_attn_umma == 1 || (g_attn_umma == 2 && d.L * d.K == 256 && d.K % 8 == 0)))
      LL_TRY(launch_attention_umma(c.qkv, c.B, d.L, d.K, D, d.n_heads, l.dist, l.same, c.att,
                                   c.status, st));
    else if (c.tc_attn)
      LL_TRY(launch_attention_tc(c.qkv, c.B, d.L, d.K, D, d.n_heads, l.dist, l.same, c.att, st));
    else
      LL_TRY(launch_attention(static_cast<const float*>(c.qkv), c.B, d.L, d.K, D, d.n_heads,
                              l.dist, l.same, c.att, adt, st));
    g = c.G(c.att, adt, D, l.wo, D, c.x, F32, D, N, D, D);
    g.bias = l.bo;
    g.residual = c.x; g.ldr = D;
    if (fold) c.norm_out(g, l.fn);
    LL_TRY(run_gemm(g, st));
    if (!fold) LL_TRY(launch_rmsnorm(c.x, N, D, l.fn, c.xn, adt, st));
    g = c.G(c.xn, adt, D, l.w1, D, c.hf, adt, F, N, F, D);
    g.bias = l.b1;
    g.act = ACT_SILU;
    if (fold) c.norm_in(g);
    LL_TRY(run_gemm(g, st));
    g = c.G(c.hf, adt, F, l.w2, F, c.x, F32, D, N, D, F);
    g.bias = l.b2;
    g.residual = c.x; g.ldr = D;
    // the last layer's output feeds the final norm: both blocks of the fusion input
    if (fold) {
      if (i + 1 < d.n_layers) c.norm_out(g, h->layer[i + 1].an);
      else c.final_norm_out(g, h->final_norm);
    }
    LL_TRY(run_gemm(g, st));
  }
  // fusion u = SiLU(W_f [x; t; x*t] + b_f) with x the final-normed state (the t block is
  // the per-sequence bias cb)
  if (!fold) LL_TRY(launch_fusion_input(c.x, c.B, c.LK, D, h->final_norm, c.t, c.xn, adt, st));
  g = c.G(c.xn, adt, 2 * D, h->fuse_x, 2 * D, c.u, adt, D, N, D, 2 * D);
  g.bias_rows = c.cb;
  g.rows_per_bias = c.LK;
  g.act = ACT_SILU;
  if (fold) c.norm_in(g);
  LL_TRY(run_gemm(g, st));
  // out and in heads in one product: oi = [W_o u + b_o | W_i u + b_i]
  g = c.G(c.u, adt, D, h->woi, D, c.oi, F32, 2 * d.d, N, 2 * d.d, D);
  g.bias = h->boi;
  return run_gemm(g, st);
}

// The whole scoring network on one stream.
lilicorr_status_t run_head(const lilicorr_head* h, int B, const int32_t* ids, const float* logp,
                           const void* hidden, const void* target, void* ws, const WsLayout& w,
                           cudaStream_t st) {
  const HeadCall c(h, B, ws, w);
  const lilicorr_status_t sp = fork_prologue(c, hidden, target, st);
  LL_TRY(join_prologue(h, st));
  LL_TRY(sp);
  return run_body(c, ids, logp, st);
}

}  // namespace

extern "C" {

const char* lilicorr_status_str(lilicorr_status_t s) {
  switch (s) {
    case LILICORR_OK: return "ok";
    case LILICORR_ERR_ARG: return "invalid argument";
    case LILICORR_ERR_SHAPE: return "unsupported or inconsistent shape";
    case LILICORR_ERR_DTYPE: return "unsupported dtype";
    case LILICORR_ERR_CUDA: return "CUDA error";
    case LILICORR_ERR_NONFINITE: return "non-finite logit row";
    case LILICORR_ERR_TIMEOUT: return "device wait timed out";
    case LILICORR_ERR_WORKSPACE: return "workspace too small";
  }
  return "unknown status";
}

int lilicorr_version(void) { return LILICORR_VERSION; }

size_t lilicorr_head_param_count(const lilicorr_head_desc* desc) {
  if (!desc_ok(desc)) return 0;
  return blob_index(*desc).total;
}

lilicorr_status_t lilicorr_head_create(const lilicorr_head_desc* desc, const void* host_weight_blob,
                                       const void* host_embed_table, lilicorr_head** out) {
  if (!out || !host_weight_blob || !host_embed_table) return LILICORR_ERR_ARG;
  *out = nullptr;
  if (!desc) return LILICORR_ERR_ARG;
  if (desc->dtype != LILICORR_F32 && desc->dtype != LILICORR_BF16) return LILICORR_ERR_DTYPE;
  if (!desc_ok(desc)) return LILICORR_ERR_SHAPE;
  const lilicorr_head_desc d = *desc;
  const BlobIndex bi = blob_index(d);
  const size_t D = d.D, H = d.H, F = d.ffn, dd = d.d, es = esize(d.dtype);

  Stager sg;
  sg.dt = d.dtype;
  sg.blob = static_cast<const unsigned char*>(host_weight_blob);
  struct Offs {
    size_t fold, emb_w, emb_b, hid_w, hid_b, conf1_w, conf1_b, conf2_w, conf2_b, slot, rank;
    size_t tgt_norm, tgt_w, tgt_b, final_norm, fuse_x, fuse_t, fuse_b, woi, boi, anc_w, anc_b;
    size_t wqkv[8], bqkv[8], wo[8], bo[8], w1[8], b1[8], w2[8], b2[8], an[8], fn[8], dist[8], same[8];
  } o;
  o.fold = sg.alloc((size_t)d.V * D * 4);
  o.emb_w = sg.mat(bi.emb_w, D, H);
  o.emb_b = sg.vec(bi.emb_b, D);
  o.hid_w = sg.mat(bi.hid_w, D, H);
  o.hid_b = sg.vec(bi.hid_b, D);
  o.conf1_w = sg.vec(bi.conf1_w, D * LILICORR_N_CONF);
  o.conf1_b = sg.vec(bi.conf1_b, D);
  o.conf2_w = sg.mat(bi.conf2_w, D, D);
  o.conf2_b = sg.vec(bi.conf2_b, D);
  o.slot = sg.vec(bi.slot, (size_t)d.L * D);
  o.rank = sg.vec(bi.rank, (size_t)d.K * D);
  o.tgt_norm = sg.vec(bi.tgt_norm, H);
  o.tgt_w = sg.mat(bi.tgt_w, D, H);
  o.tgt_b = sg.vec(bi.tgt_b, D);
  for (int i = 0; i < d.n_layers; ++i) {
    const BlobIndex::Layer& l = bi.layer[i];
    o.wqkv[i] = sg.alloc(3 * D * D * es);
    sg.put_mat(o.wqkv[i], l.wq, D, 0, D, 0, D, D, 0);
    sg.put_mat(o.wqkv[i] + D * D * es, l.wk, D, 0, D, 0, D, D, 0);
    sg.put_mat(o.wqkv[i] + 2 * D * D * es, l.wv, D, 0, D, 0, D, D, 0);
    o.bqkv[i] = sg.vec_cat({{l.bq, D}, {l.bk, D}, {l.bv, D}});
    o.wo[i] = sg.mat(l.wo, D, D);
    o.bo[i] = sg.vec(l.bo, D);
    o.w1[i] = sg.mat(l.w1, F, D);
    o.b1[i] = sg.vec(l.b1, F);
    o.w2[i] = sg.mat(l.w2, D, F);
    o.b2[i] = sg.vec(l.b2, D);
    o.an[i] = sg.vec(l.an, D);
    o.fn[i] = sg.vec(l.fn, D);
    o.dist[i] = sg.vec(l.dist, (size_t)d.n_heads * (2 * d.L - 1));
    o.same[i] = sg.vec(l.same, d.n_heads);
  }
  o.final_norm = sg.vec(bi.final_norm, D);
  // W_f [D, 3D] acts on [x; t; x*t]: keep the x and x*t column blocks together
  o.fuse_x = sg.alloc(D * 2 * D * es);
  sg.put_mat(o.fuse_x, bi.fuse_w, 3 * D, 0, D, 0, D, 2 * D, 0);
  sg.put_mat(o.fuse_x, bi.fuse_w, 3 * D, 0, D, 2 * D, D, 2 * D, D);
  o.fuse_t = sg.alloc(D * D * es);
  sg.put_mat(o.fuse_t, bi.fuse_w, 3 * D, 0, D, D, D, D, 0);
  o.fuse_b = sg.vec(bi.fuse_b, D);
  o.woi = sg.alloc(2 * dd * D * es);
  sg.put_mat(o.woi, bi.out_w, D, 0, dd, 0, D, D, 0);
  sg.put_mat(o.woi + dd * D * es, bi.in_w, D, 0, dd, 0, D, D, 0);
  o.boi = sg.vec_cat({{bi.out_b, dd}, {bi.in_b, dd}});
  o.anc_w = sg.mat(bi.anc_w, dd, D);
  o.anc_b = sg.vec(bi.anc_b, dd);
  const size_t pool_bytes = align_up(sg.off, 256);

  lilicorr_head* h = static_cast<lilicorr_head*>(calloc(1, sizeof(lilicorr_head)));
  if (!h) return LILICORR_ERR_ARG;
  h->desc = d;
  cudaGetDevice(&h->device);
  void* embed_dev = nullptr;
  auto fail = [&](lilicorr_status_t s) {
    (void)cudaGetLastError();
    if (embed_dev) cudaFree(embed_dev);
    if (h->pool) cudaFree(h->pool);
    if (h->side) cudaStreamDestroy(h->side);
    if (h->side2) cudaStreamDestroy(h->side2);
    if (h->ev_fork) cudaEventDestroy(h->ev_fork);
    if (h->ev_join) cudaEventDestroy(h->ev_join);
    if (h->ev_join2) cudaEventDestroy(h->ev_join2);
    if (h->ev_t) cudaEventDestroy(h->ev_t);
    free(h);
    return s;
  };
  if (cudaStreamCreateWithFlags(&h->side, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&h->side2, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_join2, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_t, cudaEventDisableTiming) != cudaSuccess)
    return fail(LILICORR_ERR_CUDA);
  if (cudaMalloc(&h->pool, pool_bytes) != cudaSuccess) return fail(LILICORR_ERR_CUDA);
  h->pool_bytes = pool_bytes;
  // the fold region is written on the device; copy everything after it
  if (cudaMemcpy(static_cast<unsigned char*>(h->pool) + o.emb_w, sg.host.data() + o.emb_w,
                 sg.off - o.emb_w, cudaMemcpyHostToDevice) != cudaSuccess)
    return fail(LILICORR_ERR_CUDA);
  auto P = [&](size_t off) { return static_cast<const void*>(static_cast<unsigned char*>(h->pool) + off); };
  auto Pf = [&](size_t off) { return static_cast<const float*>(P(off)); };
  h->fold = P(o.fold);
  h->hid_w = P(o.hid_w); h->hid_b = Pf(o.hid_b);
  h->conf1_w = Pf(o.conf1_w); h->conf1_b = Pf(o.conf1_b);
  h->conf2_w = P(o.conf2_w); h->conf2_b = Pf(o.conf2_b);
  h->slot = Pf(o.slot); h->rank = Pf(o.rank);
  h->tgt_norm = Pf(o.tgt_norm); h->tgt_w = P(o.tgt_w); h->tgt_b = Pf(o.tgt_b);
  for (int i = 0; i < d.n_layers; ++i) {
    HeadW& l = h->layer[i];
    l.wqkv = P(o.wqkv[i]); l.bqkv = Pf(o.bqkv[i]);
    l.wo = P(o.wo[i]); l.bo = Pf(o.bo[i]);
    l.w1 = P(o.w1[i]); l.b1 = Pf(o.b1[i]);
    l.w2 = P(o.w2[i]); l.b2 = Pf(o.b2[i]);
    l.an = Pf(o.an[i]); l.fn = Pf(o.fn[i]);
    l.dist = Pf(o.dist[i]); l.same = Pf(o.same[i]);
  }
  h->final_norm = Pf(o.final_norm);
  h->fuse_x = P(o.fuse_x); h->fuse_t = P(o.fuse_t); h->fuse_b = Pf(o.fuse_b);
  h->woi = P(o.woi); h->boi = Pf(o.boi);
  h->anc_w = P(o.anc_w); h->anc_b = Pf(o.anc_b);

  // fold the frozen, linear embedding projection once: fold = E W_e^T + b_e  [V, D] fp32
  const size_t emb_bytes = (size_t)d.V * H * es;
  if (cudaMalloc(&embed_dev, emb_bytes) != cudaSuccess) return fail(LILICORR_ERR_CUDA);
  if (cudaMemcpy(embed_dev, host_embed_table, emb_bytes, cudaMemcpyHostToDevice) != cudaSuccess)
    return fail(LILICORR_ERR_CUDA);
  GemmArgs g = gemm(embed_dev, d.dtype, (int)H, P(o.emb_w), d.dtype, (int)H,
                    const_cast<void*>(h->fold), LILICORR_F32, (int)D, d.V, (int)D, (int)H);
  g.bias = Pf(o.emb_b);
  lilicorr_status_t s = launch_gemm_simt(g, 0);
  if (s != LILICORR_OK) return fail(s);
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(LILICORR_ERR_CUDA);
  cudaFree(embed_dev);
  embed_dev = nullptr;
  h->net_maps = net_fused_maps_create(h);
  h->cluster_maps = net_cluster_maps_create(h);
  h->pair_maps = net_pair_maps_create(h);
  *out = h;
  return LILICORR_OK;
}

lilicorr_status_t lilicorr_head_destroy(lilicorr_head* h) {
  if (!h) return LILICORR_ERR_ARG;
  int cur = 0;
  cudaGetDevice(&cur);
  if (cur != h->device) cudaSetDevice(h->device);
  cudaError_t e = cudaFree(h->pool);
  net_fused_maps_free(h->net_maps);
  net_cluster_maps_free(h->cluster_maps);
  net_pair_maps_free(h->pair_maps);
  if (h->side) cudaStreamDestroy(h->side);
  if (h->side2) cudaStreamDestroy(h->side2);
  if (h->ev_fork) cudaEventDestroy(h->ev_fork);
  if (h->ev_join) cudaEventDestroy(h->ev_join);
  if (h->ev_join2) cudaEventDestroy(h->ev_join2);
  if (h->ev_t) cudaEventDestroy(h->ev_t);
  if (cur != h->device) cudaSetDevice(cur);
  free(h);
  return e == cudaSuccess ? LILICORR_OK : LILICORR_ERR_CUDA;
}

lilicorr_status_t lilicorr_workspace_init(void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (!ws && ws_bytes) return LILICORR_ERR_ARG;
  if (!ws_bytes) return LILICORR_OK;
  LL_CUDA_TRY(cudaMemsetAsync(ws, 0, ws_bytes, stream));
  return LILICORR_OK;
}

size_t lilicorr_topk_lse_workspace_bytes(int rows, int V, int K) {
  if (rows < 0 || V <= 0 || K <= 0 || K > LILICORR_MAX_K || K > V) return 0;
  // sized for the larger (fp32) plan so the same workspace serves both dtypes
  size_t a = topk_ws_bytes(rows, V, K, LILICORR_F32), b = topk_ws_bytes(rows, V, K, LILICORR_BF16);
  return a > b ? a : b;
}

lilicorr_status_t lilicorr_topk_lse(const void* logits, lilicorr_dtype_t dtype, int rows, int V,
                                    int K, int32_t* ids, float* logp, float* lse, void* ws,
                                    size_t ws_bytes, cudaStream_t stream) {
  if (dtype != LILICORR_F32 && dtype != LILICORR_BF16) return LILICORR_ERR_DTYPE;
  if (rows < 0 || V <= 0 || K <= 0 || K > LILICORR_MAX_K || K > V) return LILICORR_ERR_SHAPE;
  if (rows == 0) return LILICORR_OK;
  if (!logits || !ids || !logp || !lse || !ws) return LILICORR_ERR_ARG;
  if (!aligned16(logits) || !aligned16(ws)) return LILICORR_ERR_ARG;
  if (ws_bytes < lilicorr_topk_lse_workspace_bytes(rows, V, K)) return LILICORR_ERR_WORKSPACE;
  unsigned char* w = static_cast<unsigned char*>(ws);
  uint32_t* status = reinterpret_cast<uint32_t*>(w);
  uint32_t* counters = reinterpret_cast<uint32_t*>(w + 256);
  void* partials = w + 256 + align_up((size_t)rows * 4, 256);
  return launch_topk_lse(logits, dtype, rows, V, K, ids, logp, lse, status, counters, partials,
                         stream);
}

size_t lilicorr_topk_partial_bytes(int K) {
  return K > 0 && K <= LILICORR_MAX_K ? topk_partial_bytes(K) : 0;
}

size_t lilicorr_topk_lse_partial_workspace_bytes(int rows, int V, int K) {
  if (rows < 0 || V <= 0 || K <= 0 || K > LILICORR_MAX_K) return 0;
  size_t a = topk_ws_bytes(rows, V, K, LILICORR_F32), b = topk_ws_bytes(rows, V, K, LILICORR_BF16);
  return a > b ? a : b;
}

lilicorr_status_t lilicorr_topk_lse_partial(const void* logits, lilicorr_dtype_t dtype, int rows,
                                            int V, int K, int32_t id_offset, void* partial,
                                            void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (dtype != LILICORR_F32 && dtype != LILICORR_BF16) return LILICORR_ERR_DTYPE;
  if (rows < 0 || V <= 0 || K <= 0 || K > LILICORR_MAX_K) return LILICORR_ERR_SHAPE;
  if (id_offset < 0 || (int64_t)id_offset + V > INT32_MAX) return LILICORR_ERR_ARG;
  if (rows == 0) return LILICORR_OK;
  if (!logits || !partial || !ws) return LILICORR_ERR_ARG;
  if (!aligned16(logits) || !aligned16(ws) || (reinterpret_cast<uintptr_t>(partial) & 7))
    return LILICORR_ERR_ARG;
  if (ws_bytes < lilicorr_topk_lse_partial_workspace_bytes(rows, V, K)) return LILICORR_ERR_WORKSPACE;
  unsigned char* w = static_cast<unsigned char*>(ws);
  return launch_topk_lse(logits, dtype, rows, V, K, nullptr, nullptr, nullptr,
                         reinterpret_cast<uint32_t*>(w), reinterpret_cast<uint32_t*>(w + 256),
                         w + 256 + align_up((size_t)rows * 4, 256), stream, partial, id_offset);
}

lilicorr_status_t lilicorr_topk_lse_merge(const void* partials, int P, int rows, int K,
                                          int32_t* ids, float* logp, float* lse, uint32_t* status,
                                          cudaStream_t stream) {
  if (rows < 0 || P < 1 || K <= 0 || K > LILICORR_MAX_K || P * K > TOPK_MERGE_KEYS_MAX)
    return LILICORR_ERR_SHAPE;
  if (rows == 0) return LILICORR_OK;
  if (!partials || !ids || !logp || !lse) return LILICORR_ERR_ARG;
  if (reinterpret_cast<uintptr_t>(partials) & 7) return LILICORR_ERR_ARG;
  return launch_topk_merge(partials, P, rows, K, ids, logp, lse, status, stream);
}

size_t lilicorr_lm_head_topk_workspace_bytes(int rows, int H, int V, int K) {
  if (!lm_head_supported(rows, H, V, K)) return 0;
  return 256 + align_up(lm_head_records_bytes(rows, V, K), 256);
}

lilicorr_status_t lilicorr_lm_head_topk(const void* hidden, const void* w_vocab, int rows, int H,
                                        int V, int K, int32_t* ids, float* logp, float* lse,
                                        void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (rows < 0 || H <= 0 || V <= 0 || K <= 0 || K > LILICORR_MAX_K || K > V)
    return LILICORR_ERR_SHAPE;
  if (rows == 0) return LILICORR_OK;
  if (!lm_head_supported(rows, H, V, K)) return LILICORR_ERR_SHAPE;
  if (!hidden || !w_vocab || !ids || !logp || !lse || !ws) return LILICORR_ERR_ARG;
  if (!aligned16(hidden) || !aligned16(w_vocab) || !aligned16(ws)) return LILICORR_ERR_ARG;
  if (ws_bytes < lilicorr_lm_head_topk_workspace_bytes(rows, H, V, K)) return LILICORR_ERR_WORKSPACE;
  unsigned char* w = static_cast<unsigned char*>(ws);
  return launch_lm_head_topk(hidden, w_vocab, rows, H, V, K, w + 256, ids, logp, lse,
                             reinterpret_cast<uint32_t*>(w), stream);
}

size_t lilicorr_workspace_bytes(const lilicorr_head* head, int B) {
  if (!head || B < 0) return 0;
  return ws_layout(head->desc, B).total;
}

lilicorr_status_t lilicorr_embed_in_out(const lilicorr_head* head, int B, const int32_t* ids,
                                        const float* logp, const void* drafter_hidden,
                                        const void* target_hidden, float* out_vec, float* in_vec,
                                        float* anchor_out, void* ws, size_t ws_bytes,
                                        cudaStream_t stream) {
  if (!head || B < 0) return LILICORR_ERR_ARG;
  if (B == 0) return LILICORR_OK;
  if (!ids || !logp || !drafter_hidden || !target_hidden || !out_vec || !in_vec || !anchor_out || !ws)
    return LILICORR_ERR_ARG;
  if (!aligned16(drafter_hidden) || !aligned16(target_hidden) || !aligned16(ws))
    return LILICORR_ERR_ARG;
  const WsLayout w = ws_layout(head->desc, B);
  if (ws_bytes < w.total) return LILICORR_ERR_WORKSPACE;
  const lilicorr_head_desc& d = head->desc;
  LL_TRY(run_head(head, B, ids, logp, drafter_hidden, target_hidden, ws, w, stream));
  const int N = B * d.L * d.K;
  const float* oi = at<float>(ws, w.oi);
  LL_TRY(launch_unit_rows(oi, N, d.d, 2 * d.d, out_vec, d.d, stream));
  LL_TRY(launch_unit_rows(oi + d.d, N, d.d, 2 * d.d, in_vec, d.d, stream));
  LL_TRY(launch_unit_rows(at<float>(ws, w.anc), B, d.d, d.d, anchor_out, d.d, stream));
  return LILICORR_OK;
}

lilicorr_status_t lilicorr_pair_scores(int B, int L, int K, int d, const float* out_vec,
                                       const float* in_vec, const float* anchor_out,
                                       float* anchor_scores, float* pair_scores,
                                       cudaStream_t stream) {
  if (B < 0 || L <= 0 || L > LILICORR_MAX_L || K <= 0 || K > LILICORR_MAX_K || d <= 0)
    return LILICORR_ERR_SHAPE;
  if (B == 0) return LILICORR_OK;
  if (!out_vec || !in_vec || !anchor_out || !anchor_scores || (L > 1 && !pair_scores))
    return LILICORR_ERR_ARG;
  if (pair_walk_smem_bytes(L, K, d) > 200 * 1024) return LILICORR_ERR_SHAPE;
  PairWalkArgs a;
  memset(&a, 0, sizeof(a));
  a.B = B; a.L = L; a.K = K; a.d = d;
  a.out = out_vec; a.in = in_vec; a.ld_vec = d; a.anchor = anchor_out;
  a.A = anchor_scores; a.P = pair_scores;
  a.do_pairs = true; a.do_walk = false;
  return launch_pair_walk(a, stream);
}

lilicorr_status_t lilicorr_greedy_walk(int B, int L, int K, const float* anchor_scores,
                                       const float* pair_scores, const int32_t* ids,
                                       int32_t* choice, int32_t* tokens, float* margin,
                                       cudaStream_t stream) {
  if (B < 0 || L <= 0 || L > LILICORR_MAX_L || K <= 0 || K > LILICORR_MAX_K)
    return LILICORR_ERR_SHAPE;
  if (B == 0) return LILICORR_OK;
  if (!anchor_scores || (L > 1 && !pair_scores) || !ids || !choice || !tokens)
    return LILICORR_ERR_ARG;
  if (pair_walk_smem_bytes(L, K, 0) > 200 * 1024) return LILICORR_ERR_SHAPE;
  PairWalkArgs a;
  memset(&a, 0, sizeof(a));
  a.B = B; a.L = L; a.K = K; a.d = 0;
  a.A = const_cast<float*>(anchor_scores); a.P = const_cast<float*>(pair_scores);
  a.ids = ids; a.choice = choice; a.tokens = tokens; a.margin = margin;
  a.do_pairs = false; a.do_walk = true;
  return launch_pair_walk(a, stream);
}

lilicorr_status_t lilicorr_best_path(int B, int L, int K, const float* anchor_scores,
                                     const float* pair_scores, const int32_t* ids, float sigma,
                                     int32_t* choice, int32_t* tokens, float* path_score,
                                     cudaStream_t stream) {
  if (B < 0 || L <= 0 || L > LILICORR_MAX_L || K <= 0 || K > LILICORR_MAX_K)
    return LILICORR_ERR_SHAPE;
  if (!(sigma > 0.f) || !isfinite(sigma)) return LILICORR_ERR_ARG;
  if (B == 0) return LILICORR_OK;
  if (!anchor_scores || (L > 1 && !pair_scores) || !ids || !choice || !tokens)
    return LILICORR_ERR_ARG;
  if (pair_walk_smem_bytes(L, K, 0) > 200 * 1024) return LILICORR_ERR_SHAPE;
  PairWalkArgs a;
  memset(&a, 0, sizeof(a));
  a.B = B; a.L = L; a.K = K; a.d = 0;
  a.A = const_cast<float*>(anchor_scores); a.P = const_cast<float*>(pair_scores);
  a.ids = ids; a.choice = choice; a.tokens = tokens;
  a.walk_mode = LILICORR_WALK_VITERBI; a.sigma = sigma; a.path_score = path_score;
  a.do_pairs = false; a.do_walk = true;
  return launch_pair_walk(a, stream);
}

lilicorr_status_t lilicorr_select_block(const lilicorr_head* head, int B, const void* logits,
                                        const void* drafter_hidden, const void* target_hidden,
                                        int32_t* tokens, void* ws, size_t ws_bytes,
                                        cudaStream_t stream) {
  return lilicorr_select_block_walk(head, B, logits, drafter_hidden, target_hidden,
                                    LILICORR_WALK_GREEDY, tokens, ws, ws_bytes, stream);
}

lilicorr_status_t lilicorr_select_block_walk(const lilicorr_head* head, int B, const void* logits,
                                             const void* drafter_hidden,
                                             const void* target_hidden, lilicorr_walk_t walk,
                                             int32_t* tokens, void* ws, size_t ws_bytes,
                                             cudaStream_t stream) {
  if (walk != LILICORR_WALK_GREEDY && walk != LILICORR_WALK_VITERBI) return LILICORR_ERR_ARG;
  if (!head || B < 0) return LILICORR_ERR_ARG;
  if (B == 0) return LILICORR_OK;
  if (!logits || !drafter_hidden || !target_hidden || !tokens || !ws) return LILICORR_ERR_ARG;
  if (!aligned16(logits) || !aligned16(drafter_hidden) || !aligned16(target_hidden) ||
      !aligned16(ws))
    return LILICORR_ERR_ARG;
  const WsLayout w = ws_layout(head->desc, B);
  if (ws_bytes < w.total) return LILICORR_ERR_WORKSPACE;
  const lilicorr_head_desc& d = head->desc;
  const int R = B * d.L;
  int32_t* ids = at<int32_t>(ws, w.ids);
  float* logp = at<float>(ws, w.logp);
  // the candidate-independent projections run beside the top-K pass
  const HeadCall call(head, B, ws, w);
  const lilicorr_status_t sp = fork_prologue(call, drafter_hidden, target_hidden, stream);
  const lilicorr_status_t st = sp != LILICORR_OK ? sp
      : launch_topk_lse(logits, d.dtype, R, d.V, d.K, ids, logp, at<float>(ws, w.lse),
                        at<uint32_t>(ws, w.status), at<uint32_t>(ws, w.counters),
                        at<void>(ws, w.partials), stream);
  LL_TRY(join_prologue(head, stream));                      // always rejoin, even on error
  LL_TRY(st);
  ClusterTail tail;
  tail.anchor = at<float>(ws, w.anc);
  tail.A = at<float>(ws, w.A);
  tail.P = at<float>(ws, w.P);
  tail.choice = at<int32_t>(ws, w.choice);
  tail.tokens = tokens;
  bool tail_done = false;
  LL_TRY(run_body(call, ids, logp, stream, walk == LILICORR_WALK_GREEDY ? &tail : nullptr,
                  &tail_done));
  if (tail_done) return LILICORR_OK;
  PairWalkArgs a;
  memset(&a, 0, sizeof(a));
  a.B = B; a.L = d.L; a.K = d.K; a.d = d.d;
  const float* oi = at<float>(ws, w.oi);
  a.out = oi; a.in = oi + d.d; a.ld_vec = 2 * d.d;
  a.anchor = at<float>(ws, w.anc);
  a.A = at<float>(ws, w.A); a.P = at<float>(ws, w.P);
  a.ids = ids; a.choice = at<int32_t>(ws, w.choice); a.tokens = tokens; a.margin = nullptr;
  a.do_pairs = true; a.do_walk = true;
  a.walk_mode = walk; a.sigma = LILICORR_SIGMA;
  a.counters = at<uint32_t>(ws, w.pw_counters);
  return launch_pair_walk(a, stream);
}

lilicorr_status_t lilicorr_select_block_intermediates(const lilicorr_head* head, int B, void* ws,
                                                      size_t ws_bytes, int32_t** ids, float** logp,
                                                      float** lse, float** anchor_scores,
                                                      float** pair_scores, int32_t** choice) {
  if (!head || B < 0 || !ws) return LILICORR_ERR_ARG;
  const WsLayout w = ws_layout(head->desc, B);
  if (ws_bytes < w.total) return LILICORR_ERR_WORKSPACE;
  if (ids) *ids = at<int32_t>(ws, w.ids);
  if (logp) *logp = at<float>(ws, w.logp);
  if (lse) *lse = at<float>(ws, w.lse);
  if (anchor_scores) *anchor_scores = at<float>(ws, w.A);
  if (pair_scores) *pair_scores = at<float>(ws, w.P);
  if (choice) *choice = at<int32_t>(ws, w.choice);
  return LILICORR_OK;
}

lilicorr_status_t lilicorr_test_linear(const void* A, lilicorr_dtype_t a_dt, int lda, const void* W,
                                       lilicorr_dtype_t w_dt, int ldw, void* C,
                                       lilicorr_dtype_t c_dt, int ldc, int M, int N, int Kd,
                                       const float* bias, const float* residual, int act, int path,
                                       uint32_t* status, cudaStream_t stream) {
  if (!A || !W || !C || M < 0 || N < 0 || Kd <= 0) return LILICORR_ERR_ARG;
  GemmArgs g = gemm(A, a_dt, lda, W, w_dt, ldw, C, c_dt, ldc, M, N, Kd);
  g.bias = bias;
  g.residual = residual;
  g.ldr = ldc;
  g.act = act;
  g.status = status;
  switch (path) {
    case 0: return run_gemm(g, stream);
    case 1: return launch_gemm_simt(g, stream);
    case 2: return launch_gemm_skinny(g, stream);
    case 3: return gemm_tc_supported(g) ? launch_gemm_tc(g, stream) : LILICORR_ERR_DTYPE;
    case 4: return gemm_small_supported(g) ? launch_gemm_small(g, stream) : LILICORR_ERR_SHAPE;
    case 5: return launch_gemm_rows(g, stream);
  }
  return LILICORR_ERR_ARG;
}

lilicorr_status_t lilicorr_test_linear_timeout(const void* A, const void* W, float* C, int M, int N,
                                               int Kd, long long wait_cycles, uint32_t* status,
                                               cudaStream_t stream) {
  if (!A || !W || !C || !status || M <= 0 || N <= 0 || Kd <= 0) return LILICORR_ERR_ARG;
  if (wait_cycles < 100000 || wait_cycles > 4000000000ll) return LILICORR_ERR_ARG;
  GemmArgs g = gemm(A, LILICORR_BF16, Kd, W, LILICORR_BF16, Kd, C, LILICORR_F32, N, M, N, Kd);
  g.status = status;
  g.wait_limit = wait_cycles;
  g.test_starve = 1;
  return gemm_tc_supported(g) ? launch_gemm_tc(g, stream) : LILICORR_ERR_SHAPE;
}

int lilicorr_test_attention_path(int mode) {
  const int prev = g_attn_umma;
  g_attn_umma = mode < 0 ? 0 : mode > 2 ? 2 : mode;
  return prev;
}

int lilicorr_test_fused_path(const lilicorr_head* head, int mode) {
  g_fused_enabled = mode < 0 ? 0 : mode > 3 ? 3 : mode;
  if (!head) return 0;
  if (mode == 3) return head->cluster_maps ? 1 : 0;
  return (head->net_maps || head->pair_maps) ? 1 : 0;
}

uint64_t lilicorr_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

lilicorr_status_t lilicorr_get_device_status(void* ws, cudaStream_t stream) {
  if (!ws) return LILICORR_ERR_ARG;
  uint32_t v = 0;
  LL_CUDA_TRY(cudaMemcpyAsync(&v, ws, 4, cudaMemcpyDeviceToHost, stream));
  LL_CUDA_TRY(cudaStreamSynchronize(stream));
  if (v != 0) LL_CUDA_TRY(cudaMemsetAsync(ws, 0, 4, stream));
  LL_CUDA_TRY(cudaStreamSynchronize(stream));
  return static_cast<lilicorr_status_t>(v);
}

}  // extern "C"
