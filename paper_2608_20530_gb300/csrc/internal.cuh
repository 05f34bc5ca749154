// Internal declarations of the LiLiCorr selection library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <string.h>
#include <utility>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stddef.h>

#include "lilicorr.h"

namespace lilicorr {

// ----------------------------------------------------------------------------- host helpers
#define LL_CUDA_TRY(expr)                                   \
  do {                                                      \
    cudaError_t _e = (expr);                                \
    if (_e != cudaSuccess) {                                \
      (void)cudaGetLastError(); /* do not leak into later calls */ \
      return LILICORR_ERR_CUDA;                             \
    }                                                       \
  } while (0)

#define LL_TRY(expr)                                        \
  do {                                                      \
    lilicorr_status_t _s = (expr);                          \
    if (_s != LILICORR_OK) return _s;                       \
  } while (0)

void count_launch();   // host-side launch counter (lilicorr_launch_count)

// Call right after each kernel launch: counts it and reports a launch error.
inline lilicorr_status_t last_launch() {
  count_launch();
  return cudaGetLastError() == cudaSuccess ? LILICORR_OK : LILICORR_ERR_CUDA;
}

// Launch with programmatic dependent launch allowed: the kernel may start while its
// predecessor on the stream finishes. Every kernel of this library begins with
// pdl_wait() before it reads or writes memory that an earlier launch touches, so the
// stream order of results is unchanged; what overlaps is the launch itself and the
// setup that needs no inputs.
template <typename... KArgs, typename... Args>
lilicorr_status_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                           cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
  count_launch();
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    return LILICORR_ERR_CUDA;
  }
  return LILICORR_OK;
}

// Wait for the preceding launch on the stream to complete and its writes to be visible
// (a no-op when the kernel was not launched as a dependent), then let the next launch
// on the stream start its own setup.
__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

constexpr int SMEM_PER_BLOCK_MAX = 227 * 1024;   // opt-in shared memory per block (sm_103a)

// Raise a kernel's dynamic shared-memory cap to what is left beside its static shared
// memory, once per device.
template <typename F>
lilicorr_status_t allow_max_dynamic_smem(F* func, bool (&done)[64]) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) { (void)cudaGetLastError(); return LILICORR_ERR_CUDA; }
  if (dev < 0 || dev >= 64 || done[dev]) return LILICORR_OK;
  cudaFuncAttributes attr;
  if (cudaFuncGetAttributes(&attr, func) != cudaSuccess) {
    (void)cudaGetLastError();
    return LILICORR_ERR_CUDA;
  }
  const int dyn = SMEM_PER_BLOCK_MAX - (int)attr.sharedSizeBytes;
  if (cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn) != cudaSuccess) {
    (void)cudaGetLastError();
    return LILICORR_ERR_CUDA;
  }
  done[dev] = true;
  return LILICORR_OK;
}
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline int ceil_div(long long a, long long b) { return (int)((a + b - 1) / b); }

int num_sms();   // of the current device, cached per device

// ----------------------------------------------------------------------------- device helpers
__device__ __forceinline__ float bf16_to_f32(uint16_t b) {
  return __uint_as_float(((uint32_t)b) << 16);
}
__device__ __forceinline__ float ld_elem(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ld_elem(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void st_elem(float* p, size_t i, float v) { p[i] = v; }
__device__ __forceinline__ void st_elem(__nv_bfloat16* p, size_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float silu_f(float z) { return z / (1.0f + __expf(-z)); }
// two floats as a bf16 pair (round to nearest even), lo in the low half
__device__ __forceinline__ uint32_t bf16_pack2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}
// SiLU(z) = z (1 + tanh(z / 2)) / 2 with one MUFU operation, for outputs rounded to bf16
// (tanh.approx's error is below the bf16 rounding that follows)
__device__ __forceinline__ float silu_tanh(float z) {
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(0.5f * z));
  return 0.5f * z * (1.0f + t);
}

// Record the first device-detected error in the workspace status word.
__device__ __forceinline__ void set_status(uint32_t* status, uint32_t code) {
  if (status) atomicCAS(status, 0u, code);
}

// ----------------------------------------------------------------------------- head
struct HeadW {          // device pointers of one Transformer layer
  const void* wqkv;     // [3D, D] (q rows, then k, then v)
  const float* bqkv;    // [3D]
  const void* wo;       // [D, D]
  const float* bo;
  const void* w1;       // [F, D]
  const float* b1;
  const void* w2;       // [D, F]
  const float* b2;
  const float* an;      // [D] attention RMSNorm gain
  const float* fn;      // [D] FFN RMSNorm gain
  const float* dist;    // [n_heads, 2L-1]
  const float* same;    // [n_heads]
};

}  // namespace lilicorr

struct lilicorr_head {
  lilicorr_head_desc desc;
  int device;
  // the projections that do not depend on the top-K pass run on two side streams that
  // fork from and join the caller's stream (fork/join nodes under graph capture)
  cudaStream_t side, side2;
  cudaEvent_t ev_fork, ev_join, ev_join2, ev_t;   // ev_t: the target state t is ready
  void* pool;                 // one device allocation holding everything below
  size_t pool_bytes;
  // matrices in head dtype; vectors and tables in fp32
  const void* fold;           // [V, D] folded embedding table E W_e^T + b_e (head dtype)
  const void* hid_w;  const float* hid_b;
  const float* conf1_w; const float* conf1_b;     // [D, 5], [D] (fp32)
  const void* conf2_w; const float* conf2_b;
  const float* slot; const float* rank;           // [L, D], [K, D]
  const float* tgt_norm;                          // [H]
  const void* tgt_w; const float* tgt_b;
  lilicorr::HeadW layer[8];
  const float* final_norm;
  const void* fuse_x;         // [D, 2D]: columns of W_f acting on x and on x*t
  const void* fuse_t;         // [D, D]:  columns of W_f acting on t
  const float* fuse_b;
  const void* woi;            // [2d, D]: out_w rows then in_w rows
  const float* boi;           // [2d]
  const void* anc_w; const float* anc_b;
  void* net_maps;             // tensor maps of the fused scoring network, or null
  void* cluster_maps;         // tensor maps of the cluster scoring network, or null
  void* pair_maps;            // tensor maps of the two-CTA network (129-256 nodes), or null
};

namespace lilicorr {

// ----------------------------------------------------------------------------- workspace
struct TopkPlan {
  int splits;          // CTAs per row
  int threads;         // threads per CTA
  int unroll;          // 16-byte vectors per thread per batch
  int chunk_vecs;      // 16-byte vectors per split
  int pieces;          // partial records per row in the workspace
  size_t rec_bytes;    // bytes of one partial record
};
TopkPlan topk_plan(int rows, int V, int K, lilicorr_dtype_t dt);

struct WsLayout {
  size_t status, counters, partials;
  size_t ids, logp, lse;
  size_t hproj, tn, t, anc, cb;
  size_t x, c1, xn, qkv, att, hf, u, oi;
  size_t A, P, choice, pw_counters;
  size_t ss;           // folded RMSNorm: row sums of squares [N, SS_LD]
  size_t total;
};
WsLayout ws_layout(const lilicorr_head_desc& d, int B);
size_t topk_ws_bytes(int rows, int V, int K, lilicorr_dtype_t dt);

// ----------------------------------------------------------------------------- launchers
// (1) top-K + log-normaliser. ws: status word at offset 0, then counters, partials.
// partial_out non-null: write each row's public partial record (see
// lilicorr_topk_lse_partial) with id_offset added to its ids instead of ids/logp/lse
lilicorr_status_t launch_topk_lse(const void* logits, lilicorr_dtype_t dt, int rows, int V, int K,
                                  int32_t* ids, float* logp, float* lse, uint32_t* status,
                                  uint32_t* counters, void* partials, cudaStream_t st,
                                  void* partial_out = nullptr, int32_t id_offset = 0);
// bytes of one row's partial record: max, sum, K values, K ids
__host__ __device__ constexpr size_t topk_partial_bytes(int K) { return 8 + 8 * (size_t)K; }
// the merge holds P*K keys (and as many survivors) in shared memory
constexpr int TOPK_MERGE_KEYS_MAX = 8192;

// Order-preserving 64-bit candidate key: larger value first, equal values by lower id;
// -0.0 == +0.0. Key 0 never occurs for a real element and marks an empty slot.
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
// LM-head projection fused with step (1) (lm_head.cu): records [P][rows] in ws, then merged
bool lm_head_supported(int rows, int H, int V, int K);
size_t lm_head_records_bytes(int rows, int V, int K);
lilicorr_status_t launch_lm_head_topk(const void* hidden, const void* w_vocab, int rows, int H,
                                      int V, int K, void* recs, int32_t* ids, float* logp,
                                      float* lse, uint32_t* status, cudaStream_t st);
// merge P shards' records [P][rows][topk_partial_bytes(K)] into the final outputs
lilicorr_status_t launch_topk_merge(const void* partials, int P, int rows, int K, int32_t* ids,
                                    float* logp, float* lse, uint32_t* status, cudaStream_t st);

// Generic linear layer C = act(A W^T + bias [+ bias_rows[m / rows_per_bias]]) [+ residual].
enum { ACT_NONE = 0, ACT_SILU = 1 };
struct GemmArgs {
  const void* A; lilicorr_dtype_t a_dt; int lda;
  const void* W; lilicorr_dtype_t w_dt; int ldw;
  void* C; lilicorr_dtype_t c_dt; int ldc;
  const float* bias;
  const float* bias_rows; int rows_per_bias;
  const float* residual; int ldr;
  int act;
  int M, N, Kd;
  uint32_t* status;        // device status word (bounded-wait timeouts), may be null
  long long wait_limit;    // SM cycles per bounded wait of the tensor-core kernel; 0: ~2 s
  int test_starve;         // test hook only: the tensor-core kernel's producer issues no
                           // copies, so its consumers' waits run out (see the testing header)
  // RMSNorm folded into the products around it (tensor-core kernel only). Producer (fp32 C):
  // c2 [M, ldc2] (bf16) receives C times c2_gain per column, ss_out [M, SS_LD] partial sums of
  // squares of C's rows (gemm_tc_ss_slots(M, N) slots per row). Consumer: the product is
  // scaled per row by rsqrt(sum of ss_in's first ss_slots slots / Kd + eps) before the bias.
  void* c2; int ldc2; const float* c2_gain; float* ss_out;
  const float* ss_in; int ss_slots;
  int ss_dim;              // the norm's row length (0: Kd)
  // producer, also: c3 [M, ldc2] (bf16) receives C times c2_gain times c3_t's row
  // m / c3_rows_per (c3_t [*, N], fp32), e.g. the x*t block of the fusion input
  void* c3; const float* c3_t; int c3_rows_per;
};
constexpr int SS_LD = 16;  // floats per row of a folded-RMSNorm sums-of-squares buffer
int gemm_tc_ss_slots(int M, int N);
lilicorr_status_t launch_gemm_simt(const GemmArgs& g, cudaStream_t st);
lilicorr_status_t launch_gemm_skinny(const GemmArgs& g, cudaStream_t st);   // M <= 64
// fp32 activations, per-sequence row counts (16 x 32 output blocks, no K split)
bool gemm_rows_supported(const GemmArgs& g);
lilicorr_status_t launch_gemm_rows(const GemmArgs& g, cudaStream_t st);
bool gemm_tc_supported(const GemmArgs& g);
lilicorr_status_t launch_gemm_tc(const GemmArgs& g, cudaStream_t st);
// one tile of rows (M <= 128, Kd <= 512, a multiple of 64): whole-K TMA copies (gemm_small.cu)
bool gemm_small_supported(const GemmArgs& g);
lilicorr_status_t launch_gemm_small(const GemmArgs& g, cudaStream_t st);

// scoring-network helpers (head_kernels.cu)
// fused scoring network (net_fused.cu): one CTA per sequence, bf16 head with D = 256,
// 8 heads, FFN 2D, L*K <= 128. Writes oi like run_body's unfused chain.
bool net_fused_supported(const lilicorr_head_desc& d);
void* net_fused_maps_create(const lilicorr_head* h);
void net_fused_maps_free(void* maps);
lilicorr_status_t launch_net_fused(const lilicorr_head* h, int B, const int32_t* ids,
                                   const float* logp, const float* hproj, const float* t,
                                   const float* cb, float* oi, uint32_t* status, cudaStream_t st);
// the same network for 129-256 nodes per sequence on a cluster of two CTAs, one 128-node
// tile each (net_pair.cu)
bool net_pair_supported(const lilicorr_head_desc& d);
void* net_pair_maps_create(const lilicorr_head* h);
void net_pair_maps_free(void* p);
lilicorr_status_t launch_net_pair(const lilicorr_head* h, int B, const int32_t* ids,
                                  const float* logp, const float* hproj, const float* t,
                                  const float* cb, float* oi, uint32_t* status, cudaStream_t st);
// the same network on a cluster of four CTAs per sequence (net_cluster.cu)
bool net_cluster_supported(const lilicorr_head_desc& d);
void* net_cluster_maps_create(const lilicorr_head* h);
void net_cluster_maps_free(void* p);
int net_cluster_capacity();   // clusters that fit on the device at once
// Steps (3) and (4) fused into the cluster kernel's tail: the anchor and pair scores
// (written to A [B, K] and P [B, L-1, K, K]) and the greedy walk (choice, tokens [B, L]).
struct ClusterTail {
  const float* anchor;      // [B, d] anchor out vectors
  float* A;
  float* P;
  int32_t* choice;
  int32_t* tokens;
};
lilicorr_status_t launch_net_cluster(const lilicorr_head* h, int B, const int32_t* ids,
                                     const float* logp, const float* hproj, const float* t,
                                     const float* cb, float* oi, uint32_t* status, cudaStream_t st,
                                     const ClusterTail* tail = nullptr);
extern int g_fused_enabled;   // 0 never, 1 by batch size (default), 2 the one-CTA kernel
                              // always, 3 the cluster kernel always
constexpr int FUSED_MIN_B = 8;

lilicorr_status_t launch_target_norm(const void* T, lilicorr_dtype_t dt, int B, int n_tgt, int H,
                                     const float* gain, void* tn, lilicorr_dtype_t tn_dt,
                                     cudaStream_t st);
lilicorr_status_t launch_node_build(const lilicorr_head* h, int B, const int32_t* ids,
                                    const float* logp, const float* hproj, void* c1,
                                    lilicorr_dtype_t c1_dt, float* x, uint32_t* status,
                                    cudaStream_t st);
lilicorr_status_t launch_rmsnorm(const float* x, int M, int D, const float* gain, void* y,
                                 lilicorr_dtype_t y_dt, cudaStream_t st);
lilicorr_status_t launch_attention(const float* qkv, int B, int L, int K, int D, int n_heads,
                                   const float* dist, const float* same, void* out,
                                   lilicorr_dtype_t out_dt, cudaStream_t st);
// bf16 attention core on warp-level tensor-core instructions (attention_tc.cu)
bool attention_tc_supported(int hd);
size_t attention_tc_smem_bytes(int LK, int hd, int L);
lilicorr_status_t launch_attention_tc(const void* qkv, int B, int L, int K, int D, int n_heads,
                                      const float* dist, const float* same, void* out,
                                      cudaStream_t st);
// the same core on tcgen05 (attention_umma.cu): 32- or 64-wide heads, up to 256 nodes per
// sequence; g_attn_umma (api.cu) says where the chain uses it
bool attention_umma_supported(int L, int K, int D, int n_heads);
lilicorr_status_t launch_attention_umma(const void* qkv, int B, int L, int K, int D, int n_heads,
                                        const float* dist, const float* same, void* out,
                                        uint32_t* status, cudaStream_t st);
extern int g_attn_umma;
lilicorr_status_t launch_fusion_input(const float* x, int B, int LK, int D, const float* gain,
                                      const float* t, void* fin, lilicorr_dtype_t dt,
                                      cudaStream_t st);
lilicorr_status_t launch_unit_rows(const float* src, int rows, int n, int ld_src, float* dst,
                                   int ld_dst, cudaStream_t st);

// (3)+(4) pair scores and greedy walk (pair_walk.cu)
struct PairWalkArgs {
  int B, L, K, d;
  const float* out; const float* in; int ld_vec;  // node rows, row stride in floats
  const float* anchor;                            // [B, d]
  float* A; float* P;                             // outputs (pair mode) or inputs (walk-only)
  const int32_t* ids;                             // [B, L, K] (walk)
  int32_t* choice; int32_t* tokens; float* margin;
  bool do_pairs, do_walk;
  int walk_mode;                                  // LILICORR_WALK_GREEDY / _VITERBI
  float sigma;                                    // score scale of the exact path (Viterbi)
  float* path_score;                              // [B] g of the chosen path (Viterbi), may be null
  uint32_t* counters;                             // [B] zeroed tickets (pairs + walk fused)
  bool scores_in_smem;                            // set by the launcher
};
lilicorr_status_t launch_pair_walk(const PairWalkArgs& a, cudaStream_t st);

}  // namespace lilicorr
