/*
 * lilicorr.h - C ABI of the LiLiCorr per-block draft-selection path on sm_103a.
 *
 * After a block drafter emits per-slot logits [B, L, V], the path
 *   (1) keeps each slot's top-K candidates and log-normaliser      (Sec. 3.2; App. A "Serving")
 *   (2) runs the scoring network once over all B*L*K candidates,
 *       producing unit out/in vectors and an anchor out vector     (Sec. 3.2; App. A "Architecture")
 *   (3) scores adjacent slots by cosine similarity                   (Eq. "pair"; Sec. 3.5)
 *   (4) commits one candidate per slot by a greedy left-to-right walk (Sec. 3.5)
 * and returns the chosen L token ids per sequence.
 *
 * Conventions shared by every call:
 *   - Tensor arguments are DEVICE pointers unless a name says host_. The caller
 *     owns them; they are dense, row-major, and 16-byte aligned. The library owns
 *     only what lilicorr_head_create allocates.
 *   - Calls are asynchronous on the given stream: no host synchronisation, no
 *     allocation (scratch comes from the caller's workspace), so a sequence of
 *     calls can be captured in a CUDA graph. lilicorr_head_create/destroy and
 *     lilicorr_get_device_status are the exceptions and synchronise.
 *   - Argument and shape errors are detected on the host and returned before any
 *     work is enqueued. Errors found on the device (a non-finite logit row) are
 *     recorded in the workspace's status word; read it with
 *     lilicorr_get_device_status. Launch failures return LILICORR_ERR_CUDA.
 *   - Index conventions: slot s in [0, L) is the s-th drafted slot (the paper's
 *     slot s+1; slot 0 of the paper is the anchor). Candidate k in [0, K) is the
 *     k-th largest logit of its slot; equal logits order by lower token id and
 *     -0.0 equals +0.0. Node j = s*K + k.
 *   - Workspaces must be zero-filled once before first use (lilicorr_workspace_init);
 *     every call leaves them reusable. Two calls that run concurrently must not
 *     share a workspace.
 *   - lilicorr_select_block and lilicorr_embed_in_out run the candidate-independent
 *     projections on two side streams owned by the head (the drafter-state
 *     projection on one, the target-state chain on the other), forked from and
 *     joined back to the caller's stream (fork/join nodes under graph capture).
 *     Calls that use one head must be issued from one host thread at a time.
 */
#ifndef LILICORR_H_
#define LILICORR_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LILICORR_VERSION 1
#define LILICORR_MAX_K 32          /* candidates per slot */
#define LILICORR_MAX_L 64          /* drafted slots per block */
#define LILICORR_MAX_NODES 512     /* L*K per sequence */
#define LILICORR_N_CONF 5          /* confidence scalars per candidate (App. A) */

typedef enum {
  LILICORR_OK = 0,
  LILICORR_ERR_ARG = 1,        /* null pointer, misaligned pointer, bad enum */
  LILICORR_ERR_SHAPE = 2,      /* size out of range or inconsistent with the head */
  LILICORR_ERR_DTYPE = 3,      /* unsupported dtype combination */
  LILICORR_ERR_CUDA = 4,       /* a CUDA runtime call or launch failed */
  LILICORR_ERR_NONFINITE = 5,  /* device: a logit row held NaN/+inf or was all -inf */
  LILICORR_ERR_TIMEOUT = 6,    /* device: a bounded wait gave up */
  LILICORR_ERR_WORKSPACE = 7   /* workspace too small */
} lilicorr_status_t;

typedef enum { LILICORR_F32 = 0, LILICORR_BF16 = 1 } lilicorr_dtype_t;

/* How the last step picks one candidate per slot: the greedy left-to-right walk of
 * Sec. 3.5, or the exact maximiser of the path score (App. E, Viterbi). */
typedef enum { LILICORR_WALK_GREEDY = 0, LILICORR_WALK_VITERBI = 1 } lilicorr_walk_t;

/* The paper's score scale sigma of the pair cosines (App. A "Architecture"). */
#define LILICORR_SIGMA 8.0f

/* Shapes of a scoring head (App. A; Table "hparams": D = 1024, d = 1024, 8 heads,
 * F = 2048, 2 layers, 5 captured target layers, K = 8, L = 15).
 *   H         drafter/target hidden width (input width of the two projections)
 *   D         head width; must be a multiple of n_heads; head dim D/n_heads <= 128
 *   d         in/out vector dimension d_e
 *   n_heads   attention heads
 *   ffn       feed-forward width F
 *   n_layers  Transformer layers
 *   L, K      drafted slots and candidates per slot (L*K <= LILICORR_MAX_NODES)
 *   V         vocabulary size (rows of the embedding table)
 *   n_tgt     captured target layers averaged into the target state
 *   dtype     storage type of the weights, the embedding table, the logits and
 *             the hidden states passed to every call that takes this head.
 *             F32: every step runs in fp32. BF16: matrix products take bf16
 *             operands with fp32 accumulation; residuals, norms, softmax and
 *             the vectors stay fp32. */
typedef struct {
  int H, D, d, n_heads, ffn, n_layers, L, K, V, n_tgt;
  lilicorr_dtype_t dtype;
} lilicorr_head_desc;

typedef struct lilicorr_head lilicorr_head;   /* opaque; device-resident weights */

const char* lilicorr_status_str(lilicorr_status_t s);
int lilicorr_version(void);

/* Number of elements the weight blob of `desc` must hold (0 if desc is invalid).
 * Blob order, each tensor row-major, Linear weights stored [out, in]:
 *   emb_w [D,H] emb_b [D]            projection of the frozen token embedding
 *   hid_w [D,H] hid_b [D]            projection of the drafter hidden state
 *   conf1_w [D,5] conf1_b [D] conf2_w [D,D] conf2_b [D]   confidence network
 *   slot [L,D] rank [K,D]            learned slot and rank tables
 *   tgt_norm [H] tgt_w [D,H] tgt_b [D]                      target state
 *   per layer i < n_layers:
 *     an [D] wq [D,D] bq [D] wk [D,D] bk [D] wv [D,D] bv [D] wo [D,D] bo [D]
 *     dist [n_heads, 2L-1] same [n_heads] fn [D] w1 [F,D] b1 [F] w2 [D,F] b2 [D]
 *   final_norm [D] fuse_w [D,3D] fuse_b [D]
 *   out_w [d,D] out_b [d] in_w [d,D] in_b [d] anc_w [d,D] anc_b [d]
 * (App. A "Architecture": node = sum of four terms; 2-layer bidirectional
 * pre-RMSNorm Transformer with per-head signed-slot-distance and same-slot
 * attention biases; fusion SiLU(W_f [x; t; x*t] + b_f); out/in/anchor heads.) */
size_t lilicorr_head_param_count(const lilicorr_head_desc* desc);

/* Upload a head. host_weight_blob holds lilicorr_head_param_count(desc) values of
 * desc->dtype in the order above; host_embed_table is the frozen token-embedding
 * table [V, H] of desc->dtype (App. A: the target's input embedding, held frozen).
 * The embedding projection is linear and frozen, so the head stores the folded
 * table E W_e^T + b_e [V, D] instead of E. Synchronous; allocates device memory
 * on the current device. On success *out owns it until lilicorr_head_destroy. */
lilicorr_status_t lilicorr_head_create(const lilicorr_head_desc* desc, const void* host_weight_blob,
                                       const void* host_embed_table, lilicorr_head** out);
lilicorr_status_t lilicorr_head_destroy(lilicorr_head* head);

/* Zero-fill a workspace (enqueued on stream). Required once before first use. */
lilicorr_status_t lilicorr_workspace_init(void* ws, size_t ws_bytes, cudaStream_t stream);

/* Step (1): top-K candidates and log-normaliser of `rows` logit rows of length V
 * (Sec. 3.2 top-K pool; App. A "Serving": top-K extraction fused with
 * vocabulary-wide normalisation). One pass over the logits.
 *   logits  [rows, V] of dtype (F32 or BF16)
 *   ids     [rows, K] int32, candidates by descending logit, ties to lower id
 *   logp    [rows, K] fp32, logits[ids] - lse
 *   lse     [rows] fp32, log sum_v exp(logits[v])
 *   ws      workspace of at least lilicorr_topk_lse_workspace_bytes(rows, V, K)
 * 1 <= K <= min(V, LILICORR_MAX_K). A row holding NaN or +inf, or only -inf,
 * sets LILICORR_ERR_NONFINITE in the device status; its outputs are undefined. */
size_t lilicorr_topk_lse_workspace_bytes(int rows, int V, int K);
lilicorr_status_t lilicorr_topk_lse(const void* logits, lilicorr_dtype_t dtype, int rows, int V,
                                    int K, int32_t* ids, float* logp, float* lse, void* ws,
                                    size_t ws_bytes, cudaStream_t stream);

/* Step (1) over a vocabulary split into P shards (the logits of a tensor-parallel LM
 * head, each rank holding the columns of its vocabulary slice). Each shard emits one
 * partial record per row; the records of all shards, gathered in shard order, merge into
 * exactly what lilicorr_topk_lse computes on the whole row (the same ids; the normaliser
 * up to fp32 rounding of the combination). The log-sum-exp combines associatively:
 * lse = M + log sum_p s_p exp(m_p - M), M = max_p m_p, and every global top-K element is
 * in its shard's top-K (the lower-id rule holds across shards through the ids).
 * Partial record of one row, lilicorr_topk_partial_bytes(K) = 8 + 8K bytes:
 *   float m;        the shard row's maximum logit (-inf if it has none)
 *   float s;        sum_v exp(logits[v] - m) over the shard row
 *   float val[K];   the shard row's K largest logits, descending, ties to the lower id
 *   int32 id[K];    their vocabulary ids (column + id_offset); -1 (val -inf) when the
 *                   shard row has fewer than K elements
 * lilicorr_topk_lse_partial: logits [rows, V] of dtype is the shard (V >= 1, any K <=
 *   LILICORR_MAX_K, K may exceed V), id_offset the vocabulary id of its column 0 (>= 0),
 *   partial [rows] records (device, 8-byte aligned), ws a zero-filled workspace of at least
 *   lilicorr_topk_lse_partial_workspace_bytes(rows, V, K) bytes. A shard row may be all
 *   -inf; non-finite results are reported by the merge.
 * lilicorr_topk_lse_merge: partials [P][rows] records (the shards' outputs in any order;
 *   the ids carry the offsets), 1 <= P and P*K <= 8192; ids/logp/lse as lilicorr_topk_lse;
 *   status: a device uint32 word (may be NULL) that receives LILICORR_ERR_NONFINITE for a
 *   row whose merged normaliser is not finite. */
size_t lilicorr_topk_partial_bytes(int K);
size_t lilicorr_topk_lse_partial_workspace_bytes(int rows, int V, int K);
lilicorr_status_t lilicorr_topk_lse_partial(const void* logits, lilicorr_dtype_t dtype, int rows,
                                            int V, int K, int32_t id_offset, void* partial,
                                            void* ws, size_t ws_bytes, cudaStream_t stream);
lilicorr_status_t lilicorr_topk_lse_merge(const void* partials, int P, int rows, int K,
                                          int32_t* ids, float* logp, float* lse, uint32_t* status,
                                          cudaStream_t stream);

/* Step (1) with the LM-head projection in front of it, fused: the logits
 * logits[r, v] = sum_h hidden[r, h] * w_vocab[v, h] (fp32 accumulation of bf16 products)
 * are formed tile by tile on the tensor cores and reduced in place to what
 * lilicorr_topk_lse returns for them (top-K ids by descending logit, ties to the lower id;
 * logp = logit - lse; lse = log sum_v exp(logit)), so the [rows, V] logits never reach
 * memory (the projection that produces the drafter's logits, Table "cost"; Sec. 3.2).
 *   hidden    [rows, H] bf16, the final hidden states of the rows (row-major)
 *   w_vocab   [V, H] bf16, the LM-head weight (row v produces logit v)
 *   ids, logp [rows, K]; lse [rows]
 *   ws        zero-filled workspace of at least lilicorr_lm_head_topk_workspace_bytes(rows,
 *             H, V, K) bytes (0: unsupported shape); its first word is the device status
 * H a multiple of 64, 1 <= K <= min(V, LILICORR_MAX_K); hidden, w_vocab and ws 16-byte
 * aligned. A non-finite normaliser (NaN or inf in the inputs) sets LILICORR_ERR_NONFINITE
 * in the device status. */
size_t lilicorr_lm_head_topk_workspace_bytes(int rows, int H, int V, int K);
lilicorr_status_t lilicorr_lm_head_topk(const void* hidden, const void* w_vocab, int rows, int H,
                                        int V, int K, int32_t* ids, float* logp, float* lse,
                                        void* ws, size_t ws_bytes, cudaStream_t stream);

/* Step (1) without a caller workspace. Not from the paper (it has no counterpart
 * there): an addition for callers that cannot allocate device memory at the point
 * where they select a block. Examples: a serving process whose memory pool has claimed
 * the free device memory up front, a runtime that forbids allocation after start-up
 * (cudaMalloc may synchronise the device and fail late), or a plug-in running on a
 * stream it does not own. It computes what lilicorr_topk_lse computes, same arguments
 * minus the workspace, but keeps its scratch (status word, per-row tickets, per-split
 * partial records) in one fixed array of lilicorr_topk_lse_noalloc_max_bytes() = 4 MiB
 * compiled into the library; every GPU that loads the library holds that array until
 * the process exits. It calls no cudaMalloc, cudaFree or allocating routine.
 *   - Sizes whose scratch would exceed the array are rejected with
 *     LILICORR_ERR_WORKSPACE before anything is enqueued (4 MiB covers, e.g., 4096
 *     rows of V = 151936 at K = 16; the scratch grows with rows and K).
 *   - The first call on each device looks up the array's device address (once per
 *     device, with that device current); make that first call before any stream
 *     capture.
 *   - Every call clears the array's status word and tickets on `stream` first (the
 *     array keeps whatever the previous call left) and then reuses it, so two calls
 *     that overlap on the GPU (different streams, or different host threads) race
 *     and give undefined results; order them on one stream.
 *   - A non-finite row is detected as in lilicorr_topk_lse, but the status word lives
 *     in the fixed array and is not reported. Such a row's lse comes out non-finite
 *     (NaN for a row holding NaN or +inf, -inf for a row of only -inf), which the
 *     caller can test; its ids and logp are undefined. */
size_t lilicorr_topk_lse_noalloc_max_bytes(void);
lilicorr_status_t lilicorr_topk_lse_noalloc(const void* logits, lilicorr_dtype_t dtype, int rows,
                                            int V, int K, int32_t* ids, float* logp, float* lse,
                                            cudaStream_t stream);

/* Step (2): the scoring network over B sequences' candidates (Sec. 3.2; App. A).
 *   ids, logp         [B, L, K] from step (1) (logp in rank order)
 *   drafter_hidden    [B, L, H] of head dtype, the drafter's state per slot
 *   target_hidden     [B, n_tgt, H] of head dtype, the captured target layers at
 *                     the last verified token
 *   out_vec, in_vec   [B, L, K, d] fp32 unit vectors o_{s,k}, i_{s,k}
 *   anchor_out        [B, d] fp32 unit vector o_0
 *   ws                at least lilicorr_workspace_bytes(head, B) */
size_t lilicorr_workspace_bytes(const lilicorr_head* head, int B);
lilicorr_status_t lilicorr_embed_in_out(const lilicorr_head* head, int B, const int32_t* ids,
                                        const float* logp, const void* drafter_hidden,
                                        const void* target_hidden, float* out_vec, float* in_vec,
                                        float* anchor_out, void* ws, size_t ws_bytes,
                                        cudaStream_t stream);

/* Step (3): matching terms of Eq. "pair" without the scale sigma (sigma never
 * changes an argmax): (L-1) K^2 + K cosines per sequence (Sec. 3.5).
 *   out_vec, in_vec [B, L, K, d] fp32, anchor_out [B, d] fp32 (any norm; the
 *   cosine divides by max(||v||, 1e-12))
 *   anchor_scores [B, K]         A[b,k]      = cos(o_0, i_{0,k})
 *   pair_scores   [B, L-1, K, K] P[b,s,k,k'] = cos(o_{s,k}, i_{s+1,k'}) */
lilicorr_status_t lilicorr_pair_scores(int B, int L, int K, int d, const float* out_vec,
                                       const float* in_vec, const float* anchor_out,
                                       float* anchor_scores, float* pair_scores,
                                       cudaStream_t stream);

/* Step (4): greedy walk (Sec. 3.5): c_0 = argmax_k A[k], c_s = argmax_k
 * P[s-1, c_{s-1}, k], ties to the lower k.
 *   anchor_scores [B, K], pair_scores [B, L-1, K, K] fp32; ids [B, L, K] int32
 *   choice [B, L] int32 (candidate index), tokens [B, L] int32 (= ids[b, s, choice])
 *   margin [B, L] fp32 best minus second-best score of each step (+inf when K = 1);
 *   may be NULL. */
lilicorr_status_t lilicorr_greedy_walk(int B, int L, int K, const float* anchor_scores,
                                       const float* pair_scores, const int32_t* ids,
                                       int32_t* choice, int32_t* tokens, float* margin,
                                       cudaStream_t stream);

/* Exact best path (App. E): the candidates c maximising
 *   g(c) = sigma * (A[c_0] + sum_{s>=1} P[s-1, c_{s-1}, c_s])
 * over all K^L paths, by one left-to-right sweep that keeps, per candidate, the best
 * path ending there and its predecessor (ties to the lower index), then a traceback
 * from the best final candidate (ties to the lower index). Same layouts as
 * lilicorr_greedy_walk; path_score [B] receives g of the chosen path (may be NULL).
 * sigma > 0 does not change the path; it scales path_score. */
lilicorr_status_t lilicorr_best_path(int B, int L, int K, const float* anchor_scores,
                                     const float* pair_scores, const int32_t* ids, float sigma,
                                     int32_t* choice, int32_t* tokens, float* path_score,
                                     cudaStream_t stream);

/* Local next-candidate distributions (Eq. "localar"): with node scores z = sigma * score,
 *   anchor_probs[b, k]      = softmax_k(sigma * A[b, :])[k]            (predecessor: the anchor)
 *   pair_probs[b, s, k, k'] = softmax_k'(sigma * P[b, s, k, :])[k']    (predecessor k at slot s)
 * anchor_scores [B, K], pair_scores [B, L-1, K, K] fp32 in; the probabilities fp32 out,
 * same layouts. sigma > 0 (the paper's LILICORR_SIGMA). */
lilicorr_status_t lilicorr_local_softmax(int B, int L, int K, const float* anchor_scores,
                                         const float* pair_scores, float sigma,
                                         float* anchor_probs, float* pair_probs,
                                         cudaStream_t stream);

/* Along a path choice [B, L] (candidate indices, e.g. a walk's choice or the ground
 * truth's): prob[b, s] = P(c_s | c_{s-1}) of Eq. "localar" (the anchor precedes slot 0),
 * gap[b, s] = z_s[c_s] - max_{k != c_s} z_s[k], the decision gap of Eq. "margin" (+inf when
 * K = 1), log_prob[b] = sum_s log prob[b, s]. A choice outside [0, K) gives NaN for its
 * step. Any output may be NULL. */
lilicorr_status_t lilicorr_path_probs(int B, int L, int K, const float* anchor_scores,
                                      const float* pair_scores, const int32_t* choice,
                                      float sigma, float* prob, float* gap, float* log_prob,
                                      cudaStream_t stream);

/* Coverage and prefix acceptance against ground-truth tokens truth [B, L] int32 (Sec. 3.3
 * "Oracle-prefix supervision"; Sec. 3.1): covered[b, s] = 1 if truth[b, s] is among
 * ids[b, s, :] (the top-K candidates) else 0; oracle_prefix[b] = the longest leading run of
 * covered slots; accepted[b] = the longest leading run of slots whose chosen token
 * tokens[b, s] equals the truth (the verifier keeps tokens up to the first mismatch).
 * ids [B, L, K], tokens [B, L] int32. Any output may be NULL. */
lilicorr_status_t lilicorr_block_acceptance(int B, int L, int K, const int32_t* ids,
                                            const int32_t* tokens, const int32_t* truth,
                                            int32_t* covered, int32_t* oracle_prefix,
                                            int32_t* accepted, cudaStream_t stream);

/* Steps (1)-(4) fused: raw inputs to the chosen tokens.
 *   logits [B, L, V], drafter_hidden [B, L, H], target_hidden [B, n_tgt, H], all of
 *   head dtype; tokens [B, L] int32. ws: lilicorr_workspace_bytes(head, B). */
lilicorr_status_t lilicorr_select_block(const lilicorr_head* head, int B, const void* logits,
                                        const void* drafter_hidden, const void* target_hidden,
                                        int32_t* tokens, void* ws, size_t ws_bytes,
                                        cudaStream_t stream);

/* lilicorr_select_block with the last step chosen by `walk`: LILICORR_WALK_GREEDY (the
 * same as lilicorr_select_block) or LILICORR_WALK_VITERBI (the exact best path, App. E,
 * fused into the pair-score kernel like the walk). */
lilicorr_status_t lilicorr_select_block_walk(const lilicorr_head* head, int B, const void* logits,
                                             const void* drafter_hidden,
                                             const void* target_hidden, lilicorr_walk_t walk,
                                             int32_t* tokens, void* ws, size_t ws_bytes,
                                             cudaStream_t stream);

/* Device view of a select_block workspace after the call, for inspection:
 * pointers into ws of the intermediates of the last call (ids [B,L,K] int32,
 * logp [B,L,K] fp32, lse [B,L] fp32, anchor [B,K] fp32, pair [B,L-1,K,K] fp32,
 * choice [B,L] int32). Any output pointer may be NULL. */
lilicorr_status_t lilicorr_select_block_intermediates(const lilicorr_head* head, int B, void* ws,
                                                      size_t ws_bytes, int32_t** ids, float** logp,
                                                      float** lse, float** anchor_scores,
                                                      float** pair_scores, int32_t** choice);

/* Number of kernel launches this library has enqueued in this process (host-side
 * count; replays of a captured CUDA graph do not pass through the library and are
 * not counted). Lets a caller verify how many kernels one call launches. */
uint64_t lilicorr_launch_count(void);

/* Read (and clear) the device status word of a workspace: synchronises `stream`,
 * returns LILICORR_OK or the first device-detected error since the last read. */
lilicorr_status_t lilicorr_get_device_status(void* ws, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* LILICORR_H_ */
