/*
 * lilicorr_testing.h - test hooks of the LiLiCorr library. Not part of the
 * selection path; they expose internal building blocks so tests can check them
 * one at a time.
 *
 * The path switches below (lilicorr_test_fused_path, lilicorr_test_attention_path) change
 * process-global dispatch state that every head and every host thread reads when it
 * enqueues a call. They are not synchronised: set it only while no other thread is enqueueing work through the library,
 * and put the default back afterwards.
 */
#ifndef LILICORR_TESTING_H_
#define LILICORR_TESTING_H_

#include "lilicorr.h"

#ifdef __cplusplus
extern "C" {
#endif

/* One linear layer as the scoring network runs it:
 *   C[M, N] = act(A[M, Kd] W[N, Kd]^T + bias[N]) + residual[M, N]
 * A, W, C row-major device arrays with leading dimensions lda, ldw, ldc (elements);
 * bias and residual (fp32, residual with leading dimension ldc) may be NULL;
 * act 0 = none, 1 = SiLU. path selects the kernel: 0 = the network's own choice,
 * 1 = tiled CUDA-core kernel, 2 = few-row (split-N) CUDA-core kernel,
 * 3 = tensor cores (bf16 A and W only; LILICORR_ERR_DTYPE otherwise),
 * 4 = tensor cores for one tile of rows (M <= 128, Kd <= 512 a multiple of 64, N a
 *     multiple of 32 (fp32 out) or 64 (bf16 out); LILICORR_ERR_SHAPE otherwise),
 * 5 = row-block CUDA-core kernel for fp32 A (Kd a multiple of 8, lda of 4, ldw of 8, A and
 *     W 16-byte aligned; LILICORR_ERR_SHAPE otherwise).
 * status: a device uint32 word that receives bounded-wait timeouts (may be NULL). */
lilicorr_status_t lilicorr_test_linear(const void* A, lilicorr_dtype_t a_dt, int lda, const void* W,
                                       lilicorr_dtype_t w_dt, int ldw, void* C,
                                       lilicorr_dtype_t c_dt, int ldc, int M, int N, int Kd,
                                       const float* bias, const float* residual, int act, int path,
                                       uint32_t* status, cudaStream_t stream);

/* The failure branch of the tensor-core linear layer's bounded waits (path 3 of
 * lilicorr_test_linear, with C = A W^T, bf16 A [M, Kd] and W [N, Kd] row-major, fp32 C
 * [M, N]), made to run: the kernel's producer issues none of its copies, so the MMA
 * warp waits on a barrier that nothing arrives on. Every wait gives up after wait_cycles
 * SM cycles (1e5 .. 4e9; the production limit is 4e9, about 2 s); the kernel then records
 * LILICORR_ERR_TIMEOUT in *status (a device uint32 word, required), stops issuing, frees
 * its tensor memory and returns, leaving the context usable. C receives unspecified
 * values. LILICORR_ERR_SHAPE for shapes the tensor-core kernel does not take. */
lilicorr_status_t lilicorr_test_linear_timeout(const void* A, const void* W, float* C, int M, int N,
                                               int Kd, long long wait_cycles, uint32_t* status,
                                               cudaStream_t stream);

/* Switch for the fused scoring-network kernels (bf16 heads with D = 256, 8 heads,
 * FFN 2D, L*K <= 128): mode 1 (the default) takes the cluster kernel (four CTAs per
 * sequence) while every sequence's cluster fits on the GPU and the one-CTA kernel for
 * calls of 8 or more sequences beyond that, mode 2 the one-CTA kernel for every call,
 * mode 3 the cluster kernel for every call, mode 0 neither (the chain of kernels), so a
 * test can run the paths on the same inputs. Process-wide; set it between calls, not
 * while another thread is enqueueing. Returns 1 if `head` (may be NULL) can take the
 * kernel that `mode` names, else 0. */
int lilicorr_test_fused_path(const lilicorr_head* head, int mode);

/* Switch for the chain's attention core (Sec. 3.2 and App. A: bidirectional attention
 * with the slot-distance and same-slot biases, bf16 heads): mode 1 runs it on the
 * tcgen05 tensor cores where the head width is 32 or 64 and a sequence has at most 256
 * nodes, mode 0 on the mma.sync kernel, mode 2 (the default) on tcgen05 for sequences of
 * exactly 256 nodes whose slots hold a multiple of 8 candidates and on mma.sync otherwise.
 * Process-wide, like the switch above. Returns the previous mode. */
int lilicorr_test_attention_path(int mode);

#ifdef __cplusplus
}
#endif
#endif /* LILICORR_TESTING_H_ */
