/*
 * elasto_ops.h -- stateless kernel-level entry points of libelasto. Each is
 * one step of the DN forward (Section 4.1, Eq. 2-7) that elasto_forward
 * composes; they exist so that every kernel can be checked on its own
 * against the fp64 definition of that step.
 *
 * All pointers are CUDA device memory of the current device, 16-byte aligned,
 * row-major, caller-owned. Calls are asynchronous on `stream` (void* =
 * cudaStream_t). `status_device` (nullable) is an int the kernels set to
 * ELASTO_ERR_TIMEOUT if one of their bounded device-side waits gives up.
 * Errors: ELASTO_ERR_INVALID_ARG for null pointers, non-positive or
 * unsupported sizes; ELASTO_ERR_CUDA for launch failures.
 */
#ifndef ELASTO_OPS_H
#define ELASTO_OPS_H

#include "elasto.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Epilogues fused into the tensor-core GEMM (acc = A W^T in fp32). */
typedef enum {
  ELASTO_EPI_BIAS_BF16 = 0,       /* out bf16 = acc + bias                  (QKV, Eq. 2) */
  ELASTO_EPI_BIAS_GELU_BF16 = 1,  /* out bf16 = GELU(acc + bias)            (FC1, Eq. 5) */
  ELASTO_EPI_BIAS_RESID_F32 = 2,  /* out fp32 += acc + bias                 (proj, FC2: residual) */
  ELASTO_EPI_BIAS_F32 = 3,        /* out fp32 = acc + bias */
  ELASTO_EPI_BIAS_RELU_BF16 = 4,  /* out bf16 = ReLU(acc + bias)            (conv + folded BN) */
  ELASTO_EPI_BIAS_RESID_RELU_BF16 = 5, /* out bf16 = ReLU(acc + bias + resid) (block output) */
  /* The same with A, W, resid and out in IEEE f16 (ResNet-50 path: f16 has
   * 3 more mantissa bits than bf16 at the same tensor-core rate) */
  ELASTO_EPI_BIAS_RELU_F16 = 6,       /* out f16 = ReLU(acc + bias)             (conv + folded BN) */
  ELASTO_EPI_BIAS_F16 = 7,            /* out f16 = acc + bias                   (shortcut projection) */
  ELASTO_EPI_BIAS_RESID_RELU_F16 = 8  /* out f16 = ReLU(acc + bias + resid)     (block output) */
} elasto_epilogue;

/* out[M,N] = epilogue(A[M,K] W[N,K]^T): A, W bf16 (f16 for the *_F16
 * epilogues), K contiguous; bias fp32 [N] or NULL (= 0); resid [M,N] of the
 * same 16-bit type only for the ..._RESID_RELU epilogues. Output
 * row stride is N. Requires K % 8 == 0, N % 2 == 0, M, N, K >= 1 (K may be 0:
 * then acc = 0). tcgen05 MMA (M = 128 tiles), TMA-fed, persistent grid. */
elasto_status elasto_op_gemm(void* stream, const void* A, const void* W, const float* bias, void* out,
                             const void* resid, int M, int N, int K, int epilogue, int* status_device);

/* y bf16 [rows, d] = LayerNorm(x fp32 [rows, d]) * gamma + beta, eps = 1e-6,
 * biased variance, statistics in fp32 (one warp per row). d % 64 == 0,
 * d <= 4096. */
elasto_status elasto_op_layernorm(void* stream, const float* x, const float* gamma, const float* beta,
                                  void* y, int rows, int d);

/* y fp32 [rows, cols] = softmax over each row of x fp32 [rows, cols]
 * (exp(x - max) / sum, one warp per row, warp-shuffle reductions). */
elasto_status elasto_op_softmax(void* stream, const float* x, float* y, int rows, int cols);

/* k x k convolution (Eq. 7's conv over the kept channels) as an implicit
 * GEMM: out f16 [B, Ho, Wo, N] = act(conv(x) + bias), Ho = (H + 2 pad - k) /
 * stride + 1 (likewise Wo), act = ReLU if relu != 0 else identity.
 *   x f16 [B, H, W, C] NHWC, C % 8 == 0;
 *   w f16 [N, k, k, Cp] with Cp = 16 if C <= 16, else C rounded up to 64;
 *     channels >= C zero (the packed layout the ResNet path uses: one
 *     64-channel group per k-block of the tensor-core GEMM, or for at most 16
 *     channels one tap per 16-wide k-block in the 32-byte swizzle);
 *   bias fp32 [N] or NULL. N % 2 == 0, stride 1 or 2.
 * No im2col buffer: each k-block is one 4-D TMA tile of x (padding read as
 * zeros, the stride by TMA traversal strides). */
elasto_status elasto_op_conv2d(void* stream, const void* x, int B, int H, int W, int C, const void* w, int N, int k,
                               int stride, int pad, const float* bias, int relu, void* out, int* status_device);

/* Multi-head attention over the kept heads (Eq. 3), all heads of width 64:
 * qkv bf16 [batch, n, 3, heads, 64] (q | k | v blocks, head-major, as the
 * QKV GEMM writes them) -> out bf16 [batch, n, heads * 64] (heads
 * concatenated in order, Eq. 2). Scale 1/8. 1 <= n <= 256. */
elasto_status elasto_op_attention(void* stream, const void* qkv, void* out, int batch, int n, int heads,
                                  int* status_device);

/* Self-test of the bounded device-side wait that every kernel above (and the
 * forward's kernels) uses instead of an unbounded spin: one thread waits on an
 * mbarrier of one arrival. armed != 0: the arrival is made first and the wait
 * returns at once (status untouched). armed == 0: nothing arrives, the wait
 * gives up after its limit (1 s), the kernel writes ELASTO_ERR_TIMEOUT to
 * *status_device (if it still holds 0) and returns; the context stays usable.
 * *elapsed_ns_device (uint64) receives the time waited. */
elasto_status elasto_op_bounded_wait(void* stream, int armed, int* status_device,
                                     unsigned long long* elapsed_ns_device);

/* Self-test of the grid-wide barrier of the one-image one-launch forward
 * (elasto_set_one_launch): a cooperative launch of one block per SM passes
 * two barriers (arrival counter and abort flag in sync_device, 2 uint32 of
 * device scratch, zeroed here on the stream). unreachable != 0: the second
 * barrier waits for arrivals that never come, gives up after its limit (1 s),
 * writes ELASTO_ERR_TIMEOUT to *status_device (if it still holds 0) and
 * raises the abort flag, so every block returns; the context stays usable.
 * *elapsed_ns_device (uint64): block 0's time in the two barriers. */
elasto_status elasto_op_grid_barrier(void* stream, int unreachable, unsigned* sync_device, int* status_device,
                                     unsigned long long* elapsed_ns_device);

#ifdef __cplusplus
}
#endif
#endif /* ELASTO_OPS_H */
