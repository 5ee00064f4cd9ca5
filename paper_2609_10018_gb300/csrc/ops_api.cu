// Stateless kernel-level entry points (elasto_ops.h): each DN forward step on
// its own, so every kernel can be checked against the fp64 definition of that
// step at arbitrary (odd, ragged) shapes.
#include "common.h"
#include "handle.h"
#include "elasto_internal.h"
#include "ptx.cuh"

using namespace elasto;

namespace {

// The bounded wait every kernel uses (mbar_wait: a time limit, then false),
// on an mbarrier of one arrival. armed != 0: that arrival is made first, so
// the wait returns at once; armed == 0: nothing ever arrives, the wait gives
// up after its limit and the kernel records ELASTO_ERR_TIMEOUT in *status
// and returns, leaving the context usable. *elapsed_ns: how long it waited.
__global__ void bounded_wait_kernel(int armed, int* status, unsigned long long* elapsed_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_barrier_init();
  if (armed) mbar_arrive(&bar);
  const uint64_t t0 = global_timer_ns();
  const bool ok = mbar_wait(&bar, 0);
  *elapsed_ns = global_timer_ns() - t0;
  if (!ok) record_status(status, ELASTO_ERR_TIMEOUT);
}

}  // namespace

extern "C" {

elasto_status elasto_op_bounded_wait(void* stream, int armed, int* status_device,
                                     unsigned long long* elapsed_ns_device) {
  clear_error();
  if (!status_device || !elapsed_ns_device) {
    set_error("elasto_op_bounded_wait: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  elasto_status st = check_device();
  if (st != ELASTO_OK) return st;
  bounded_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(armed, status_device, elapsed_ns_device);
  ELASTO_CUDA_TRY(cudaGetLastError());
  return ELASTO_OK;
}


elasto_status elasto_op_grid_barrier(void* stream, int unreachable, unsigned* sync_device, int* status_device,
                                     unsigned long long* elapsed_ns_device) {
  clear_error();
  if (!sync_device || !status_device || !elapsed_ns_device) {
    set_error("elasto_op_grid_barrier: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  elasto_status st = check_device();
  if (st != ELASTO_OK) return st;
  ELASTO_CUDA_TRY(pk_barrier_selftest(static_cast<cudaStream_t>(stream), unreachable, sync_device, status_device,
                                      elapsed_ns_device));
  return ELASTO_OK;
}

elasto_status elasto_op_gemm(void* stream, const void* A, const void* W, const float* bias, void* out,
                             const void* resid, int M, int N, int K, int epilogue, int* status_device) {
  clear_error();
  if (!out || M <= 0 || N <= 0 || K < 0 || (K > 0 && (!A || !W)) || epilogue < 0 || epilogue > 8 ||
      ((epilogue == ELASTO_EPI_BIAS_RESID_RELU_BF16 || epilogue == ELASTO_EPI_BIAS_RESID_RELU_F16) && !resid)) {
    set_error("elasto_op_gemm: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  elasto_status st = check_device();
  if (st != ELASTO_OK) return st;
  GemmPlan p;
  st = gemm_plan(&p, static_cast<const bf16*>(A), M, static_cast<const bf16*>(W), N, K, bias, out, N, epilogue,
                 status_device);
  if (st != ELASTO_OK) return st;
  if (epilogue == ELASTO_EPI_BIAS_RESID_RELU_BF16 || epilogue == ELASTO_EPI_BIAS_RESID_RELU_F16) {
    st = gemm_set_residual_source(&p, resid, M);
    if (st != ELASTO_OK) return st;
  }
  ELASTO_CUDA_TRY(gemm_launch(p, M, static_cast<cudaStream_t>(stream)));
  return ELASTO_OK;
}

elasto_status elasto_op_conv2d(void* stream, const void* x, int B, int H, int W, int C, const void* w, int N, int k,
                               int stride, int pad, const float* bias, int relu, void* out, int* status_device) {
  clear_error();
  if (!x || !w || !out || B <= 0 || H <= 0 || W <= 0 || C <= 0 || N <= 0 || k <= 0 || stride <= 0 || pad < 0) {
    set_error("elasto_op_conv2d: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  elasto_status st = check_device();
  if (st != ELASTO_OK) return st;
  GemmPlan p;
  st = gemm_plan_conv(&p, x, B, H, W, C, k, stride, pad, w, N, bias, out, N, relu ? EPI_BIAS_RELU_F16 : EPI_BIAS_F16,
                      status_device);
  if (st != ELASTO_OK) return st;
  ELASTO_CUDA_TRY(gemm_launch(p, B, static_cast<cudaStream_t>(stream)));
  return ELASTO_OK;
}

elasto_status elasto_op_layernorm(void* stream, const float* x, const float* gamma, const float* beta, void* y,
                                  int rows, int d) {
  clear_error();
  if (!x || !gamma || !beta || !y || rows <= 0 || d <= 0) {
    set_error("elasto_op_layernorm: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (d % 64 != 0 || d > 1024) {
    set_error("elasto_op_layernorm: d must be a multiple of 64 up to 1024");
    return ELASTO_ERR_UNSUPPORTED;
  }
  ELASTO_CUDA_TRY(
      layernorm_launch(x, gamma, beta, static_cast<bf16*>(y), rows, d, d, static_cast<cudaStream_t>(stream)));
  return ELASTO_OK;
}

elasto_status elasto_op_softmax(void* stream, const float* x, float* y, int rows, int cols) {
  clear_error();
  if (!x || !y || rows <= 0 || cols <= 0) {
    set_error("elasto_op_softmax: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  ELASTO_CUDA_TRY(softmax_launch(x, y, rows, cols, static_cast<cudaStream_t>(stream)));
  return ELASTO_OK;
}

elasto_status elasto_op_attention(void* stream, const void* qkv, void* out, int batch, int n, int heads,
                                  int* status_device) {
  clear_error();
  if (!qkv || !out || batch <= 0 || n <= 0 || heads <= 0) {
    set_error("elasto_op_attention: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  elasto_status st = check_device();
  if (st != ELASTO_OK) return st;
  AttnPlan p;
  st = attn_plan(&p, static_cast<const bf16*>(qkv), static_cast<bf16*>(out), batch, n, heads, status_device);
  if (st != ELASTO_OK) return st;
  ELASTO_CUDA_TRY(attn_launch(p, batch, static_cast<cudaStream_t>(stream)));
  return ELASTO_OK;
}

}  // extern "C"
