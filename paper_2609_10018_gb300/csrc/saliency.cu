// L1-norm saliency of the Compress stage (Section 4.1) on the GPU, and the
// kept tables it induces.
//
// Section 4.1 scores each row of a weight matrix by its average absolute
// magnitude and masks the lowest rows (Eq. 4, 6, 7). At the granularity the
// descendant networks keep (heads, MLP channels, inner conv channels), a unit
// owns several such rows; its saliency is the mean of their averages:
//   ViT head j:        its 64 output rows in each of W^Q, W^K, W^V and its 64
//                      input columns of W^O (the paper's rows of W^O);
//   ViT MLP channel c: row c of W1 and column c of W2;
//   ResNet S_a channel: conv1's output row and conv2's input slice;
//   ResNet S_b channel: conv2's output row and conv3's input column;
//   ViT embedding channel: the rows that write it (patch projection, W^O, W2)
//                      and the columns that read it (W_qkv, W1, classifier).
// The reductions are memory-bound passes over the weights (each weight read
// once): a warp per row for row averages, a thread per column for column
// averages, fp32 sums of |w|.
#include <math.h>

#include <algorithm>
#include <string>
#include <vector>

#include "common.h"
#include "elasto_internal.h"

namespace elasto {
namespace {

// out[r] = mean_c |W[r, c]| for W [R, C] (bf16 bits or fp32).
template <typename T>
__global__ void row_abs_mean_kernel(const T* __restrict__ W, int R, int C, float* __restrict__ out) {
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= R) return;
  float s = 0.0f;
  for (int c = lane; c < C; c += 32) s += fabsf(static_cast<float>(W[static_cast<size_t>(r) * C + c]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) out[r] = s / static_cast<float>(C);
}

// out[c] = mean_r |W[r, c]|: consecutive threads read consecutive columns.
template <typename T>
__global__ void col_abs_mean_kernel(const T* __restrict__ W, int R, int C, float* __restrict__ out) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= C) return;
  float s = 0.0f;
  for (int r = 0; r < R; ++r) s += fabsf(static_cast<float>(W[static_cast<size_t>(r) * C + c]));
  out[c] = s / static_cast<float>(R);
}

// Uploads a host tensor of `count` elements and reduces it as [R, C].
struct Reducer {
  int dtype;
  void* dev = nullptr;
  float* red = nullptr;
  size_t cap = 0, red_cap = 0;
  ~Reducer() {
    if (dev) cudaFree(dev);
    if (red) cudaFree(red);
  }
  cudaError_t reserve(size_t elems, size_t outs) {
    const size_t es = dtype == ELASTO_BF16 ? 2 : 4;
    if (elems * es > cap) {
      if (dev) cudaFree(dev);
      dev = nullptr;
      cap = elems * es;
      if (cudaError_t e = cudaMalloc(&dev, cap)) return e;
    }
    if (outs > red_cap) {
      if (red) cudaFree(red);
      red = nullptr;
      red_cap = outs;
      if (cudaError_t e = cudaMalloc(&red, outs * 4)) return e;
    }
    return cudaSuccess;
  }
  // rows: out [R] row averages; else out [C] column averages. Host result.
  cudaError_t reduce(const void* host, int R, int C, bool rows, std::vector<float>& out) {
    const size_t n = size_t(R) * C, es = dtype == ELASTO_BF16 ? 2 : 4;
    const int outs = rows ? R : C;
    if (cudaError_t e = reserve(n, outs)) return e;
    if (cudaError_t e = cudaMemcpy(dev, host, n * es, cudaMemcpyHostToDevice)) return e;
    if (rows) {
      const unsigned grid = (R + 7) / 8;
      if (dtype == ELASTO_BF16)
        row_abs_mean_kernel<bf16><<<grid, 256>>>(static_cast<const bf16*>(dev), R, C, red);
      else
        row_abs_mean_kernel<float><<<grid, 256>>>(static_cast<const float*>(dev), R, C, red);
    } else {
      const unsigned grid = (C + 255) / 256;
      if (dtype == ELASTO_BF16)
        col_abs_mean_kernel<bf16><<<grid, 256>>>(static_cast<const bf16*>(dev), R, C, red);
      else
        col_abs_mean_kernel<float><<<grid, 256>>>(static_cast<const float*>(dev), R, C, red);
    }
    if (cudaError_t e = cudaGetLastError()) return e;
    out.resize(outs);
    return cudaMemcpy(out.data(), red, size_t(outs) * 4, cudaMemcpyDeviceToHost);
  }
};

}  // namespace
}  // namespace elasto

using namespace elasto;

extern "C" {

elasto_status elasto_saliency(const elasto_model_desc* d, const elasto_weights* w, float* scores_a,
                              float* scores_b) {
  clear_error();
  if (!d || !w || !w->tensors || !scores_a || !scores_b ||
      (d->weight_dtype != ELASTO_F32 && d->weight_dtype != ELASTO_BF16)) {
    set_error("elasto_saliency: null argument or bad weight_dtype");
    return ELASTO_ERR_INVALID_ARG;
  }
  for (int i = 0; i < w->n_tensors; ++i)
    if (!w->tensors[i]) {
      set_error("elasto_saliency: null weight tensor " + std::to_string(i));
      return ELASTO_ERR_INVALID_ARG;
    }
  Reducer red{d->weight_dtype};
  std::vector<float> a, b;
  if (d->arch == ELASTO_ARCH_VIT) {
    const int L = d->layers, D = d->dim, H = d->heads, F = d->mlp;
    if (L <= 0 || H <= 0 || D != 64 * H || F <= 0 || w->n_tensors != 8 + 12 * L) {
      set_error("elasto_saliency: inconsistent ViT descriptor or tensor count");
      return ELASTO_ERR_INVALID_ARG;
    }
    for (int l = 0; l < L; ++l) {
      const int t0 = 4 + 12 * l;  // ln1_w, ln1_b, qkv_w, qkv_b, proj_w, proj_b, ln2_w, ln2_b, fc1_w, fc1_b, fc2_w, fc2_b
      ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 2], 3 * D, D, true, a));   // W^Q, W^K, W^V output rows
      ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 4], D, D, false, b));     // W^O input columns
      for (int j = 0; j < H; ++j) {
        double s = 0.0;
        for (int r = 0; r < 64; ++r) s += double(a[j * 64 + r]) + a[D + j * 64 + r] + a[2 * D + j * 64 + r] + b[j * 64 + r];
        scores_a[size_t(l) * H + j] = static_cast<float>(s / 256.0);
      }
      ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 8], F, D, true, a));      // W1 rows
      ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 10], D, F, false, b));    // W2 columns
      for (int c = 0; c < F; ++c) scores_b[size_t(l) * F + c] = 0.5f * (a[c] + b[c]);
    }
    return ELASTO_OK;
  }
  if (d->arch == ELASTO_ARCH_RESNET50) {
    static const int nb[4] = {3, 4, 6, 3}, wd[4] = {64, 128, 256, 512};
    int n_t = 7;
    for (int s = 0; s < 4; ++s) n_t += nb[s] * 15 + 5;
    if (w->n_tensors != n_t) {
      set_error("elasto_saliency: ResNet-50 expects " + std::to_string(n_t) + " weight tensors");
      return ELASTO_ERR_INVALID_ARG;
    }
    int t = 5, cin = 64;
    size_t off = 0;
    std::vector<float> c;
    for (int s = 0; s < 4; ++s)
      for (int i = 0; i < nb[s]; ++i) {
        const int W = wd[s];
        // conv1 [W, cin], conv2 [W, W, 3, 3], conv3 [4W, W]
        ELASTO_CUDA_TRY(red.reduce(w->tensors[t], W, cin, true, a));          // conv1 output rows
        ELASTO_CUDA_TRY(red.reduce(w->tensors[t + 5], W, W * 9, false, b));   // conv2 columns (cin, ky, kx)
        ELASTO_CUDA_TRY(red.reduce(w->tensors[t + 5], W, W * 9, true, c));    // conv2 output rows
        for (int k = 0; k < W; ++k) {
          double in = 0.0;
          for (int q = 0; q < 9; ++q) in += b[k * 9 + q];
          scores_a[off + k] = static_cast<float>(0.5 * (double(a[k]) + in / 9.0));
        }
        ELASTO_CUDA_TRY(red.reduce(w->tensors[t + 10], 4 * W, W, false, b));  // conv3 input columns
        for (int k = 0; k < W; ++k) scores_b[off + k] = 0.5f * (c[k] + b[k]);
        off += W;
        t += 15 + (i == 0 ? 5 : 0);
        cin = 4 * W;
      }
    return ELASTO_OK;
  }
  set_error("elasto_saliency: unknown arch");
  return ELASTO_ERR_INVALID_ARG;
}

elasto_status elasto_saliency_embed(const elasto_model_desc* d, const elasto_weights* w, float* scores_e) {
  clear_error();
  if (!d || !w || !w->tensors || !scores_e || d->arch != ELASTO_ARCH_VIT ||
      (d->weight_dtype != ELASTO_F32 && d->weight_dtype != ELASTO_BF16)) {
    set_error("elasto_saliency_embed: null argument, not a ViT, or bad weight_dtype");
    return ELASTO_ERR_INVALID_ARG;
  }
  const int L = d->layers, D = d->dim, H = d->heads, F = d->mlp, C = d->classes;
  if (L <= 0 || H <= 0 || D != 64 * H || F <= 0 || C <= 0 || d->patch <= 0 || d->img_c <= 0 ||
      w->n_tensors != 8 + 12 * L) {
    set_error("elasto_saliency_embed: inconsistent ViT descriptor or tensor count");
    return ELASTO_ERR_INVALID_ARG;
  }
  for (int i = 0; i < w->n_tensors; ++i)
    if (!w->tensors[i]) {
      set_error("elasto_saliency_embed: null weight tensor " + std::to_string(i));
      return ELASTO_ERR_INVALID_ARG;
    }
  // The rows that write channel c and the columns that read it: patch
  // projection rows, classifier columns, and per layer W_qkv / W1 columns and
  // W^O / W2 rows; the score is the mean of those 2 + 4L averages.
  Reducer red{d->weight_dtype};
  std::vector<double> sum(D, 0.0);
  std::vector<float> a;
  auto add = [&]() {
    for (int c = 0; c < D; ++c) sum[c] += a[c];
  };
  const int kpe = d->patch * d->patch * d->img_c;
  ELASTO_CUDA_TRY(red.reduce(w->tensors[0], D, kpe, true, a));  // patch_w [d, C, P, P] rows
  add();
  ELASTO_CUDA_TRY(red.reduce(w->tensors[4 + 12 * L + 2], C, D, false, a));  // head_w [C, d] columns
  add();
  for (int l = 0; l < L; ++l) {
    const int t0 = 4 + 12 * l;
    ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 2], 3 * D, D, false, a));  // W_qkv columns
    add();
    ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 4], D, D, true, a));      // W^O rows
    add();
    ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 8], F, D, false, a));     // W1 columns
    add();
    ELASTO_CUDA_TRY(red.reduce(w->tensors[t0 + 10], D, F, true, a));     // W2 rows
    add();
  }
  for (int c = 0; c < D; ++c) scores_e[c] = static_cast<float>(sum[c] / (2 + 4 * L));
  return ELASTO_OK;
}

elasto_status elasto_topk(const float* scores, int n, int k, int32_t* out) {
  if (!scores || !out || n <= 0 || k < 0 || k > n) {
    set_error("elasto_topk: null argument or k outside [0, n]");
    return ELASTO_ERR_INVALID_ARG;
  }
  std::vector<int32_t> idx(n);
  for (int i = 0; i < n; ++i) idx[i] = i;
  std::stable_sort(idx.begin(), idx.end(), [&](int32_t x, int32_t y) { return scores[x] > scores[y]; });
  std::sort(idx.begin(), idx.begin() + k);
  std::copy(idx.begin(), idx.begin() + k, out);
  return ELASTO_OK;
}

}  // extern "C"
