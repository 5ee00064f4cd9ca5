// Memory-bound kernels of the DN forward and create-time packing:
//  - LayerNorm (pre-norm blocks and the class-token norm, Section 4.1 / 5.2):
//    one warp per row, fp32 statistics, vector loads, warp-shuffle reductions;
//  - row softmax (Eq. 3's softmax as a standalone op): one warp per row;
//  - patch extraction for the patch projection (N = HW/P^2 patches, Section
//    4.1) and the class-token rows of the residual stream;
//  - class-token LayerNorm + linear classifier in fp32;
//  - the index gathers that build each mode's packed weights (the structured
//    masks of Eq. 4 and 6 applied as deletion), and dtype conversions.
// Also: TMA map encoding, error strings, device facts.
#include <stdarg.h>
#include <stdio.h>

#include <mutex>

#include <cudaTypedefs.h>

#include "common.h"
#include "ptx.cuh"

namespace elasto {

// ---------------------------------------------------------------- errors
namespace {
thread_local std::string g_last_error;
}
void set_error(const std::string& msg) { g_last_error = msg; }
void clear_error() { g_last_error.clear(); }
const char* last_error_cstr() { return g_last_error.c_str(); }
elasto_status cuda_fail(cudaError_t e, const char* what) {
  set_error(std::string(what) + ": " + cudaGetErrorString(e));
  return ELASTO_ERR_CUDA;
}

int num_sms() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cached[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess) cached[dev] = v;
  }
  return cached[dev];
}

// ---------------------------------------------------------------- TMA maps
namespace {
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}
}  // namespace

bool encode_tmap_2d(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_stride_bytes,
                    uint32_t box_inner, uint32_t box_outer, bool fp32) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return enc(tm, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
             const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_4d(CUtensorMap* tm, const void* base, const uint64_t dims[4], const uint64_t strides_bytes[3],
                    const uint32_t box[4], const uint32_t elem_strides[4], bool sw32) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t d[4] = {dims[0], dims[1], dims[2], dims[3]};
  cuuint64_t st[3] = {strides_bytes[0], strides_bytes[1], strides_bytes[2]};
  cuuint32_t bx[4] = {box[0], box[1], box[2], box[3]};
  cuuint32_t es[4] = {elem_strides[0], elem_strides[1], elem_strides[2], elem_strides[3]};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void*>(base), d, st, bx, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, sw32 ? CU_TENSOR_MAP_SWIZZLE_32B : CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_2d_sw32(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_stride_bytes,
                         uint32_t box_inner, uint32_t box_outer) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_32B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_plain(CUtensorMap* tm, const void* base, int rank, const uint64_t* dims,
                       const uint64_t* strides_bytes, const uint32_t* box, bool fp32, bool sw128) {
  auto enc = get_encode();
  if (!enc || rank < 1 || rank > 5) return false;
  cuuint64_t d[5], st[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i + 1 < rank) st[i] = strides_bytes[i];
  }
  return enc(tm, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank,
             const_cast<void*>(base), d, st, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
             sw128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_3d(CUtensorMap* tm, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1,
                    uint64_t s2, uint32_t b0, uint32_t b1, uint32_t b2) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {s1, s2};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---------------------------------------------------------------- LayerNorm
namespace {

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

// One warp per row; each lane holds VEC float2 pairs (row width 64 * VEC).
// Rows are taken from the last to the first: the GEMM that produced x wrote
// its rows in increasing order, so the most recent ones (still in L2) are
// read first (8 % faster at ViT-B batch 256, where x is larger than L2).
// The statistics are over the first d_true channels: the remaining `pad`
// channels hold zeros (an embedding-pruned width padded to 64), so they add
// nothing to the sum and pad * mean^2 to the centred sum of squares, which is
// taken back out. gamma and beta are zero there, so y is zero there too.
template <int VEC>
__global__ void __launch_bounds__(256) layernorm_kernel(const float* __restrict__ x, const float* __restrict__ g,
                                                        const float* __restrict__ b, bf16* __restrict__ y,
                                                        int rows, float inv_d, float pad) {
  pdl_wait();
  pdl_trigger();
  const int row = rows - 1 - (blockIdx.x * 8 + (threadIdx.x >> 5));
  const int lane = threadIdx.x & 31;
  if (row < 0) return;
  constexpr int D = 64 * VEC;
  const float2* xr = reinterpret_cast<const float2*>(x + static_cast<size_t>(row) * D);
  float2 v[VEC];
  float s = 0.0f;
#pragma unroll
  for (int i = 0; i < VEC; ++i) {
    v[i] = xr[i * 32 + lane];
    s += v[i].x + v[i].y;
  }
  const float mean = warp_sum(s) * inv_d;
  float ss = 0.0f;
#pragma unroll
  for (int i = 0; i < VEC; ++i) {
    const float a = v[i].x - mean, c = v[i].y - mean;
    ss += a * a + c * c;
  }
  const float rstd = rsqrtf((warp_sum(ss) - pad * mean * mean) * inv_d + 1e-6f);
  const float2* g2 = reinterpret_cast<const float2*>(g);
  const float2* b2 = reinterpret_cast<const float2*>(b);
  uint32_t* yr = reinterpret_cast<uint32_t*>(y + static_cast<size_t>(row) * D);
#pragma unroll
  for (int i = 0; i < VEC; ++i) {
    const float2 gg = g2[i * 32 + lane], bb = b2[i * 32 + lane];
    yr[i * 32 + lane] = pack_bf16x2((v[i].x - mean) * rstd * gg.x + bb.x, (v[i].y - mean) * rstd * gg.y + bb.y);
  }
}

__global__ void __launch_bounds__(256) softmax_kernel(const float* __restrict__ x, float* __restrict__ y, int rows,
                                                      int cols) {
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const float* xr = x + static_cast<size_t>(row) * cols;
  float* yr = y + static_cast<size_t>(row) * cols;
  float m = -INFINITY;
  for (int c = lane; c < cols; c += 32) m = fmaxf(m, xr[c]);
  m = warp_max(m);
  float s = 0.0f;
  for (int c = lane; c < cols; c += 32) s += expf(xr[c] - m);
  s = warp_sum(s);
  const float inv = 1.0f / s;
  for (int c = lane; c < cols; c += 32) yr[c] = expf(xr[c] - m) * inv;
}

}  // namespace

cudaError_t layernorm_launch(const float* x, const float* g, const float* b, bf16* y, int rows, int d, int d_true,
                             cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (d % 64 != 0 || d_true <= 0 || d_true > d) return cudaErrorInvalidValue;
  const dim3 grid((rows + 7) / 8);
  const float inv_d = 1.0f / static_cast<float>(d_true), pad = static_cast<float>(d - d_true);
  switch (d / 64) {
#define LN_CASE(V) \
  case V: return launch_pdl(layernorm_kernel<V>, grid, dim3(256), 0, s, x, g, b, y, rows, inv_d, pad);
    LN_CASE(1) LN_CASE(2) LN_CASE(3) LN_CASE(4) LN_CASE(5) LN_CASE(6) LN_CASE(7) LN_CASE(8) LN_CASE(9)
    LN_CASE(10) LN_CASE(11) LN_CASE(12) LN_CASE(13) LN_CASE(14) LN_CASE(15) LN_CASE(16)
#undef LN_CASE
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t softmax_launch(const float* x, float* y, int rows, int cols, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  softmax_kernel<<<(rows + 7) / 8, 256, 0, s>>>(x, y, rows, cols);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- patches
namespace {

// A [B * n, K] in token order, K = P*P*C in (ky, kx, c) order. One thread per
// 16-byte piece (8 bf16): within a patch row, the P*C values (kx, c) are
// contiguous in the NHWC image, so a piece is one aligned 16-byte copy.
__global__ void patch_rows_vec_kernel(const bf16* __restrict__ img, int B, int H, int W, int C, int P,
                                      uint4* __restrict__ A) {
  pdl_wait();
  pdl_trigger();
  const int gw = W / P, np = (H / P) * gw, n = np + 1, K = P * P * C;
  const int row_pieces = K / 8, seg = P * C / 8;  // pieces per A row, per patch row
  const size_t total = static_cast<size_t>(B) * n * row_pieces;
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < total;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int j = static_cast<int>(t % row_pieces);
    const size_t row = t / row_pieces;
    const int tok = static_cast<int>(row % n), bb = static_cast<int>(row / n);
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (tok > 0) {
      const int p = tok - 1, ky = j / seg, jj = j - ky * seg;
      const int yy = (p / gw) * P + ky, x0 = (p % gw) * P;
      v = *reinterpret_cast<const uint4*>(img + ((static_cast<size_t>(bb) * H + yy) * W + x0) * C + jj * 8);
    }
    A[t] = v;
  }
}

// Generic version (fp32 images or P*C not a multiple of 8): one thread per element.
template <typename T>
__global__ void patch_rows_kernel(const T* __restrict__ img, int B, int H, int W, int C, int P, bf16* __restrict__ A) {
  pdl_wait();
  pdl_trigger();
  const int gw = W / P, np = (H / P) * gw, n = np + 1, K = P * P * C;
  const size_t total = static_cast<size_t>(B) * n * K;
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < total;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int k = static_cast<int>(t % K);
    const size_t row = t / K;
    const int tok = static_cast<int>(row % n), bb = static_cast<int>(row / n);
    float v = 0.0f;
    if (tok > 0) {
      const int p = tok - 1, c = k % C, kx = (k / C) % P, ky = k / (C * P);
      const T val = img[((static_cast<size_t>(bb) * H + (p / gw) * P + ky) * W + (p % gw) * P + kx) * C + c];
      if constexpr (sizeof(T) == 2)
        v = __bfloat162float(val);
      else
        v = static_cast<float>(val);
    }
    A[t] = __float2bfloat16_rn(v);
  }
}

__global__ void token_addend_kernel(const float* __restrict__ cls, const float* __restrict__ pos,
                                    const float* __restrict__ pb, int n, int d, size_t total, float* __restrict__ dst) {
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < total;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(t % d);
    const int tok = static_cast<int>((t / d) % n);
    dst[t] = tok == 0 ? cls[c] + pos[c] : pos[static_cast<size_t>(tok) * d + c] + pb[c];
  }
}

unsigned grid_1d(size_t n) {
  const size_t b = (n + 255) / 256;
  return static_cast<unsigned>(b < 16384 ? (b > 0 ? b : 1) : 16384);
}

}  // namespace

cudaError_t patch_rows_launch(const void* images, int img_dtype, int B, int H, int W, int C, int P, bf16* A,
                              cudaStream_t s) {
  const int n = (H / P) * (W / P) + 1, K = P * P * C;
  if (img_dtype == ELASTO_BF16 && (P * C) % 8 == 0) {
    const size_t total = static_cast<size_t>(B) * n * (K / 8);
    return launch_pdl(patch_rows_vec_kernel, dim3(grid_1d(total)), dim3(256), 0, s, static_cast<const bf16*>(images),
                      B, H, W, C, P, reinterpret_cast<uint4*>(A));
  }
  const unsigned blocks = grid_1d(static_cast<size_t>(B) * n * K);
  if (img_dtype == ELASTO_BF16)
    return launch_pdl(patch_rows_kernel<bf16>, dim3(blocks), dim3(256), 0, s, static_cast<const bf16*>(images), B, H,
                      W, C, P, A);
  return launch_pdl(patch_rows_kernel<float>, dim3(blocks), dim3(256), 0, s, static_cast<const float*>(images), B, H,
                    W, C, P, A);
}

cudaError_t token_addend_launch(const float* cls, const float* pos, const float* patch_b, int n, int d, int B,
                                float* dst, cudaStream_t s) {
  const size_t total = static_cast<size_t>(B) * n * d;
  token_addend_kernel<<<grid_1d(total), 256, 0, s>>>(cls, pos, patch_b, n, d, total, dst);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- classifier
namespace {

constexpr int HEAD_IMGS = 8;                  // class-token rows per CTA
constexpr int HEAD_CPW = 4;                   // classes per warp, computed together
constexpr int HEAD_CLASSES = 8 * HEAD_CPW;    // classes per CTA

// grid (ceil(B / 8), ceil(C / 32)), 256 threads: LayerNorm of up to 8 class
// tokens into shared memory (fp32), then each warp computes 4 classes x 8
// images of dot products at once: every normalised float4 it reads from shared
// memory feeds 16 FMAs, every classifier float4 32.
// d is the row width of X and Wh; the LayerNorm statistics cover the first
// d_true channels (the rest are the zero padding of a pruned width).
__global__ void __launch_bounds__(256) head_kernel(const float* __restrict__ X, int B, int n, int d, int d_true,
                                                   const float* __restrict__ g, const float* __restrict__ bta,
                                                   const float* __restrict__ Wh, const float* __restrict__ bh, int C,
                                                   float* __restrict__ logits) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float sy[];  // [HEAD_IMGS][d]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b0 = blockIdx.x * HEAD_IMGS;
  const int nimg = min(HEAD_IMGS, B - b0);
  if (warp < nimg) {
    const float* xr = X + static_cast<size_t>(b0 + warp) * n * d;  // class token row
    float s = 0.0f;
    for (int c = lane; c < d_true; c += 32) s += xr[c];
    const float mean = warp_sum(s) / d_true;
    float ss = 0.0f;
    for (int c = lane; c < d_true; c += 32) {
      const float a = xr[c] - mean;
      ss += a * a;
    }
    const float rstd = rsqrtf(warp_sum(ss) / d_true + 1e-6f);
    for (int c = lane; c < d; c += 32) sy[warp * d + c] = c < d_true ? (xr[c] - mean) * rstd * g[c] + bta[c] : 0.0f;
  }
  __syncthreads();
  const int c0 = blockIdx.y * HEAD_CLASSES + warp * HEAD_CPW;
  if (c0 >= C) return;
  const float* wr[HEAD_CPW];
#pragma unroll
  for (int j = 0; j < HEAD_CPW; ++j) wr[j] = Wh + static_cast<size_t>(min(c0 + j, C - 1)) * d;
  float acc[HEAD_CPW][HEAD_IMGS];
#pragma unroll
  for (int j = 0; j < HEAD_CPW; ++j)
#pragma unroll
    for (int i = 0; i < HEAD_IMGS; ++i) acc[j][i] = 0.0f;
#pragma unroll 2
  for (int c = lane * 4; c < d; c += 128) {
    float4 wv[HEAD_CPW];
#pragma unroll
    for (int j = 0; j < HEAD_CPW; ++j) wv[j] = *reinterpret_cast<const float4*>(wr[j] + c);
#pragma unroll
    for (int i = 0; i < HEAD_IMGS; ++i) {
      if (i < nimg) {
        const float4 yv = *reinterpret_cast<const float4*>(sy + i * d + c);
#pragma unroll
        for (int j = 0; j < HEAD_CPW; ++j)
          acc[j][i] += wv[j].x * yv.x + wv[j].y * yv.y + wv[j].z * yv.z + wv[j].w * yv.w;
      }
    }
  }
#pragma unroll
  for (int j = 0; j < HEAD_CPW; ++j)
#pragma unroll
    for (int i = 0; i < HEAD_IMGS; ++i) {
      const float v = warp_sum(acc[j][i]);
      if (lane == 0 && i < nimg && c0 + j < C) logits[static_cast<size_t>(b0 + i) * C + c0 + j] = v + bh[c0 + j];
    }
}

}  // namespace

cudaError_t head_launch(const float* X, int B, int n, int d, int d_true, const float* g, const float* b,
                        const float* Wh, const float* bh, int C, float* logits, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  if (d % 4 != 0 || d_true <= 0 || d_true > d) return cudaErrorInvalidValue;
  dim3 grid((B + HEAD_IMGS - 1) / HEAD_IMGS, (C + HEAD_CLASSES - 1) / HEAD_CLASSES);
  return launch_pdl(head_kernel, grid, dim3(256), HEAD_IMGS * d * sizeof(float), s, X, B, n, d, d_true, g, b, Wh, bh,
                    C, logits);
}

// ---------------------------------------------------------------- packing
namespace {

__global__ void gather_rows_kernel(const bf16* __restrict__ src, int cols, const int32_t* __restrict__ idx,
                                   int nidx, bf16* __restrict__ dst) {
  const size_t total = static_cast<size_t>(nidx) * cols;
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < total;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const size_t r = t / cols, c = t % cols;
    dst[t] = src[static_cast<size_t>(idx[r]) * cols + c];
  }
}

__global__ void gather_cols_kernel(const bf16* __restrict__ src, int rows, int cols, const int32_t* __restrict__ idx,
                                   int nidx, bf16* __restrict__ dst) {
  const size_t total = static_cast<size_t>(rows) * nidx;
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < total;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const size_t r = t / nidx, c = t % nidx;
    const int32_t k = idx[c];
    dst[t] = k >= 0 ? src[r * cols + k] : __float2bfloat16_rn(0.0f);
  }
}

__global__ void gather_f32_kernel(const float* __restrict__ src, const int32_t* __restrict__ idx, int nidx,
                                  float* __restrict__ dst) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t < nidx) dst[t] = idx[t] >= 0 ? src[idx[t]] : 0.0f;
}

// dst [nr, nc] = src [ri, ci] (src row-major with src_cols columns); an index
// of -1 in either list gives a zero (padding rows or columns).
template <typename T>
__global__ void gather2d_kernel(const T* __restrict__ src, int src_cols, const int32_t* __restrict__ ri, int nr,
                                const int32_t* __restrict__ ci, int nc, T* __restrict__ dst) {
  const size_t total = static_cast<size_t>(nr) * nc;
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < total;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int r = ri[t / nc], c = ci[t % nc];
    dst[t] = (r >= 0 && c >= 0) ? src[static_cast<size_t>(r) * src_cols + c] : T(0.0f);
  }
}

template <typename T>
__global__ void to_bf16_kernel(const T* __restrict__ src, size_t n, bf16* __restrict__ dst) {
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < n;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    if constexpr (sizeof(T) == 2)
      dst[t] = src[t];
    else
      dst[t] = __float2bfloat16_rn(src[t]);
  }
}

template <typename T>
__global__ void to_f32_kernel(const T* __restrict__ src, size_t n, float* __restrict__ dst) {
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < n;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    if constexpr (sizeof(T) == 2)
      dst[t] = __bfloat162float(src[t]);
    else
      dst[t] = src[t];
  }
}

unsigned grid_for(size_t n) {
  const size_t b = (n + 255) / 256;
  return static_cast<unsigned>(b < 65536 ? (b > 0 ? b : 1) : 65536);
}

}  // namespace

cudaError_t gather_rows_bf16(const bf16* src, int cols, const int32_t* idx, int nidx, bf16* dst, cudaStream_t s) {
  if (nidx <= 0 || cols <= 0) return cudaSuccess;
  gather_rows_kernel<<<grid_for(static_cast<size_t>(nidx) * cols), 256, 0, s>>>(src, cols, idx, nidx, dst);
  return cudaGetLastError();
}
cudaError_t gather_cols_bf16(const bf16* src, int rows, int cols, const int32_t* idx, int nidx, bf16* dst,
                             cudaStream_t s) {
  if (nidx <= 0 || rows <= 0) return cudaSuccess;
  gather_cols_kernel<<<grid_for(static_cast<size_t>(rows) * nidx), 256, 0, s>>>(src, rows, cols, idx, nidx, dst);
  return cudaGetLastError();
}
cudaError_t gather2d_bf16(const bf16* src, int src_cols, const int32_t* ri, int nr, const int32_t* ci, int nc, bf16* dst,
                          cudaStream_t s) {
  if (nr <= 0 || nc <= 0) return cudaSuccess;
  gather2d_kernel<bf16><<<grid_for(static_cast<size_t>(nr) * nc), 256, 0, s>>>(src, src_cols, ri, nr, ci, nc, dst);
  return cudaGetLastError();
}
cudaError_t gather2d_f32(const float* src, int src_cols, const int32_t* ri, int nr, const int32_t* ci, int nc,
                         float* dst, cudaStream_t s) {
  if (nr <= 0 || nc <= 0) return cudaSuccess;
  gather2d_kernel<float><<<grid_for(static_cast<size_t>(nr) * nc), 256, 0, s>>>(src, src_cols, ri, nr, ci, nc, dst);
  return cudaGetLastError();
}
cudaError_t gather_f32(const float* src, const int32_t* idx, int nidx, float* dst, cudaStream_t s) {
  if (nidx <= 0) return cudaSuccess;
  gather_f32_kernel<<<(nidx + 255) / 256, 256, 0, s>>>(src, idx, nidx, dst);
  return cudaGetLastError();
}
cudaError_t convert_to_bf16(const void* src, int src_dtype, size_t n, bf16* dst, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  if (src_dtype == ELASTO_BF16)
    to_bf16_kernel<bf16><<<grid_for(n), 256, 0, s>>>(static_cast<const bf16*>(src), n, dst);
  else
    to_bf16_kernel<float><<<grid_for(n), 256, 0, s>>>(static_cast<const float*>(src), n, dst);
  return cudaGetLastError();
}
namespace {
__global__ void to_bf16_lo_kernel(const float* __restrict__ src, size_t n, bf16* __restrict__ dst) {
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < n;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const float x = src[t];
    dst[t] = __float2bfloat16_rn(x - __bfloat162float(__float2bfloat16_rn(x)));
  }
}
}  // namespace

cudaError_t convert_to_bf16_lo(const void* src, int src_dtype, size_t n, bf16* dst, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  if (src_dtype == ELASTO_BF16) return cudaMemsetAsync(dst, 0, n * sizeof(bf16), s);
  to_bf16_lo_kernel<<<grid_for(n), 256, 0, s>>>(static_cast<const float*>(src), n, dst);
  return cudaGetLastError();
}

cudaError_t convert_to_f32(const void* src, int src_dtype, size_t n, float* dst, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  if (src_dtype == ELASTO_BF16)
    to_f32_kernel<bf16><<<grid_for(n), 256, 0, s>>>(static_cast<const bf16*>(src), n, dst);
  else
    to_f32_kernel<float><<<grid_for(n), 256, 0, s>>>(static_cast<const float*>(src), n, dst);
  return cudaGetLastError();
}

}  // namespace elasto
