// Internal declarations shared by the translation units of libelasto.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "elasto.h"
#include "elasto_ops.h"

namespace elasto {

using bf16 = __nv_bfloat16;

// ---------------------------------------------------------------- errors
void set_error(const std::string& msg);
void clear_error();
elasto_status cuda_fail(cudaError_t e, const char* what);  // records "<what>: <cuda msg>"

#define ELASTO_CUDA_TRY(expr)                                  \
  do {                                                         \
    cudaError_t e_ = (expr);                                   \
    if (e_ != cudaSuccess) return ::elasto::cuda_fail(e_, #expr); \
  } while (0)

// ---------------------------------------------------------------- device facts
int num_sms();  // of the current device

// ---------------------------------------------------------------- launches
// Programmatic dependent launch. A kernel launched with launch_pdl may be
// scheduled while the kernel before it on the stream is still finishing, so
// its prologue (barrier set-up, TMEM allocation, descriptor prefetch) overlaps
// that kernel's tail. Such a kernel calls pdl_wait() before its first access
// to global memory: it returns once the previous kernel has completed and its
// writes are visible, so stream order holds for all data. pdl_trigger() lets
// the next kernel be scheduled (it still waits in its own pdl_wait()).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// ---------------------------------------------------------------- TMA maps
// 2-D bf16 tensor [outer][inner] (inner contiguous, row stride in bytes),
// box {box_inner, box_outer}, 128-byte swizzle, out-of-bounds reads as zero.
bool encode_tmap_2d(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_stride_bytes,
                    uint32_t box_inner, uint32_t box_outer, bool fp32 = false);
// 4-D f16 tensor (NHWC activations: dims {C, W, H, B}), byte strides of
// dims 1..3, box in traversed elements, traversal strides (the box loads
// ceil(box[i] / elem_strides[i]) elements along dim i), 128-byte swizzle.
// 16-bit f16 4-D map (NHWC activations), 128-byte swizzle, or 32-byte when
// sw32 (16-channel boxes: one 32-byte row per pixel).
bool encode_tmap_4d(CUtensorMap* tm, const void* base, const uint64_t dims[4], const uint64_t strides_bytes[3],
                    const uint32_t box[4], const uint32_t elem_strides[4], bool sw32 = false);
// 16-bit f16 2-D map with the 32-byte swizzle.
bool encode_tmap_2d_sw32(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint64_t row_stride_bytes,
                         uint32_t box_inner, uint32_t box_outer);
// Map of rank 1-5 (fp32 or bf16) for TMA stores of dense boxes: dims
// innermost first, byte strides of dims 1..rank-1, box in elements;
// unswizzled, or with the 128-byte swizzle (box rows of exactly 128 bytes).
bool encode_tmap_plain(CUtensorMap* tm, const void* base, int rank, const uint64_t* dims,
                       const uint64_t* strides_bytes, const uint32_t* box, bool fp32, bool sw128 = false);
// 3-D bf16 tensor [d2][d1][d0] with byte strides s1 (between d1 rows) and s2.
bool encode_tmap_3d(CUtensorMap* tm, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1,
                    uint64_t s2, uint32_t b0, uint32_t b1, uint32_t b2);

// ---------------------------------------------------------------- GEMM
enum GemmEpi : int {
  EPI_BIAS_BF16 = ELASTO_EPI_BIAS_BF16,
  EPI_BIAS_GELU_BF16 = ELASTO_EPI_BIAS_GELU_BF16,
  EPI_BIAS_RESID_F32 = ELASTO_EPI_BIAS_RESID_F32,
  EPI_BIAS_F32 = ELASTO_EPI_BIAS_F32,
  EPI_BIAS_RELU_BF16 = ELASTO_EPI_BIAS_RELU_BF16,
  EPI_BIAS_RESID_RELU_BF16 = ELASTO_EPI_BIAS_RESID_RELU_BF16,
  EPI_BIAS_RELU_F16 = ELASTO_EPI_BIAS_RELU_F16,
  EPI_BIAS_F16 = ELASTO_EPI_BIAS_F16,
  EPI_BIAS_RESID_RELU_F16 = ELASTO_EPI_BIAS_RESID_RELU_F16,
};

struct GemmArgs {
  int M, N, K;
  int bn;                 // N tile (multiple of 32, <= 256)
  const float* bias;      // [N] or null
  void* out;              // [*, ldo]
  int ldo;
  int* status;
  int stages;             // operand ring depth (<= 8)
  int b_stage;            // bytes of one B stage (both planes; half of B for a CTA pair)
  int cbufs;              // output staging buffers (16 KB each) for the TMA-store epilogues
  int b_planes;           // 2: W held as bf16 hi + lo planes (fp32-stored models), both multiplied
  int pair;               // 1: clusters of two CTAs sharing 256-row tiles (tcgen05 cta_group::2)
  int f16;                // 1: A, W, the residual and 16-bit outputs are f16 (the *_F16 epilogues), else bf16
  // Implicit-GEMM convolution (conv != 0): A is never materialised. An M
  // tile is a block of bw x bh output pixels of nb images; k-block kb = (tap,
  // 64-channel group) is loaded straight from the NHWC input by a 4-D TMA
  // tile at (cg * 64, ox0 * stride - pad + kx, oy0 * stride - pad + ky, b0),
  // the padding read as zeros; W's K axis is (ky, kx, channel padded to 64).
  int conv;
  int cv_ks, cv_stride, cv_pad, cv_cgroups;  // kernel size, stride, padding, 64-channel groups per tap
  int cv_ho, cv_wo, cv_bw, cv_bh, cv_nb;     // output size and the pixel block of one M tile
  int cv_batch;                              // images in this launch (set at launch)
  int cv_a_bytes;                            // bytes one A tile load delivers
  int resid_row_mod;                         // > 0: periodic residual source (gemm_set_residual_source)
  int m_reverse;                             // 1: tile rows scheduled last to first (L2 reuse of A)
  int k16;                                   // implicit conv on <= 16 channels: k-blocks of 16 (one tap each),
                                             // operands in the 32-byte swizzle
  int b_resident;                            // 1: all of W (one N tile) is loaded once per CTA and kept in
                                             // shared memory; the ring carries A only
  int ksplit;                                // > 1: split-K, tile t reduces k-block range t / (mt * nt) of
                                             // ksplit and writes its fp32 partial to out + split * split_stride
  long long split_stride;                    // elements between the partial sums of two splits
};

struct GemmPlan {
  CUtensorMap tmA, tmB, tmB2;  // tmB2: low bf16 plane of W (b_planes == 2)
  CUtensorMap tmC;        // output [M_cap, ldo] (bf16 or fp32), box 128 B x 128 rows, 128B swizzle
  CUtensorMap tmR;        // residual source of EPI_BIAS_RESID_F32 (the output itself by default)
  GemmArgs args;          // M here is the capacity the A map was encoded for
  int epi = 0;
  bool valid = false;
  // split-K residual plan (gemm_plan_split_resid): after the kernel,
  // rout[r, c] += rbias[c] + sum over splits of the partials, in split order
  const float* rbias = nullptr;
  float* rout = nullptr;
  int rldo = 0, rcap = 0;  // rout row stride; rows the partial buffer holds
  // optional LayerNorm of the finished rows, fused into that sum
  // (gemm_split_fuse_layernorm): ln_y = LN(rout) over the first ln_d channels
  const float* ln_g = nullptr;
  const float* ln_b = nullptr;
  bf16* ln_y = nullptr;
  int ln_d = 0;
};

// Pick the N tile for an M x N problem.
int gemm_pick_bn(int M, int N, int step = 32, bool pair = false);
// Build maps/arguments for out = epi(A[M_cap, K] W[N, K]^T). A and W must stay
// allocated for the plan's life.
// W_lo (optional): second bf16 plane so that W = W + W_lo carries ~16
// mantissa bits (used for models stored in fp32); both products accumulate.
// M_hint (optional, <= M_cap): the row count the tiling is chosen for (the
// plan still covers M_cap rows); small batches get narrower N tiles, more
// CTAs and deeper operand rings.
// ldw (optional, >= K): row stride of W (and W_lo) in elements, when W is the
// first K columns of a wider matrix (a mode's prefix of a shared packed copy).
elasto_status gemm_plan(GemmPlan* p, const bf16* A, int M_cap, const bf16* W, int N, int K, const float* bias,
                        void* out, int ldo, int epi, int* status, const bf16* W_lo = nullptr, int M_hint = 0,
                        int ldw = 0, int bn_force = 0);
// EPI_BIAS_RESID_F32 (out[r, :] += A W^T + bias) for at most M_rows rows with
// the reduction split over up to kSplitMax CTAs per tile when the tiles alone
// would leave most SMs idle (a long K on a few rows: FC2 at batch 1). The
// partial sums go to part [ksplit, M_rows, N] fp32 (kSplitMax * M_rows * N
// floats), then a second launch adds them in split order with the bias to
// out: deterministic. Falls back to the single-pass plan when splitting
// would not spread the work.
constexpr int kSplitMax = 8;
elasto_status gemm_plan_split_resid(GemmPlan* p, const bf16* A, int M_cap, const bf16* W, int N, int K,
                                    const float* bias, float* out, int ldo, int* status, const bf16* W_lo, int M_rows,
                                    int ldw, float* part);
// For a split plan (does nothing otherwise, and says so by returning false):
// the launch that adds the partial sums also writes y = LayerNorm(out row)
// (gamma g, beta b, statistics over the first d_true of the N channels, the
// rest zero padding), the LayerNorm layernorm_launch computes (summed in
// another order), so the caller skips that launch. Needs ldo == N,
// N % 64 == 0, N <= 1024.
bool gemm_split_fuse_layernorm(GemmPlan* p, const float* g, const float* b, bf16* y, int d_true);

// Launch plans of one GEMM for a few batch sizes: the forward picks the plan
// made for the smallest row count that covers its rows.
struct GemmPlanSet {
  static constexpr int kMax = 4;
  GemmPlan plan[kMax];
  int rows[kMax] = {};
  int n = 0;
  const GemmPlan& pick(int M) const {
    for (int i = 0; i < n; ++i)
      if (M <= rows[i]) return plan[i];
    return plan[n - 1];
  }
};
// Residual epilogues: read the addend from src [M_cap, ldo] (fp32 for
// RESID_F32, 16-bit for the RESID_RELU ones) instead of the output
// (out = src + acc + bias). The 16-bit residual epilogues need it.
// row_period > 0: the addend repeats every row_period rows and src holds
// M_cap >= row_period + 128 of them; output row r adds src row r mod period
// (a tile starting at m0 reads rows m0 mod period ... + 127).
elasto_status gemm_set_residual_source(GemmPlan* p, const void* src, int M_cap, int row_period = 0);
// Per-tap K stride of an implicit-GEMM convolution's weights: 16 for up to 16
// channels (one 16-wide k-block per tap, 32-byte swizzle), else C rounded up
// to 64 (64-channel k-blocks).
inline int conv_tap_stride(int C) { return C <= 16 ? 16 : (C + 63) / 64 * 64; }
// Implicit-GEMM k x k convolution (stride, padding `pad`) of the f16 NHWC
// input x [B_cap, H, W, C] (C % 8 == 0) with W [N, k * k * conv_tap_stride(C)]
// f16 (each tap's channels zero-padded), out = epi(conv + bias) f16 [B_cap,
// Ho, Wo, ldo] (EPI_BIAS_RELU_F16 or EPI_BIAS_F16). gemm_launch's M is the
// batch.
// Ho_out / Wo_out > 0 replace the output size (a smaller output window).
elasto_status gemm_plan_conv(GemmPlan* p, const void* x, int B_cap, int H, int W, int C, int k, int stride, int pad,
                             const void* Wt, int N, const float* bias, void* out, int ldo, int epi, int* status,
                             int Ho_out = 0, int Wo_out = 0);
// Stride-1 convolution without padding of an input already padded in memory,
// x [B_cap, Hp, Wp, C] f16, whose kernel rows are kw * C == 64 contiguous
// values: kernel row ky of output pixel (y, x) reads x[b, y + ky, x .. x + kw
// - 1, :], which is one 64-wide k-block. W [N, kh * kw * C] f16 in (ky, kx,
// c) order; out as for gemm_plan_conv, over Ho = Hp - kh + 1, Wo = Wp - kw + 1
// or the smaller window Ho_out x Wo_out.
elasto_status gemm_plan_conv_rows(GemmPlan* p, const void* x, int B_cap, int Hp, int Wp, int C, int kh, int kw,
                                  const void* Wt, int N, const float* bias, void* out, int ldo, int epi, int* status,
                                  int Ho_out = 0, int Wo_out = 0);
// Launch for the first M (<= M_cap) rows.
cudaError_t gemm_launch(const GemmPlan& p, int M, cudaStream_t s);
cudaError_t gemm_init_attributes();

// ---------------------------------------------------------------- attention
struct AttnPlan {
  CUtensorMap tmQ, tmKV;
  const bf16* qkv;
  bf16* out;
  int n, n_pad, heads, batch_cap;
  int blk_stride, head_stride;  // column of (q|k|v block b, head j) = b * blk_stride + j * head_stride
  int* status;
  bool valid = false;
};
// interleaved: qkv columns are [head][q|k|v][64] instead of [q|k|v][head][64].
elasto_status attn_plan(AttnPlan* p, const bf16* qkv, bf16* out, int batch_cap, int n, int heads, int* status,
                        bool interleaved = false);
cudaError_t attn_launch(const AttnPlan& p, int batch, cudaStream_t s);
cudaError_t attn_init_attributes();
// The CNN classifier's shared-memory limit (its pooled rows: 8 x d fp32, up
// to d = kCnnMaxFeatures).
constexpr int kCnnMaxFeatures = 4096;
cudaError_t cnn_init_attributes();

// ---------------------------------------------------------------- small kernels
// y [rows, d] bf16 = LayerNorm of x [rows, d] fp32 (eps 1e-6) with statistics
// over the first d_true channels; channels [d_true, d) of x must be zero and
// of g, b zero (the padding of a pruned embedding width). d % 64 == 0, d <= 1024.
cudaError_t layernorm_launch(const float* x, const float* g, const float* b, bf16* y, int rows, int d, int d_true,
                             cudaStream_t s);
cudaError_t softmax_launch(const float* x, float* y, int rows, int cols, cudaStream_t s);
// images [B, H, W, C] -> A [B * n, P*P*C] bf16 in token order: row b*n is the
// class token's slot (zeros), row b*n + 1 + p holds patch p in (ky, kx, c)
// order. 16-byte copies when the images are bf16 and P*C % 8 == 0.
cudaError_t patch_rows_launch(const void* images, int img_dtype, int B, int H, int W, int C, int P, bf16* A,
                              cudaStream_t s);
// dst [B * n, d] fp32 = the per-token addend of the patch projection, tiled
// over the batch: row 0 of an image = cls + pos[0], row t >= 1 = pos[t] + b_pe.
cudaError_t token_addend_launch(const float* cls, const float* pos, const float* patch_b, int n, int d, int B,
                                float* dst, cudaStream_t s);
// logits[b, c] = LN(X[b * n, :]) . head_w[c, :] + head_b[c], all fp32; rows of
// width d, LayerNorm statistics over the first d_true channels (the rest zero).
cudaError_t head_launch(const float* X, int B, int n, int d, int d_true, const float* g, const float* b, const float* Wh,
                        const float* bh, int C, float* logits, cudaStream_t s);
// gathers for create-time packing
cudaError_t gather_rows_bf16(const bf16* src, int cols, const int32_t* idx, int nidx, bf16* dst, cudaStream_t s);
cudaError_t gather_cols_bf16(const bf16* src, int rows, int cols, const int32_t* idx, int nidx, bf16* dst,
                             cudaStream_t s);
cudaError_t gather_f32(const float* src, const int32_t* idx, int nidx, float* dst, cudaStream_t s);  // -1: zero
// dst [nr, nc] = src[ri, ci] of a row-major source with src_cols columns; -1 in ri or ci gives zero.
cudaError_t gather2d_bf16(const bf16* src, int src_cols, const int32_t* ri, int nr, const int32_t* ci, int nc, bf16* dst,
                          cudaStream_t s);
cudaError_t gather2d_f32(const float* src, int src_cols, const int32_t* ri, int nr, const int32_t* ci, int nc,
                         float* dst, cudaStream_t s);
cudaError_t convert_to_bf16(const void* src, int src_dtype, size_t n, bf16* dst, cudaStream_t s);
// dst = bf16(x - bf16(x)) for fp32 sources (the low plane of a bf16 pair); zeros for bf16 sources.
cudaError_t convert_to_bf16_lo(const void* src, int src_dtype, size_t n, bf16* dst, cudaStream_t s);
cudaError_t convert_to_f32(const void* src, int src_dtype, size_t n, float* dst, cudaStream_t s);

}  // namespace elasto
