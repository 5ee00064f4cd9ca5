// ResNet-50 v1.5 descendant networks (Eq. 7), NHWC activations in IEEE f16.
//
// A DN keeps, per bottleneck block, a set S_a of conv1's output channels
// (= conv2's input channels) and a set S_b of conv2's output channels (=
// conv3's input channels); Eq. 7's channel masks zero everything else, which
// is computed as deleting it. At create time each mode's kept channels are
// gathered and every inference BatchNorm is folded into its convolution
// (W' = W * g / sqrt(var + eps) per output channel, b' = beta - mean * g /
// sqrt(var + eps)); kept counts are padded with zero channels to a multiple
// of 8 (a zero channel stays zero through bias 0 and ReLU and meets zero
// weights downstream, so the padding changes no output).
//
// Forward, all convolutions on the tcgen05 GEMM of gemm.cu:
//   stem     7x7/2 conv as a 4x4 stride-1 conv over the space-to-depth
//            image (2x2 pixel blocks -> 12 channels, padded to 16, with a
//            zero border): one kernel row of an output pixel is 64
//            contiguous values, one k-block (gemm_plan_conv_rows); + bias +
//            ReLU, then 3x3/2 max pool (padding never wins);
//   block    conv1 1x1: GEMM straight on the NHWC activation [B*H*W, cin];
//            conv2 3x3/stride: implicit GEMM (gemm_plan_conv): each k-block
//            (tap, 64 kept channels; 16 when at most 16 are kept) is a 4-D
//            TMA tile of the conv1 output, padding read as zeros, stride by
//            TMA traversal strides; + bias + ReLU;
//            projection (first block of a stage): 1x1/stride conv + bias
//            (an implicit GEMM too when the stride is 2);
//            conv3 1x1: GEMM + bias + shortcut + ReLU in the epilogue;
//   head     global average pool (fp32), classifier in fp32 (pooled rows
//            staged in shared memory).
//
// Operands are f16, not bf16: the tensor cores multiply both at the same rate
// (kind::f16 with f16 A and B, fp32 accumulation), and f16's 11-bit
// significand keeps the rounding of 53 stacked convolutions ~8x smaller.
// Post-BN ResNet activations stay far inside f16's range (|x| < 65504).
#include <math.h>
#include <string.h>

#include <algorithm>
#include <string>
#include <vector>

#include "common.h"
#include "elasto_internal.h"
#include "guard.h"

namespace elasto {

namespace {

constexpr double kBnEps = 1e-5;
constexpr int kStemC = 64;
constexpr int kStemK = 7 * 7 * 3;  // multiply-adds per output value of the 7x7 stem
// The stem runs as a 4x4 stride-1 convolution over the space-to-depth image
// (2x2 pixel blocks -> 12 channels, padded to 16) with a zero border of 2
// before and 1 after in memory: W [64, 4, 4, 16], one 64-wide k-block per
// kernel row (4 pixels x 16 channels, contiguous in memory).
constexpr int kS2dC = 16;
constexpr int kStemKs = 4 * 4 * kS2dC;
constexpr size_t kAlignB = 1024;

struct BlockShape {
  int cin, w, stride;
  bool proj;
  int hin, win, ho, wo;
};

int round8(int v) { return (v + 7) / 8 * 8; }

}  // namespace

// 16-bit operand storage. The GEMM interface types its operand pointers as
// bf16; on this path they hold IEEE f16 bits (GemmArgs::f16 is set by the
// *_F16 epilogues).
using F16Buf = bf16;

struct CnnBlockPack {
  int a = 0, b = 0, a_pad = 0, b_pad = 0;  // kept |S_a|, |S_b| and their padded widths
  int a_cp = 0;                            // conv2's per-tap K stride: conv_tap_stride(a_pad)
  F16Buf *w1 = nullptr, *w2 = nullptr, *w3 = nullptr;
  float *b1 = nullptr, *b2 = nullptr, *b3 = nullptr;
  GemmPlan conv1, conv2, conv3;
};

struct CnnMode {
  std::vector<CnnBlockPack> blocks;
  size_t packed_bytes = 0;
  int64_t macs = 0;
  int launches = 0;
};

struct CnnModel {
  elasto_model_desc d{};
  int n_modes = 0;
  Profiler prof;
  char* arena = nullptr;
  GuardedArena guards;  // guard zone after every arena buffer
  size_t arena_bytes = 0, shared_bytes = 0, workspace_bytes = 0;
  int h1 = 0, w1 = 0, hp = 0, wp = 0;  // stem output and pooled sizes
  std::vector<BlockShape> shapes;
  // mode-independent parameters
  F16Buf* stem_w = nullptr;
  float* stem_b = nullptr;
  std::vector<F16Buf*> down_w;
  std::vector<float*> down_b;
  float *fc_w = nullptr, *fc_b = nullptr;
  GemmPlan stem;
  std::vector<GemmPlan> down;  // per block (valid where the block has a projection)
  // workspace
  F16Buf *s2d = nullptr, *xa = nullptr, *xb = nullptr, *t1 = nullptr, *t2 = nullptr, *sc = nullptr;
  float* pooled = nullptr;
  void* img_stage = nullptr;
  float* logit_stage = nullptr;
  int* status = nullptr;
  std::vector<CnnMode> modes;
};

namespace {

std::vector<BlockShape> block_shapes(int hp, int wp) {
  static const int nb[4] = {3, 4, 6, 3}, wd[4] = {64, 128, 256, 512};
  std::vector<BlockShape> out;
  int cin = 64, h = hp, w = wp;
  for (int s = 0; s < 4; ++s)
    for (int i = 0; i < nb[s]; ++i) {
      BlockShape b{};
      b.cin = cin;
      b.w = wd[s];
      b.stride = (i == 0 && s > 0) ? 2 : 1;
      b.proj = i == 0;
      b.hin = h;
      b.win = w;
      b.ho = (h - 1) / b.stride + 1;  // 3x3, padding 1 (and the 1x1 projection at the same stride)
      b.wo = (w - 1) / b.stride + 1;
      out.push_back(b);
      cin = 4 * wd[s];
      h = b.ho;
      w = b.wo;
    }
  return out;
}

int n_tensors_expected() {
  int n = 5 + 2;
  for (const BlockShape& b : block_shapes(1, 1)) n += 15 + (b.proj ? 5 : 0);
  return n;
}

// ---------------------------------------------------------------- kernels

__device__ __forceinline__ void unpack8(const uint4& u, float (&f)[8]) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 v = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
    f[2 * i] = v.x;
    f[2 * i + 1] = v.y;
  }
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  const __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Space-to-depth of the image for the stem, with its zero border:
// S[b, 2 + y, 2 + x, (dy * 2 + dx) * 3 + c] = img[b, 2y + dy, 2x + dx, c] as
// f16 (zero past an odd-sized image), channels 12..15 zero, S [B, Hs + 3,
// Ws + 3, 16] zero outside y < Hs, x < Ws. One thread per S pixel (32 bytes
// out), from the last pixel to the first: the stem GEMM reads them first to
// last.
template <typename T>
__global__ void stem_s2d_kernel(const T* __restrict__ src, int B, int H, int W, int Hs, int Ws,
                                uint4* __restrict__ dst) {
  pdl_wait();
  pdl_trigger();
  const int Hp = Hs + 3, Wp = Ws + 3;
  const size_t total = static_cast<size_t>(B) * Hp * Wp;
  for (size_t t0 = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t0 < total;
       t0 += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const size_t t = total - 1 - t0;
    const int x = static_cast<int>(t % Wp) - 2;
    const size_t r = t / Wp;
    const int y = static_cast<int>(r % Hp) - 2;
    const size_t b = r / Hp;
    const bool inside = y >= 0 && y < Hs && x >= 0 && x < Ws;
    float v[16];
#pragma unroll
    for (int dy = 0; dy < 2; ++dy)
#pragma unroll
      for (int dx = 0; dx < 2; ++dx) {
        const int iy = 2 * y + dy, ix = 2 * x + dx;
        const bool in = inside && iy < H && ix < W;
#pragma unroll
        for (int c = 0; c < 3; ++c)
          v[(dy * 2 + dx) * 3 + c] = in ? static_cast<float>(src[((b * H + iy) * W + ix) * 3 + c]) : 0.0f;
      }
#pragma unroll
    for (int c = 12; c < 16; ++c) v[c] = 0.0f;
    dst[2 * t] = make_uint4(pack2(v[0], v[1]), pack2(v[2], v[3]), pack2(v[4], v[5]), pack2(v[6], v[7]));
    dst[2 * t + 1] = make_uint4(pack2(v[8], v[9]), pack2(v[10], v[11]), pack2(v[12], v[13]), pack2(v[14], v[15]));
  }
}


// 3x3 max pool, stride 2, padding 1 (padding cells are skipped, so they
// never win), f16 NHWC with C % 8 == 0. Exact: the max of f16 values.
__global__ void maxpool_kernel(const uint4* __restrict__ src, int H, int W, int C8, int Ho, int Wo, size_t total,
                               uint4* __restrict__ dst) {
  pdl_wait();
  pdl_trigger();
  for (size_t t = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < total;
       t += static_cast<size_t>(gridDim.x) * blockDim.x) {
    // pixels last to first: the stem GEMM wrote its rows first to last
    const size_t u = total - 1 - t;
    const int c8 = static_cast<int>(u % C8);
    const size_t p = u / C8;
    const int ox = static_cast<int>(p % Wo);
    const size_t r2 = p / Wo;
    const int oy = static_cast<int>(r2 % Ho);
    const size_t b = r2 / Ho;
    float m[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) m[j] = -INFINITY;
#pragma unroll
    for (int ky = 0; ky < 3; ++ky) {
      const int iy = 2 * oy - 1 + ky;
      if (iy < 0 || iy >= H) continue;
#pragma unroll
      for (int kx = 0; kx < 3; ++kx) {
        const int ix = 2 * ox - 1 + kx;
        if (ix < 0 || ix >= W) continue;
        float f[8];
        unpack8(src[((b * H + iy) * W + ix) * C8 + c8], f);
#pragma unroll
        for (int j = 0; j < 8; ++j) m[j] = fmaxf(m[j], f[j]);
      }
    }
    dst[u] = make_uint4(pack2(m[0], m[1]), pack2(m[2], m[3]), pack2(m[4], m[5]), pack2(m[6], m[7]));
  }
}

// Global average pool: dst[b, c] = mean over the HW pixels of src[b, :, c]
// (f16 in, fp32 sums and result). Item t = b * C8 + c8 (8 channels) is
// taken by the 4 adjacent threads 4t .. 4t + 3: thread j sums the pixels
// p = j (mod 4), the four partial sums are combined with shuffles inside
// the 4-lane group, and thread j writes channels 2j, 2j + 1.
__global__ void avgpool_kernel(const uint4* __restrict__ src, int HW, int C8, size_t total, float* __restrict__ dst) {
  pdl_wait();
  pdl_trigger();
  const unsigned group = 0xFu << (threadIdx.x & 28);  // this thread's 4-lane group
  for (size_t u = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; u < 4 * total;
       u += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const size_t t = u >> 2;
    const int j = static_cast<int>(u & 3);
    const int c8 = static_cast<int>(t % C8);
    const size_t b = t / C8;
    float s[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
    for (int p = j; p < HW; p += 4) {
      float f[8];
      unpack8(src[(b * HW + p) * C8 + c8], f);
#pragma unroll
      for (int k = 0; k < 8; ++k) s[k] += f[k];
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      s[k] += __shfl_xor_sync(group, s[k], 1);
      s[k] += __shfl_xor_sync(group, s[k], 2);
    }
    const float inv = 1.0f / static_cast<float>(HW);
    float2 w = make_float2(s[0], s[1]);
#pragma unroll
    for (int k = 1; k < 4; ++k)
      if (k == j) w = make_float2(s[2 * k], s[2 * k + 1]);
    reinterpret_cast<float2*>(dst + t * 8)[j] = make_float2(w.x * inv, w.y * inv);
  }
}

__device__ __forceinline__ float warp_sum32(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

constexpr int FC_IMGS = 8, FC_CPW = 4, FC_CLASSES = 8 * FC_CPW;

// logits[b, c] = pooled[b, :] . Wf[c, :] + bf[c] in fp32. grid (ceil(B / 8),
// ceil(C / 32)), 256 threads: the CTA first copies its 8 pooled rows into
// shared memory (zeros past the batch), then each warp computes 4 classes x 8
// images at once: every classifier float4 it loads feeds 32 FMAs and the
// pooled values come from shared memory, so the only global loads in the loop
// are the four independent classifier rows.
__global__ void __launch_bounds__(256) fc_kernel(const float* __restrict__ pooled, int B, int d,
                                                 const float* __restrict__ Wf, const float* __restrict__ bf, int C,
                                                 float* __restrict__ logits) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float4 sy4[];  // [FC_IMGS][d / 4]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b0 = blockIdx.x * FC_IMGS;
  const int nimg = min(FC_IMGS, B - b0);
  const int d4 = d / 4;
  for (int t = threadIdx.x; t < FC_IMGS * d4; t += blockDim.x) {
    const int i = t / d4;
    sy4[t] = i < nimg ? reinterpret_cast<const float4*>(pooled + static_cast<size_t>(b0 + i) * d)[t - i * d4]
                      : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  __syncthreads();
  const int c0 = blockIdx.y * FC_CLASSES + warp * FC_CPW;
  if (c0 >= C) return;
  const float4* wr[FC_CPW];
#pragma unroll
  for (int j = 0; j < FC_CPW; ++j) wr[j] = reinterpret_cast<const float4*>(Wf + static_cast<size_t>(min(c0 + j, C - 1)) * d);
  float acc[FC_CPW][FC_IMGS];
#pragma unroll
  for (int j = 0; j < FC_CPW; ++j)
#pragma unroll
    for (int i = 0; i < FC_IMGS; ++i) acc[j][i] = 0.0f;
#pragma unroll 4
  for (int c = lane; c < d4; c += 32) {
    float4 wv[FC_CPW];
#pragma unroll
    for (int j = 0; j < FC_CPW; ++j) wv[j] = wr[j][c];
#pragma unroll
    for (int i = 0; i < FC_IMGS; ++i) {
      const float4 yv = sy4[i * d4 + c];
#pragma unroll
      for (int j = 0; j < FC_CPW; ++j)
        acc[j][i] += wv[j].x * yv.x + wv[j].y * yv.y + wv[j].z * yv.z + wv[j].w * yv.w;
    }
  }
#pragma unroll
  for (int j = 0; j < FC_CPW; ++j)
#pragma unroll
    for (int i = 0; i < FC_IMGS; ++i) {
      const float v = warp_sum32(acc[j][i]);
      if (lane == 0 && i < nimg && c0 + j < C) logits[static_cast<size_t>(b0 + i) * C + c0 + j] = v + bf[c0 + j];
    }
}

}  // namespace

cudaError_t cnn_init_attributes() {
  return cudaFuncSetAttribute(fc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              FC_IMGS * kCnnMaxFeatures * static_cast<int>(sizeof(float)));
}

namespace {

unsigned grid_for(size_t n) {
  const size_t b = (n + 255) / 256;
  return static_cast<unsigned>(b < 16384 ? (b > 0 ? b : 1) : 16384);
}

cudaError_t stem_s2d_launch(const void* images, int dtype, int B, int H, int W, int Hs, int Ws, __half* dst,
                            cudaStream_t s) {
  const size_t total = static_cast<size_t>(B) * (Hs + 3) * (Ws + 3);
  if (total == 0) return cudaSuccess;
  uint4* d = reinterpret_cast<uint4*>(dst);
  if (dtype == ELASTO_BF16)
    return launch_pdl(stem_s2d_kernel<bf16>, dim3(grid_for(total)), dim3(256), 0, s, static_cast<const bf16*>(images),
                      B, H, W, Hs, Ws, d);
  return launch_pdl(stem_s2d_kernel<float>, dim3(grid_for(total)), dim3(256), 0, s, static_cast<const float*>(images),
                    B, H, W, Hs, Ws, d);
}

// ---------------------------------------------------------------- host packing

// fp32 -> IEEE f16 bits, round to nearest even.
uint16_t f16_bits(float f) {
  const __half h = __float2half_rn(f);
  uint16_t u;
  memcpy(&u, &h, 2);
  return u;
}

struct HostTensor {
  const void* p;
  int dtype;
  double operator[](size_t i) const {
    if (dtype == ELASTO_BF16) {
      const uint32_t u = static_cast<uint32_t>(static_cast<const uint16_t*>(p)[i]) << 16;
      float f;
      memcpy(&f, &u, 4);
      return f;
    }
    return static_cast<const float*>(p)[i];
  }
};

// Folded BN of output channel o: scale g / sqrt(var + eps), bias beta - mean * scale.
struct Bn {
  HostTensor g, b, mean, var;
  double scale(int o) const { return g[o] / sqrt(var[o] + kBnEps); }
  double bias(int o) const { return b[o] - mean[o] * scale(o); }
};

elasto_launch_record rec(int kind, int layer, int m, int n, int k, double macs, double bytes) {
  elasto_launch_record r{};
  r.kind = kind;
  r.layer = layer;
  r.m = m;
  r.n = n;
  r.k = k;
  r.macs = macs;
  r.bytes = bytes;
  return r;
}

elasto_launch_record gemm_record(int layer, int M, int N, int K, bool resid) {
  const double mn = double(M) * N;
  return rec(ELASTO_K_GEMM, layer, M, N, K, mn * K, 2.0 * M * K + 2.0 * N * K + mn * 2 * (resid ? 2 : 1));
}

}  // namespace

// ---------------------------------------------------------------- C-ABI hooks

elasto_status cnn_check_inputs(const elasto_model_desc* d, const elasto_weights* w, const elasto_mode_tables* modes,
                               int n_modes) {
  if (d->img_c != 3 || d->img_h < 32 || d->img_w < 32 || d->classes < 1 || d->img_h > 4096 || d->img_w > 1024) {
    set_error("elasto_create: ResNet-50 needs img_c = 3, 32 <= img_h <= 4096, 32 <= img_w <= 1024, classes >= 1");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (w->n_tensors != n_tensors_expected()) {
    set_error("elasto_create: ResNet-50 expects " + std::to_string(n_tensors_expected()) + " weight tensors, got " +
              std::to_string(w->n_tensors));
    return ELASTO_ERR_INVALID_ARG;
  }
  for (int i = 0; i < w->n_tensors; ++i)
    if (!w->tensors[i]) {
      set_error("elasto_create: null weight tensor " + std::to_string(i));
      return ELASTO_ERR_INVALID_ARG;
    }
  const std::vector<BlockShape> sh = block_shapes(1, 1);
  for (int m = 0; m < n_modes; ++m) {
    const elasto_mode_tables& t = modes[m];
    if (!t.conv_kept_a || !t.n_conv_a || !t.conv_kept_b || !t.n_conv_b) {
      set_error("elasto_create: mode " + std::to_string(m) + ": ResNet tables missing");
      return ELASTO_ERR_INVALID_ARG;
    }
    size_t oa = 0, ob = 0;
    for (size_t i = 0; i < sh.size(); ++i) {
      const int na = t.n_conv_a[i], nb = t.n_conv_b[i], width = sh[i].w;
      if (na < 1 || na > width || nb < 1 || nb > width) {
        set_error("elasto_create: mode " + std::to_string(m) + " block " + std::to_string(i) +
                  ": kept counts must lie in [1, width]");
        return ELASTO_ERR_BAD_TABLE;
      }
      for (int s = 0; s < 2; ++s) {
        const int32_t* idx = (s == 0 ? t.conv_kept_a + oa : t.conv_kept_b + ob);
        const int n = s == 0 ? na : nb;
        for (int k = 0; k < n; ++k)
          if (idx[k] < 0 || idx[k] >= width || (k > 0 && idx[k] <= idx[k - 1])) {
            set_error("elasto_create: mode " + std::to_string(m) + " block " + std::to_string(i) +
                      ": kept channels must be strictly increasing and in [0, width)");
            return ELASTO_ERR_BAD_TABLE;
          }
      }
      oa += na;
      ob += nb;
    }
  }
  return ELASTO_OK;
}

CnnModel* cnn_new() { return new CnnModel(); }

elasto_status cnn_create(const elasto_model_desc* d, const elasto_weights* wts, const elasto_mode_tables* tables,
                         int n_modes, CnnModel* m) {
  m->d = *d;
  m->n_modes = n_modes;
  const int Bm = d->max_batch, C = d->classes, dt = d->weight_dtype;
  m->h1 = (d->img_h + 6 - 7) / 2 + 1;
  m->w1 = (d->img_w + 6 - 7) / 2 + 1;
  m->hp = (m->h1 - 1) / 2 + 1;
  m->wp = (m->w1 - 1) / 2 + 1;
  m->shapes = block_shapes(m->hp, m->wp);
  const std::vector<BlockShape>& S = m->shapes;
  const int nblk = static_cast<int>(S.size());

  // canonical tensor order: stem_w, stem BN x4, per block conv1 + bn1 x4,
  // conv2 + bn2 x4, conv3 + bn3 x4 [, down_w + down BN x4], fc_w, fc_b
  int ti = 0;
  auto T = [&](int i) { return HostTensor{wts->tensors[i], dt}; };
  const int t_stem = ti;
  ti += 5;
  std::vector<int> t_blk(nblk);
  for (int i = 0; i < nblk; ++i) {
    t_blk[i] = ti;
    ti += 15 + (S[i].proj ? 5 : 0);
  }
  const int t_fc = ti;

  // ---------------------------------------------------------------- layout
  GuardedArena& ar = m->guards;  // every buffer followed by a guard zone
  const size_t o_stem_w = ar.take(size_t(kStemC) * kStemKs * 2), o_stem_b = ar.take(kStemC * 4);
  std::vector<size_t> o_dw(nblk, 0), o_db(nblk, 0);
  for (int i = 0; i < nblk; ++i)
    if (S[i].proj) {
      o_dw[i] = ar.take(size_t(4) * S[i].w * S[i].cin * 2);
      o_db[i] = ar.take(size_t(4) * S[i].w * 4);
    }
  const size_t o_fcw = ar.take(size_t(C) * 2048 * 4), o_fcb = ar.take(size_t(C) * 4);
  m->shared_bytes = ar.off;
  m->modes.resize(n_modes);
  struct Off {
    size_t w1, w2, w3, b1, b2, b3;
  };
  std::vector<std::vector<Off>> offs(n_modes, std::vector<Off>(nblk));
  {
    for (int mo = 0; mo < n_modes; ++mo) {
      const size_t start = ar.off;
      m->modes[mo].blocks.resize(nblk);
      for (int i = 0; i < nblk; ++i) {
        CnnBlockPack& bp = m->modes[mo].blocks[i];
        bp.a = tables[mo].n_conv_a[i];
        bp.b = tables[mo].n_conv_b[i];
        bp.a_pad = round8(bp.a);
        bp.b_pad = round8(bp.b);
        bp.a_cp = conv_tap_stride(bp.a_pad);
        Off& o = offs[mo][i];
        o.w1 = ar.take(size_t(bp.a_pad) * S[i].cin * 2);
        o.b1 = ar.take(size_t(bp.a_pad) * 4);
        o.w2 = ar.take(size_t(bp.b_pad) * 9 * bp.a_cp * 2);
        o.b2 = ar.take(size_t(bp.b_pad) * 4);
        o.w3 = ar.take(size_t(4) * S[i].w * bp.b_pad * 2);
        o.b3 = ar.take(size_t(4) * S[i].w * 4);
      }
      m->modes[mo].packed_bytes = ar.off - start;
    }
  }
  // workspace (sizes for the widest mode: kept counts never exceed the width)
  const size_t rows_stem = size_t(Bm) * m->h1 * m->w1;
  // the space-to-depth image with its border: (stem output size + 3)^2 x 16
  const size_t s2d = size_t(Bm) * (m->h1 + 3) * (m->w1 + 3) * kS2dC;
  size_t xbuf = std::max(rows_stem * kStemC, size_t(Bm) * m->hp * m->wp * kStemC);
  size_t t1 = 0, t2 = 0, scb = 0;
  for (const BlockShape& b : S) {
    const size_t ri = size_t(Bm) * b.hin * b.win, ro = size_t(Bm) * b.ho * b.wo;
    xbuf = std::max(xbuf, ro * 4 * size_t(b.w));
    t1 = std::max(t1, ri * size_t(round8(b.w)));
    t2 = std::max(t2, ro * size_t(round8(b.w)));
    if (b.proj) scb = std::max(scb, ro * 4 * size_t(b.w));
  }
  const size_t ws_start = ar.off;
  const size_t o_s2d = ar.take(s2d * 2, "space-to-depth image"), o_xa = ar.take(xbuf * 2, "activation A"),
               o_xb = ar.take(xbuf * 2, "activation B");
  const size_t o_t1 = ar.take(t1 * 2, "conv1 output"), o_t2 = ar.take(t2 * 2, "conv2 output"),
               o_sc = ar.take(scb * 2, "projection shortcut");
  const size_t o_pool = ar.take(size_t(Bm) * 2048 * 4, "pooled features");
  const size_t o_img = ar.take(size_t(Bm) * d->img_h * d->img_w * 3 * (dt == ELASTO_BF16 ? 2 : 4), "image staging");
  const size_t o_logit = ar.take(size_t(Bm) * C * 4, "logit staging");
  const size_t o_status = ar.take(64, "status word");
  m->workspace_bytes = ar.off - ws_start;
  m->arena_bytes = ar.off;

  cudaError_t e = cudaMalloc(&m->arena, m->arena_bytes);
  if (e != cudaSuccess) {
    m->arena = nullptr;
    cudaGetLastError();
    set_error("elasto_create: cudaMalloc of " + std::to_string(m->arena_bytes) + " bytes failed");
    return ELASTO_ERR_OOM;
  }
  char* A = m->arena;
  ELASTO_CUDA_TRY(cudaMemset(A, 0, m->arena_bytes));
  {
    const elasto_status gs = m->guards.upload(A);
    if (gs != ELASTO_OK) return gs;
  }
  m->stem_w = reinterpret_cast<F16Buf*>(A + o_stem_w);
  m->stem_b = reinterpret_cast<float*>(A + o_stem_b);
  m->down_w.assign(nblk, nullptr);
  m->down_b.assign(nblk, nullptr);
  for (int i = 0; i < nblk; ++i)
    if (S[i].proj) {
      m->down_w[i] = reinterpret_cast<F16Buf*>(A + o_dw[i]);
      m->down_b[i] = reinterpret_cast<float*>(A + o_db[i]);
    }
  m->fc_w = reinterpret_cast<float*>(A + o_fcw);
  m->fc_b = reinterpret_cast<float*>(A + o_fcb);
  m->s2d = reinterpret_cast<F16Buf*>(A + o_s2d);
  m->xa = reinterpret_cast<F16Buf*>(A + o_xa);
  m->xb = reinterpret_cast<F16Buf*>(A + o_xb);
  m->t1 = reinterpret_cast<F16Buf*>(A + o_t1);
  m->t2 = reinterpret_cast<F16Buf*>(A + o_t2);
  m->sc = reinterpret_cast<F16Buf*>(A + o_sc);
  m->pooled = reinterpret_cast<float*>(A + o_pool);
  m->img_stage = A + o_img;
  m->logit_stage = reinterpret_cast<float*>(A + o_logit);
  m->status = reinterpret_cast<int*>(A + o_status);
  for (int mo = 0; mo < n_modes; ++mo)
    for (int i = 0; i < nblk; ++i) {
      CnnBlockPack& bp = m->modes[mo].blocks[i];
      const Off& o = offs[mo][i];
      bp.w1 = reinterpret_cast<F16Buf*>(A + o.w1);
      bp.w2 = reinterpret_cast<F16Buf*>(A + o.w2);
      bp.w3 = reinterpret_cast<F16Buf*>(A + o.w3);
      bp.b1 = reinterpret_cast<float*>(A + o.b1);
      bp.b2 = reinterpret_cast<float*>(A + o.b2);
      bp.b3 = reinterpret_cast<float*>(A + o.b3);
    }

  // ---------------------------------------------------------------- pack (host, double)
  std::vector<uint16_t> hw;
  std::vector<float> hb;
  auto up16 = [&](void* dst) { return cudaMemcpy(dst, hw.data(), hw.size() * 2, cudaMemcpyHostToDevice); };
  auto up32 = [&](void* dst) { return cudaMemcpy(dst, hb.data(), hb.size() * 4, cudaMemcpyHostToDevice); };
  {  // stem: [64, 4, 4, 16] over the space-to-depth image from [64, 3, 7, 7]: tap (ty, tx)
     // reads S rows y - 2 + ty, i.e. image rows 2y - 4 + 2 ty + dy = 2y - 3 + ky with
     // ky = 2 ty + dy - 1 (likewise kx); taps outside 0..6 stay zero
    const HostTensor W = T(t_stem);
    const Bn bn{T(t_stem + 1), T(t_stem + 2), T(t_stem + 3), T(t_stem + 4)};
    hw.assign(size_t(kStemC) * kStemKs, 0);
    hb.assign(kStemC, 0.0f);
    for (int o = 0; o < kStemC; ++o) {
      const double s = bn.scale(o);
      for (int ty = 0; ty < 4; ++ty)
        for (int tx = 0; tx < 4; ++tx)
          for (int dy = 0; dy < 2; ++dy)
            for (int dx = 0; dx < 2; ++dx) {
              const int ky = 2 * ty + dy - 1, kx = 2 * tx + dx - 1;
              if (ky < 0 || ky > 6 || kx < 0 || kx > 6) continue;
              for (int c = 0; c < 3; ++c)
                hw[size_t(o) * kStemKs + (ty * 4 + tx) * kS2dC + (dy * 2 + dx) * 3 + c] =
                    f16_bits(static_cast<float>(W[((size_t(o) * 3 + c) * 7 + ky) * 7 + kx] * s));
            }
      hb[o] = static_cast<float>(bn.bias(o));
    }
    ELASTO_CUDA_TRY(up16(m->stem_w));
    ELASTO_CUDA_TRY(up32(m->stem_b));
  }
  for (int i = 0; i < nblk; ++i) {
    if (!S[i].proj) continue;
    const int t0 = t_blk[i] + 15, co = 4 * S[i].w, ci = S[i].cin;
    const HostTensor W = T(t0);
    const Bn bn{T(t0 + 1), T(t0 + 2), T(t0 + 3), T(t0 + 4)};
    hw.assign(size_t(co) * ci, 0);
    hb.assign(co, 0.0f);
    for (int o = 0; o < co; ++o) {
      const double s = bn.scale(o);
      for (int c = 0; c < ci; ++c) hw[size_t(o) * ci + c] = f16_bits(static_cast<float>(W[size_t(o) * ci + c] * s));
      hb[o] = static_cast<float>(bn.bias(o));
    }
    ELASTO_CUDA_TRY(up16(m->down_w[i]));
    ELASTO_CUDA_TRY(up32(m->down_b[i]));
  }
  {  // classifier stays fp32
    const HostTensor W = T(t_fc), b = T(t_fc + 1);
    hb.resize(size_t(C) * 2048);
    for (size_t k = 0; k < hb.size(); ++k) hb[k] = static_cast<float>(W[k]);
    ELASTO_CUDA_TRY(up32(m->fc_w));
    hb.resize(C);
    for (int k = 0; k < C; ++k) hb[k] = static_cast<float>(b[k]);
    ELASTO_CUDA_TRY(up32(m->fc_b));
  }
  for (int mo = 0; mo < n_modes; ++mo) {
    size_t oa = 0, ob = 0;
    for (int i = 0; i < nblk; ++i) {
      CnnBlockPack& bp = m->modes[mo].blocks[i];
      const int t0 = t_blk[i], w = S[i].w, ci = S[i].cin;
      const int32_t* Sa = tables[mo].conv_kept_a + oa;
      const int32_t* Sb = tables[mo].conv_kept_b + ob;
      oa += bp.a;
      ob += bp.b;
      const HostTensor W1 = T(t0), W2 = T(t0 + 5), W3 = T(t0 + 10);
      const Bn bn1{T(t0 + 1), T(t0 + 2), T(t0 + 3), T(t0 + 4)};
      const Bn bn2{T(t0 + 6), T(t0 + 7), T(t0 + 8), T(t0 + 9)};
      const Bn bn3{T(t0 + 11), T(t0 + 12), T(t0 + 13), T(t0 + 14)};
      // conv1: rows S_a of [w, cin]
      hw.assign(size_t(bp.a_pad) * ci, 0);
      hb.assign(bp.a_pad, 0.0f);
      for (int r = 0; r < bp.a; ++r) {
        const int o = Sa[r];
        const double s = bn1.scale(o);
        for (int c = 0; c < ci; ++c) hw[size_t(r) * ci + c] = f16_bits(static_cast<float>(W1[size_t(o) * ci + c] * s));
        hb[r] = static_cast<float>(bn1.bias(o));
      }
      ELASTO_CUDA_TRY(up16(bp.w1));
      ELASTO_CUDA_TRY(up32(bp.b1));
      // conv2: rows S_b, input channels S_a, [b_pad, (ky, kx, c < a_cp)]
      const size_t k2 = size_t(9) * bp.a_cp;
      hw.assign(size_t(bp.b_pad) * k2, 0);
      hb.assign(bp.b_pad, 0.0f);
      for (int r = 0; r < bp.b; ++r) {
        const int o = Sb[r];
        const double s = bn2.scale(o);
        for (int ky = 0; ky < 3; ++ky)
          for (int kx = 0; kx < 3; ++kx)
            for (int c = 0; c < bp.a; ++c)
              hw[size_t(r) * k2 + size_t(ky * 3 + kx) * bp.a_cp + c] =
                  f16_bits(static_cast<float>(W2[((size_t(o) * w + Sa[c]) * 3 + ky) * 3 + kx] * s));
        hb[r] = static_cast<float>(bn2.bias(o));
      }
      ELASTO_CUDA_TRY(up16(bp.w2));
      ELASTO_CUDA_TRY(up32(bp.b2));
      // conv3: columns S_b of [4w, w]
      hw.assign(size_t(4) * w * bp.b_pad, 0);
      hb.assign(4 * w, 0.0f);
      for (int o = 0; o < 4 * w; ++o) {
        const double s = bn3.scale(o);
        for (int c = 0; c < bp.b; ++c)
          hw[size_t(o) * bp.b_pad + c] = f16_bits(static_cast<float>(W3[size_t(o) * w + Sb[c]] * s));
        hb[o] = static_cast<float>(bn3.bias(o));
      }
      ELASTO_CUDA_TRY(up16(bp.w3));
      ELASTO_CUDA_TRY(up32(bp.b3));
    }
  }

  // ---------------------------------------------------------------- plans
  // the stem: 4x4 stride-1 convolution over the bordered space-to-depth image
  // ((h1 + 3) x (w1 + 3) x 16), output h1 x w1 (the 7x7/2 convolution's)
  elasto_status st = gemm_plan_conv_rows(&m->stem, m->s2d, Bm, m->h1 + 3, m->w1 + 3, kS2dC, 4, 4, m->stem_w, kStemC,
                                         m->stem_b, m->xb, kStemC, EPI_BIAS_RELU_F16, m->status);
  if (st != ELASTO_OK) return st;
  m->down.assign(nblk, GemmPlan{});
  const int64_t stem_macs = int64_t(m->h1) * m->w1 * kStemC * kStemK + int64_t(2048) * C;
  for (int i = 0; i < nblk; ++i) {
    const BlockShape& b = S[i];
    F16Buf* xin = (i % 2 == 0) ? m->xa : m->xb;
    const int mo_cap = Bm * b.ho * b.wo;
    if (b.proj) {
      if (b.stride == 1)
        st = gemm_plan(&m->down[i], xin, mo_cap, m->down_w[i], 4 * b.w, b.cin, m->down_b[i], m->sc, 4 * b.w,
                       EPI_BIAS_F16, m->status);
      else
        st = gemm_plan_conv(&m->down[i], xin, Bm, b.hin, b.win, b.cin, 1, b.stride, 0, m->down_w[i], 4 * b.w,
                            m->down_b[i], m->sc, 4 * b.w, EPI_BIAS_F16, m->status);
      if (st != ELASTO_OK) return st;
    }
  }
  for (int mo = 0; mo < n_modes; ++mo) {
    CnnMode& cm = m->modes[mo];
    cm.macs = stem_macs;
    cm.launches = 3 + 2;  // stem gather, stem GEMM, max pool; average pool, classifier
    for (int i = 0; i < nblk; ++i) {
      const BlockShape& b = S[i];
      CnnBlockPack& bp = cm.blocks[i];
      F16Buf* xin = (i % 2 == 0) ? m->xa : m->xb;
      F16Buf* xout = (i % 2 == 0) ? m->xb : m->xa;
      const int mi_cap = Bm * b.hin * b.win, mo_cap = Bm * b.ho * b.wo;
      st = gemm_plan(&bp.conv1, xin, mi_cap, bp.w1, bp.a_pad, b.cin, bp.b1, m->t1, bp.a_pad, EPI_BIAS_RELU_F16,
                        m->status);
      if (st != ELASTO_OK) return st;
      // conv1 reads the previous block's output, written first row to last:
      // reading it last row first finds the most recent rows still in L2
      bp.conv1.args.m_reverse = 1;
      st = gemm_plan_conv(&bp.conv2, m->t1, Bm, b.hin, b.win, bp.a_pad, 3, b.stride, 1, bp.w2, bp.b_pad, bp.b2, m->t2,
                          bp.b_pad, EPI_BIAS_RELU_F16, m->status);
      if (st != ELASTO_OK) return st;
      st = gemm_plan(&bp.conv3, m->t2, mo_cap, bp.w3, 4 * b.w, bp.b_pad, bp.b3, xout, 4 * b.w,
                        EPI_BIAS_RESID_RELU_F16, m->status);
      if (st != ELASTO_OK) return st;
      st = gemm_set_residual_source(&bp.conv3, b.proj ? m->sc : xin, mo_cap);
      if (st != ELASTO_OK) return st;
      cm.macs += int64_t(b.hin) * b.win * bp.a * b.cin + int64_t(b.ho) * b.wo * bp.b * 9 * bp.a +
                 int64_t(b.ho) * b.wo * 4 * b.w * bp.b + (b.proj ? int64_t(b.ho) * b.wo * 4 * b.w * b.cin : 0);
      cm.launches += 3 + (b.proj ? 1 : 0);
    }
  }
  ELASTO_CUDA_TRY(cudaDeviceSynchronize());
  return ELASTO_OK;
}

#define CNN_LAUNCH(r, expr)                 \
  do {                                      \
    ELASTO_CUDA_TRY(m->prof.before(s));     \
    ELASTO_CUDA_TRY(expr);                  \
    ELASTO_CUDA_TRY(m->prof.after(s, (r))); \
  } while (0)

elasto_status cnn_forward(CnnModel* m, int mode, cudaStream_t s, const void* images, int batch, float* logits) {
  const elasto_model_desc& d = m->d;
  const CnnMode& cm = m->modes[mode];
  const int B = batch, C = d.classes;
  const double img_elt = d.weight_dtype == ELASTO_BF16 ? 2 : 4;
  m->prof.begin();
  const int ms = B * m->h1 * m->w1;
  CNN_LAUNCH(rec(ELASTO_K_IM2COL, -1, ms, kS2dC, 0, 0,
                 double(B) * d.img_h * d.img_w * 3 * img_elt + double(B) * (m->h1 + 3) * (m->w1 + 3) * kS2dC * 2),
             stem_s2d_launch(images, d.weight_dtype, B, d.img_h, d.img_w, m->h1, m->w1,
                             reinterpret_cast<__half*>(m->s2d), s));
  CNN_LAUNCH(gemm_record(-1, ms, kStemC, kStemK, false), gemm_launch(m->stem, B, s));
  {
    const size_t total = size_t(B) * m->hp * m->wp * (kStemC / 8);
    CNN_LAUNCH(rec(ELASTO_K_POOL, -1, B * m->hp * m->wp, kStemC, 0, 0,
                   double(ms) * kStemC * 2 + double(B) * m->hp * m->wp * kStemC * 2),
               launch_pdl(maxpool_kernel, dim3(grid_for(total)), dim3(256), 0, s,
                          reinterpret_cast<const uint4*>(m->xb), m->h1, m->w1, kStemC / 8, m->hp, m->wp, total,
                          reinterpret_cast<uint4*>(m->xa)));
  }
  const int nblk = static_cast<int>(m->shapes.size());
  for (int i = 0; i < nblk; ++i) {
    const BlockShape& b = m->shapes[i];
    const CnnBlockPack& bp = cm.blocks[i];
    const F16Buf* xin = (i % 2 == 0) ? m->xa : m->xb;
    const int mi = B * b.hin * b.win, mo = B * b.ho * b.wo;
    CNN_LAUNCH(gemm_record(i, mi, bp.a, b.cin, false), gemm_launch(bp.conv1, mi, s));
    // implicit GEMMs: A is read from the input activation (gemm_record's
    // A-bytes term counts the im2col view; the input itself is mi x channels)
    CNN_LAUNCH(gemm_record(i, mo, bp.b, 9 * bp.a, false), gemm_launch(bp.conv2, B, s));
    if (b.proj)
      CNN_LAUNCH(gemm_record(i, mo, 4 * b.w, b.cin, false), gemm_launch(m->down[i], b.stride == 1 ? mo : B, s));
    CNN_LAUNCH(gemm_record(i, mo, 4 * b.w, bp.b, true), gemm_launch(bp.conv3, mo, s));
  }
  const BlockShape& last = m->shapes.back();
  const F16Buf* xfin = (nblk % 2 == 0) ? m->xa : m->xb;
  const int hw = last.ho * last.wo, cfin = 4 * last.w;
  {
    const size_t total = size_t(B) * (cfin / 8);
    CNN_LAUNCH(rec(ELASTO_K_POOL, nblk, B, cfin, 0, 0, double(B) * hw * cfin * 2 + double(B) * cfin * 4),
               launch_pdl(avgpool_kernel, dim3(grid_for(4 * total)), dim3(256), 0, s, reinterpret_cast<const uint4*>(xfin),
                          hw, cfin / 8, total, m->pooled));
  }
  {
    static_assert(4 * 512 <= kCnnMaxFeatures, "the classifier's pooled rows exceed its shared-memory limit");
    dim3 grid((B + FC_IMGS - 1) / FC_IMGS, (C + FC_CLASSES - 1) / FC_CLASSES);
    CNN_LAUNCH(rec(ELASTO_K_HEAD, -1, B, C, cfin, double(B) * C * cfin,
                   double(B) * cfin * 4 + double(C) * cfin * 4 + double(B) * C * 4),
               launch_pdl(fc_kernel, grid, dim3(256), FC_IMGS * cfin * sizeof(float), s,
                          static_cast<const float*>(m->pooled), B, cfin,
                          static_cast<const float*>(m->fc_w), static_cast<const float*>(m->fc_b), C, logits));
  }
  return ELASTO_OK;
}

#undef CNN_LAUNCH

int cnn_n_modes(const CnnModel* m) { return m->n_modes; }
void* cnn_image_stage(CnnModel* m) { return m->img_stage; }
float* cnn_logit_stage(CnnModel* m) { return m->logit_stage; }
int* cnn_status_word(CnnModel* m) { return m->status; }
Profiler* cnn_profiler(CnnModel* m) { return &m->prof; }

void cnn_destroy(CnnModel* m) {
  if (m->arena) {
    cudaDeviceSynchronize();
    cudaFree(m->arena);
  }
  m->guards.release();
  m->prof.release();
  delete m;
}

elasto_status cnn_query(CnnModel* m, int what, int mode, int64_t* value) {
  const bool needs_mode = what == ELASTO_Q_PACKED_BYTES || what == ELASTO_Q_MODE_MACS || what == ELASTO_Q_LAUNCHES;
  if (needs_mode && (mode < 0 || mode >= m->n_modes)) {
    set_error("elasto_query: bad mode");
    return ELASTO_ERR_BAD_MODE;
  }
  switch (what) {
    case ELASTO_Q_N_MODES: *value = m->n_modes; break;
    case ELASTO_Q_PACKED_BYTES: *value = int64_t(m->modes[mode].packed_bytes); break;
    case ELASTO_Q_SHARED_BYTES: *value = int64_t(m->shared_bytes); break;
    case ELASTO_Q_WORKSPACE_BYTES: *value = int64_t(m->workspace_bytes); break;
    case ELASTO_Q_ARENA_BYTES: *value = int64_t(m->arena_bytes); break;
    case ELASTO_Q_MODE_MACS: *value = m->modes[mode].macs; break;
    case ELASTO_Q_LAUNCHES: *value = m->modes[mode].launches; break;
    case ELASTO_Q_PACKED_TOTAL: {
      int64_t t = 0;
      for (const CnnMode& cm : m->modes) t += int64_t(cm.packed_bytes);
      *value = t;
      break;
    }
    case ELASTO_Q_PREFIX_SHARED: *value = 0; break;
    case ELASTO_Q_GUARD_ZONES: *value = int64_t(m->guards.zones.size()); break;
    case ELASTO_Q_ONE_LAUNCH: *value = 0; break;  // the one-launch forward is ViT-only
    default: set_error("elasto_query: unknown query"); return ELASTO_ERR_INVALID_ARG;
  }
  return ELASTO_OK;
}

elasto_status cnn_export_packed(CnnModel* m, int mode, int block, int which, void* host_dst, size_t bytes) {
  if (mode < 0 || mode >= m->n_modes) {
    set_error("elasto_debug_export_packed: bad mode");
    return ELASTO_ERR_BAD_MODE;
  }
  if (block < 0 || block >= static_cast<int>(m->shapes.size()) || which < 0 || which > 5) {
    set_error("elasto_debug_export_packed: bad block or buffer index");
    return ELASTO_ERR_INVALID_ARG;
  }
  const BlockShape& b = m->shapes[block];
  const CnnBlockPack& bp = m->modes[mode].blocks[block];
  // unpadded sizes: conv1 [a, cin], bias1 [a], conv2 [b, 3, 3, a], bias2 [b], conv3 [4w, b], bias3 [4w]
  const size_t want[6] = {size_t(bp.a) * b.cin * 2, size_t(bp.a) * 4, size_t(bp.b) * 9 * bp.a * 2,
                          size_t(bp.b) * 4, size_t(4) * b.w * bp.b * 2, size_t(4) * b.w * 4};
  if (!host_dst || bytes != want[which]) {
    set_error("elasto_debug_export_packed: byte count must be " + std::to_string(want[which]));
    return ELASTO_ERR_INVALID_ARG;
  }
  switch (which) {
    case 0: ELASTO_CUDA_TRY(cudaMemcpy(host_dst, bp.w1, bytes, cudaMemcpyDeviceToHost)); break;
    case 1: ELASTO_CUDA_TRY(cudaMemcpy(host_dst, bp.b1, bytes, cudaMemcpyDeviceToHost)); break;
    case 3: ELASTO_CUDA_TRY(cudaMemcpy(host_dst, bp.b2, bytes, cudaMemcpyDeviceToHost)); break;
    case 5: ELASTO_CUDA_TRY(cudaMemcpy(host_dst, bp.b3, bytes, cudaMemcpyDeviceToHost)); break;
    case 2: {
      std::vector<uint16_t> pad(size_t(bp.b) * 9 * bp.a_cp);
      ELASTO_CUDA_TRY(cudaMemcpy(pad.data(), bp.w2, pad.size() * 2, cudaMemcpyDeviceToHost));
      uint16_t* o = static_cast<uint16_t*>(host_dst);
      for (int r = 0; r < bp.b; ++r)
        for (int t = 0; t < 9; ++t)
          memcpy(o + (size_t(r) * 9 + t) * bp.a, pad.data() + (size_t(r) * 9 + t) * bp.a_cp, size_t(bp.a) * 2);
      break;
    }
    case 4: {
      std::vector<uint16_t> pad(size_t(4) * b.w * bp.b_pad);
      ELASTO_CUDA_TRY(cudaMemcpy(pad.data(), bp.w3, pad.size() * 2, cudaMemcpyDeviceToHost));
      uint16_t* o = static_cast<uint16_t*>(host_dst);
      for (int r = 0; r < 4 * b.w; ++r) memcpy(o + size_t(r) * bp.b, pad.data() + size_t(r) * bp.b_pad, size_t(bp.b) * 2);
      break;
    }
  }
  return ELASTO_OK;
}

GuardedArena* cnn_guards(CnnModel* m, char** base) {
  *base = m->arena;
  return &m->guards;
}

}  // namespace elasto
