// elasto_forward_noalloc: the ViT forward pass with its activation scratch in
// a fixed, file-scope device array instead of the handle's workspace.
//
// Who needs it: callers that may not allocate device memory at the point
// where they run inference -- for example a process whose memory manager
// hands the whole device to its own pool at start-up and forbids later
// driver allocations, or a latency-critical loop that cannot afford the
// implicit device synchronisation a cudaMalloc/cudaFree may cause. Such a
// caller can create its handle with a small max_batch (a small workspace)
// and still run batches up to the static limit here, and this call itself
// performs no allocation of any kind (no cudaMalloc, no cudaFree, no
// allocating library routine).
//
// The array is g_noalloc_scratch, 64 MiB, resident on every GPU that loads
// the library until the process exits. In host code its name is only a
// host-side stand-in: the device address is obtained once per device with
// cudaGetSymbolAddress (with that device current) and the kernels receive
// that address. All calls share the one array and it keeps the last call's
// contents; every scratch byte a call reads it has written first in the same
// call, so nothing needs clearing, but two calls that overlap on the GPU (for
// instance on two streams) race on the array.
#include <mutex>

#include "common.h"
#include "elasto_internal.h"
#include "handle.h"

namespace elasto {

namespace {

constexpr size_t kScratchBytes = size_t(64) << 20;  // 64 MiB
constexpr size_t kAlignB = 1024;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

std::mutex g_sym_mu;
void* g_sym_addr[64] = {};

// Device address of g_noalloc_scratch on the current device (set-up on the
// first call per device).
elasto_status scratch_address(void** out) {
  int dev = 0;
  ELASTO_CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) {
    set_error("elasto_forward_noalloc: device index out of range");
    return ELASTO_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_sym_mu);
  if (!g_sym_addr[dev]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return cuda_fail(e != cudaSuccess ? e : cudaErrorInvalidSymbol,
                                                 "cudaGetSymbolAddress(g_noalloc_scratch)");
    g_sym_addr[dev] = p;
  }
  *out = g_sym_addr[dev];
  return ELASTO_OK;
}

size_t align_up(size_t v) { return (v + kAlignB - 1) / kAlignB * kAlignB; }

struct ScratchLayout {
  size_t X, Y, QKV, O, H, P, total;
};

ScratchLayout layout_for(const elasto_s* h, int batch, int wmax, int fmax) {
  const size_t rows = size_t(batch) * h->n, D = h->d.dim;
  ScratchLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t r = off;
    off = align_up(off + bytes);
    return r;
  };
  L.X = take(rows * D * 4);
  L.Y = take(rows * D * 2);
  L.QKV = take(rows * 3 * size_t(wmax) * 2);
  L.O = take(rows * size_t(wmax) * 2);
  L.H = take(rows * size_t(fmax) * 2);
  L.P = take(size_t(batch) * h->np * h->kpe * 2);
  L.total = off;
  return L;
}

}  // namespace

}  // namespace elasto

using namespace elasto;

extern "C" elasto_status elasto_forward_noalloc(elasto_t h, void* stream, const void* images, int batch,
                                                float* logits) {
  if (!h || !images || !logits) {
    set_error("elasto_forward_noalloc: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (h->cnn) {
    set_error("elasto_forward_noalloc: only ViT handles are supported");
    return ELASTO_ERR_UNSUPPORTED;
  }
  const elasto_model_desc& d = h->d;
  const VitMode& vm = h->modes[h->cur.load(std::memory_order_acquire)];
  int wmax = 64, fmax = 8;
  for (const VitLayerPack& lp : vm.layers) {
    wmax = lp.w > wmax ? lp.w : wmax;
    fmax = lp.f_pad > fmax ? lp.f_pad : fmax;
  }
  if (batch < 1 || layout_for(h, batch, wmax, fmax).total > kScratchBytes) {
    int cap = 0;
    while (layout_for(h, cap + 1, wmax, fmax).total <= kScratchBytes) ++cap;
    set_error("elasto_forward_noalloc: batch " + std::to_string(batch) +
              " is outside [1, " + std::to_string(cap) + "]: the 64 MiB static scratch holds at most " +
              std::to_string(cap) + " images of this model in this mode");
    return ELASTO_ERR_INVALID_ARG;
  }
  void* base = nullptr;
  elasto_status st = scratch_address(&base);
  if (st != ELASTO_OK) return st;
  char* S = static_cast<char*>(base);
  const ScratchLayout L = layout_for(h, batch, wmax, fmax);
  float* X = reinterpret_cast<float*>(S + L.X);
  bf16* Y = reinterpret_cast<bf16*>(S + L.Y);
  bf16* QKV = reinterpret_cast<bf16*>(S + L.QKV);
  bf16* O = reinterpret_cast<bf16*>(S + L.O);
  bf16* H = reinterpret_cast<bf16*>(S + L.H);
  bf16* P = reinterpret_cast<bf16*>(S + L.P);

  const VitEmbed& em = vm.emb;
  const int n = h->n, D = em.d_pad, M = batch * n, Mp = batch * h->np;  // D: residual-stream width of this mode
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  GemmPlan gp;
  st = gemm_plan(&gp, P, Mp, em.patch_w, D, h->kpe, em.patch_b, X, D, EPI_PATCH_POS_F32, h->status,
                 em.patch_w_lo);
  if (st != ELASTO_OK) return st;
  gp.args.patches = h->np;
  gp.args.tokens = n;
  gp.args.pos = em.pos;
  ELASTO_CUDA_TRY(
      patchify_launch(images, d.weight_dtype, batch, d.img_h, d.img_w, d.img_c, d.patch, P, X, em.cls, em.pos, D, s));
  ELASTO_CUDA_TRY(gemm_launch(gp, Mp, s));
  for (int l = 0; l < d.layers; ++l) {
    const VitLayerPack& lp = vm.layers[l];
    ELASTO_CUDA_TRY(layernorm_launch(X, em.ln1_w[l], em.ln1_b[l], Y, M, D, em.d, s));
    if (lp.w > 0) {
      GemmPlan qkv;
      AttnPlan at;
      if ((st = gemm_plan(&qkv, Y, M, lp.qkv_w, 3 * lp.w, D, lp.qkv_b, QKV, 3 * lp.w, EPI_BIAS_BF16,
                          h->status, lp.qkv_w_lo)) != ELASTO_OK)
        return st;
      if ((st = attn_plan(&at, QKV, O, batch, n, lp.w / 64, h->status, h->prefix_shared)) != ELASTO_OK) return st;
      ELASTO_CUDA_TRY(gemm_launch(qkv, M, s));
      ELASTO_CUDA_TRY(attn_launch(at, batch, s));
    }
    GemmPlan proj, fc2;
    if ((st = gemm_plan(&proj, O, M, lp.proj_w, D, lp.w, em.proj_b[l], X, D, EPI_BIAS_RESID_F32, h->status,
                        lp.proj_w_lo, 0, lp.ld_proj)) != ELASTO_OK)
      return st;
    ELASTO_CUDA_TRY(gemm_launch(proj, M, s));
    ELASTO_CUDA_TRY(layernorm_launch(X, em.ln2_w[l], em.ln2_b[l], Y, M, D, em.d, s));
    if (lp.f > 0) {
      GemmPlan fc1;
      if ((st = gemm_plan(&fc1, Y, M, lp.fc1_w, lp.f_pad, D, lp.fc1_b, H, lp.f_pad, EPI_BIAS_GELU_BF16,
                          h->status, lp.fc1_w_lo)) != ELASTO_OK)
        return st;
      ELASTO_CUDA_TRY(gemm_launch(fc1, M, s));
    }
    if ((st = gemm_plan(&fc2, H, M, lp.fc2_w, D, lp.f_pad, em.fc2_b[l], X, D, EPI_BIAS_RESID_F32, h->status,
                        lp.fc2_w_lo, 0, lp.ld_fc2)) != ELASTO_OK)
      return st;
    ELASTO_CUDA_TRY(gemm_launch(fc2, M, s));
  }
  ELASTO_CUDA_TRY(
      head_launch(X, batch, n, D, em.d, em.norm_w, em.norm_b, em.head_w, h->head_b, d.classes, logits, s));
  return ELASTO_OK;
}
