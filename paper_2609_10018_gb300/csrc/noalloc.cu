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
// performs no device allocation of any kind (no cudaMalloc, no cudaFree, no
// allocating library routine).
//
// The array is g_noalloc_scratch, 64 MiB, resident on every GPU that loads
// the library until the process exits. In host code its name is only a
// host-side stand-in: the device address is looked up with
// cudaGetSymbolAddress (with the handle's device current) on the first call
// in each CUDA context of a device, and the kernels receive that address.
// All calls share the one array and it keeps the last call's contents; every
// scratch byte a call reads it has written first in the same call, so
// nothing needs clearing, but two calls that overlap on the GPU (for
// instance on two streams) race on the array.
//
// The launch plans of a (mode, batch) pair are built on its first call and
// kept with the handle (host memory), so later calls only launch. The patch
// embedding, LayerNorms, GEMMs, attention and head are the same kernels and
// plans as elasto_forward's, pointed at the static scratch.
#include <mutex>

#include "common.h"
#include "elasto_internal.h"
#include "handle.h"

namespace elasto {

namespace {

constexpr size_t kScratchBytes = size_t(64) << 20;  // 64 MiB
constexpr size_t kAlignB = 1024;
constexpr int kMaxDevices = 64;
constexpr size_t kMaxCachedPlans = 32;  // (mode, batch) pairs kept per handle

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

using CtxGetCurrentFn = int (*)(void**);  // CUresult cuCtxGetCurrent(CUcontext*)

// The current CUDA context (null if the driver entry point is unavailable).
void* current_context() {
  static CtxGetCurrentFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<CtxGetCurrentFn>(p);
    return static_cast<CtxGetCurrentFn>(nullptr);
  }();
  void* ctx = nullptr;
  if (fn) fn(&ctx);
  return ctx;
}

std::mutex g_sym_mu;
struct SymEntry {
  void* ctx = nullptr;
  void* addr = nullptr;
};
SymEntry g_sym[kMaxDevices];

// Device address of g_noalloc_scratch on device `dev` (current), looked up
// again whenever the device's current context is not the one it was taken
// in (after a cudaDeviceReset the old address belongs to a destroyed
// context).
elasto_status scratch_address(int dev, void** out) {
  if (dev < 0 || dev >= kMaxDevices) {
    set_error("elasto_forward_noalloc: device index out of range");
    return ELASTO_ERR_UNSUPPORTED;
  }
  void* ctx = current_context();
  std::lock_guard<std::mutex> lock(g_sym_mu);
  SymEntry& e = g_sym[dev];
  if (!e.addr || e.ctx != ctx || !ctx) {
    void* p = nullptr;
    cudaError_t err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (err != cudaSuccess || !p)
      return cuda_fail(err != cudaSuccess ? err : cudaErrorInvalidSymbol, "cudaGetSymbolAddress(g_noalloc_scratch)");
    e.addr = p;
    e.ctx = ctx;
  }
  *out = e.addr;
  return ELASTO_OK;
}

size_t align_up(size_t v) { return (v + kAlignB - 1) / kAlignB * kAlignB; }

struct ScratchLayout {
  size_t X, Y, QKV, O, H, P, total;
};

// Scratch of one call: residual X fp32, LayerNorm output Y, QKV, attention
// output O, MLP hidden H and the token-ordered patch rows P, all for
// batch * n rows at the mode's widths.
ScratchLayout layout_for(const elasto_s* h, int batch, int D, int wmax, int fmax) {
  const size_t rows = size_t(batch) * h->n;
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
  L.P = take(rows * h->kpe * 2);
  L.total = off;
  return L;
}

}  // namespace

struct NoallocLayerPlans {
  GemmPlan qkv, proj, fc1, fc2;
  AttnPlan attn;
};

struct NoallocPlans {
  int mode = -1, batch = 0;
  void* base = nullptr;  // scratch address the plans point into
  GemmPlan patch;
  std::vector<NoallocLayerPlans> layers;
};

struct NoallocCache {
  std::vector<NoallocPlans> entries;  // at most kMaxCachedPlans, oldest first
};

void noalloc_cache_free(NoallocCache* c) { delete c; }

namespace {

// Plans of every launch of one forward of `mode` at `batch`, over the
// scratch at `base`: the same planners and epilogues as the handle's own
// plans (patch rows + patch GEMM adding the periodic per-token addend,
// per-layer QKV / attention / out-projection / FC1 / FC2).
elasto_status build_plans(elasto_s* h, int mode, int batch, char* base, const ScratchLayout& L, NoallocPlans* P) {
  const VitMode& vm = h->modes[mode];
  const VitEmbed& em = vm.emb;
  const int n = h->n, D = em.d_pad, M = batch * n;
  float* X = reinterpret_cast<float*>(base + L.X);
  bf16* Y = reinterpret_cast<bf16*>(base + L.Y);
  bf16* QKV = reinterpret_cast<bf16*>(base + L.QKV);
  bf16* O = reinterpret_cast<bf16*>(base + L.O);
  bf16* H = reinterpret_cast<bf16*>(base + L.H);
  bf16* Prow = reinterpret_cast<bf16*>(base + L.P);
  P->mode = mode;
  P->batch = batch;
  P->base = base;
  elasto_status st = gemm_plan(&P->patch, Prow, M, em.patch_w, D, h->kpe, nullptr, X, D, EPI_BIAS_RESID_F32,
                               h->status, em.patch_w_lo, M);
  if (st != ELASTO_OK) return st;
  st = gemm_set_residual_source(&P->patch, em.pruned ? em.addend : h->tok_addend, h->addend_rows, n);
  if (st != ELASTO_OK) return st;
  P->layers.assign(vm.layers.size(), NoallocLayerPlans{});
  for (size_t l = 0; l < vm.layers.size(); ++l) {
    const VitLayerPack& lp = vm.layers[l];
    NoallocLayerPlans& q = P->layers[l];
    if (lp.w > 0) {
      if ((st = gemm_plan(&q.qkv, Y, M, lp.qkv_w, 3 * lp.w, D, lp.qkv_b, QKV, 3 * lp.w, EPI_BIAS_BF16, h->status,
                          lp.qkv_w_lo, M)) != ELASTO_OK)
        return st;
      if ((st = attn_plan(&q.attn, QKV, O, batch, n, lp.w / 64, h->status, h->prefix_shared)) != ELASTO_OK) return st;
    }
    if ((st = gemm_plan(&q.proj, O, M, lp.proj_w, D, lp.w, em.proj_b[l], X, D, EPI_BIAS_RESID_F32, h->status,
                        lp.proj_w_lo, M, lp.ld_proj)) != ELASTO_OK)
      return st;
    if (lp.f > 0 && (st = gemm_plan(&q.fc1, Y, M, lp.fc1_w, lp.f_pad, D, lp.fc1_b, H, lp.f_pad, EPI_BIAS_GELU_BF16,
                                    h->status, lp.fc1_w_lo, M)) != ELASTO_OK)
      return st;
    if ((st = gemm_plan(&q.fc2, H, M, lp.fc2_w, D, lp.f_pad, em.fc2_b[l], X, D, EPI_BIAS_RESID_F32, h->status,
                        lp.fc2_w_lo, M, lp.ld_fc2)) != ELASTO_OK)
      return st;
  }
  return ELASTO_OK;
}

// The cached plans of (mode, batch) over `base`, built on first use.
elasto_status plans_for(elasto_s* h, int mode, int batch, char* base, const ScratchLayout& L,
                        const NoallocPlans** out) {
  if (!h->noalloc) h->noalloc = new NoallocCache();
  std::vector<NoallocPlans>& es = h->noalloc->entries;
  for (const NoallocPlans& e : es)
    if (e.mode == mode && e.batch == batch && e.base == base) {
      *out = &e;
      return ELASTO_OK;
    }
  NoallocPlans fresh;
  const elasto_status st = build_plans(h, mode, batch, base, L, &fresh);
  if (st != ELASTO_OK) return st;
  if (es.size() >= kMaxCachedPlans) es.erase(es.begin());
  es.push_back(std::move(fresh));
  *out = &es.back();
  return ELASTO_OK;
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
  int dev = -1;
  ELASTO_CUDA_TRY(cudaGetDevice(&dev));
  if (dev != h->dev) {
    set_error("elasto_forward_noalloc: the current device (" + std::to_string(dev) +
              ") is not the handle's device (" + std::to_string(h->dev) + ")");
    return ELASTO_ERR_INVALID_ARG;
  }
  const elasto_model_desc& d = h->d;
  const int mode = h->cur.load(std::memory_order_acquire);
  const VitMode& vm = h->modes[mode];
  const VitEmbed& em = vm.emb;
  int wmax = 64, fmax = 8;
  for (const VitLayerPack& lp : vm.layers) {
    wmax = lp.w > wmax ? lp.w : wmax;
    fmax = lp.f_pad > fmax ? lp.f_pad : fmax;
  }
  if (batch < 1 || layout_for(h, batch, em.d_pad, wmax, fmax).total > kScratchBytes) {
    int cap = 0;
    while (layout_for(h, cap + 1, em.d_pad, wmax, fmax).total <= kScratchBytes) ++cap;
    set_error("elasto_forward_noalloc: batch " + std::to_string(batch) + " is outside [1, " + std::to_string(cap) +
              "]: the 64 MiB static scratch holds at most " + std::to_string(cap) +
              " images of this model in this mode");
    return ELASTO_ERR_INVALID_ARG;
  }
  void* base = nullptr;
  elasto_status st = scratch_address(dev, &base);
  if (st != ELASTO_OK) return st;
  char* S = static_cast<char*>(base);
  const ScratchLayout L = layout_for(h, batch, em.d_pad, wmax, fmax);
  const NoallocPlans* P = nullptr;
  if ((st = plans_for(h, mode, batch, S, L, &P)) != ELASTO_OK) return st;
  float* X = reinterpret_cast<float*>(S + L.X);
  bf16* Y = reinterpret_cast<bf16*>(S + L.Y);
  bf16* Prow = reinterpret_cast<bf16*>(S + L.P);

  const int n = h->n, D = em.d_pad, M = batch * n;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ELASTO_CUDA_TRY(patch_rows_launch(images, d.weight_dtype, batch, d.img_h, d.img_w, d.img_c, d.patch, Prow, s));
  ELASTO_CUDA_TRY(gemm_launch(P->patch, M, s));
  for (int l = 0; l < d.layers; ++l) {
    const VitLayerPack& lp = vm.layers[l];
    const NoallocLayerPlans& q = P->layers[l];
    ELASTO_CUDA_TRY(layernorm_launch(X, em.ln1_w[l], em.ln1_b[l], Y, M, D, em.d, s));
    if (lp.w > 0) {
      ELASTO_CUDA_TRY(gemm_launch(q.qkv, M, s));
      ELASTO_CUDA_TRY(attn_launch(q.attn, batch, s));
    }
    ELASTO_CUDA_TRY(gemm_launch(q.proj, M, s));
    ELASTO_CUDA_TRY(layernorm_launch(X, em.ln2_w[l], em.ln2_b[l], Y, M, D, em.d, s));
    if (lp.f > 0) ELASTO_CUDA_TRY(gemm_launch(q.fc1, M, s));
    ELASTO_CUDA_TRY(gemm_launch(q.fc2, M, s));
  }
  ELASTO_CUDA_TRY(head_launch(X, batch, n, D, em.d, em.norm_w, em.norm_b, em.head_w, h->head_b, d.classes, logits, s));
  return ELASTO_OK;
}
