// C-ABI of libelasto: elastic model handle, create-time packing of every
// descendant network (DN), O(1) mode switching, and the forward pass.
//
// Section 4.3: all DNs share one parameter set and differ in which heads /
// MLP channels / conv channels they keep. The structured masks of Eq. 4, 6
// and 7 zero whole rows or columns; computing with zeros is wasted work, so at
// create time each mode's kept rows/columns are gathered into contiguous
// packed matrices (the kept-index tables play the role of the paper's
// "pruning metadata", Section 4.1-4.2). A mode switch then only swaps which
// packed set the next forward reads (Section 6.2 measures the paper's own
// switch cost): no weight moves on the request path.
#include <stdio.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <limits>
#include <memory>
#include <mutex>
#include <vector>

#include "common.h"
#include "elasto_internal.h"
#include "handle.h"

namespace elasto {

const char* last_error_cstr();

namespace {

constexpr size_t kAlign = 1024;

size_t dtype_size(int dt) { return dt == ELASTO_BF16 ? 2 : 4; }

bool tables_ok(const int32_t* idx, int n, int limit) {
  for (int i = 0; i < n; ++i) {
    if (idx[i] < 0 || idx[i] >= limit) return false;
    if (i > 0 && idx[i] <= idx[i - 1]) return false;
  }
  return true;
}

std::once_flag g_attr_once[64];
cudaError_t g_attr_err[64];

}  // namespace

cudaError_t ensure_kernel_attributes() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::call_once(g_attr_once[dev], [dev] {
    cudaError_t r = gemm_init_attributes();
    if (r == cudaSuccess) r = attn_init_attributes();
    if (r == cudaSuccess) r = cnn_init_attributes();
    if (r == cudaSuccess) r = pk_init_attributes();
    g_attr_err[dev] = r;
  });
  return g_attr_err[dev];
}

elasto_status check_device() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3) {
    char buf[128];
    snprintf(buf, sizeof buf, "libelasto is built for sm_103a (GB300); device %d is sm_%d%d", dev, major, minor);
    set_error(buf);
    return ELASTO_ERR_UNSUPPORTED;
  }
  e = ensure_kernel_attributes();
  if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute");
  return ELASTO_OK;
}

// ---------------------------------------------------------------- profiler
cudaError_t Profiler::enable(bool e) {
  if (e && !ev[0]) {
    for (int i = 0; i < 2 * kSlots; ++i) {
      cudaError_t r = cudaEventCreate(&ev[i]);
      if (r != cudaSuccess) return r;
    }
  }
  on = e;
  count = 0;
  return cudaSuccess;
}
cudaError_t Profiler::before(cudaStream_t s) {
  if (!on) return cudaSuccess;
  if (count >= kSlots) {
    overflow = true;
    return cudaSuccess;
  }
  return cudaEventRecord(ev[2 * count], s);
}
cudaError_t Profiler::after(cudaStream_t s, const elasto_launch_record& r) {
  if (!on || count >= kSlots) return cudaSuccess;
  rec[count] = r;
  cudaError_t e = cudaEventRecord(ev[2 * count + 1], s);
  ++count;
  return e;
}
elasto_status Profiler::read(elasto_launch_record* out, int capacity, int* n) {
  if (!on) {
    set_error("elasto_profile_read: profiling is not enabled");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (count > 0) ELASTO_CUDA_TRY(cudaEventSynchronize(ev[2 * count - 1]));
  const int m = count < capacity ? count : capacity;
  for (int i = 0; i < m; ++i) {
    out[i] = rec[i];
    ELASTO_CUDA_TRY(cudaEventElapsedTime(&out[i].ms, ev[2 * i], ev[2 * i + 1]));
  }
  *n = m;
  return ELASTO_OK;
}
void Profiler::release() {
  for (int i = 0; i < 2 * kSlots; ++i)
    if (ev[i]) cudaEventDestroy(ev[i]);
  on = false;
}

}  // namespace elasto

using namespace elasto;

// ============================================================================
// ViT
// ============================================================================

namespace {

elasto_status vit_validate(const elasto_model_desc* d) {
  if (d->img_h <= 0 || d->img_h != d->img_w || d->img_c <= 0 || d->patch <= 0 || d->img_h % d->patch != 0 ||
      d->dim <= 0 || d->heads <= 0 || d->dim != d->heads * 64 || d->mlp <= 0 || d->layers <= 0 ||
      d->classes <= 0) {
    set_error("elasto_create: inconsistent ViT descriptor (need img_h == img_w, patch | img_h, dim == 64 * heads)");
    return ELASTO_ERR_INVALID_ARG;
  }
  const int np = (d->img_h / d->patch) * (d->img_w / d->patch);
  const int kpe = d->patch * d->patch * d->img_c;
  if (np + 1 > 256) {
    set_error("elasto_create: at most 256 tokens (255 patches) are supported");
    return ELASTO_ERR_UNSUPPORTED;
  }
  if (kpe % 8 != 0 || d->dim % 64 != 0 || d->dim > 1024) {
    set_error("elasto_create: need patch*patch*channels % 8 == 0 and dim a multiple of 64 up to 1024");
    return ELASTO_ERR_UNSUPPORTED;
  }
  return ELASTO_OK;
}

elasto_status vit_validate_tables(const elasto_model_desc* d, const elasto_mode_tables* modes, int n_modes) {
  for (int m = 0; m < n_modes; ++m) {
    const elasto_mode_tables& t = modes[m];
    if (!t.n_heads_kept || !t.n_mlp_kept) {
      set_error("elasto_create: mode " + std::to_string(m) + " has no count arrays");
      return ELASTO_ERR_INVALID_ARG;
    }
    size_t ho = 0, fo = 0;
    for (int l = 0; l < d->layers; ++l) {
      const int nh = t.n_heads_kept[l], nf = t.n_mlp_kept[l];
      if (nh < 0 || nh > d->heads || nf < 0 || nf > d->mlp) {
        set_error("elasto_create: mode " + std::to_string(m) + " layer " + std::to_string(l) +
                  ": kept count out of range");
        return ELASTO_ERR_BAD_TABLE;
      }
      if ((nh > 0 && !t.heads_kept) || (nf > 0 && !t.mlp_kept)) {
        set_error("elasto_create: mode " + std::to_string(m) + ": null index table");
        return ELASTO_ERR_INVALID_ARG;
      }
      if ((nh > 0 && !tables_ok(t.heads_kept + ho, nh, d->heads)) ||
          (nf > 0 && !tables_ok(t.mlp_kept + fo, nf, d->mlp))) {
        set_error("elasto_create: mode " + std::to_string(m) + " layer " + std::to_string(l) +
                  ": kept indices must be strictly increasing and in range");
        return ELASTO_ERR_BAD_TABLE;
      }
      ho += nh;
      fo += nf;
    }
    if (t.n_embed_kept < 0 || t.n_embed_kept > d->dim || (t.n_embed_kept > 0 && !t.embed_kept)) {
      set_error("elasto_create: mode " + std::to_string(m) + ": embedding table count out of range or null");
      return ELASTO_ERR_BAD_TABLE;
    }
    if (t.n_embed_kept > 0 && !tables_ok(t.embed_kept, t.n_embed_kept, d->dim)) {
      set_error("elasto_create: mode " + std::to_string(m) +
                ": kept embedding channels must be strictly increasing and in range");
      return ELASTO_ERR_BAD_TABLE;
    }
  }
  return ELASTO_OK;
}

// Free-on-exit temporary device buffer.
struct DevTemp {
  void* p = nullptr;
  ~DevTemp() {
    if (p) cudaFree(p);
  }
};

// Everything that can be checked on the host, before any CUDA call.
elasto_status vit_check_inputs(const elasto_model_desc* d, const elasto_weights* wts,
                               const elasto_mode_tables* modes, int n_modes) {
  elasto_status st = vit_validate(d);
  if (st != ELASTO_OK) return st;
  if (wts->n_tensors != 8 + 12 * d->layers) {
    set_error("elasto_create: ViT expects 8 + 12 * layers weight tensors, got " + std::to_string(wts->n_tensors));
    return ELASTO_ERR_INVALID_ARG;
  }
  for (int i = 0; i < wts->n_tensors; ++i)
    if (!wts->tensors[i]) {
      set_error("elasto_create: weight tensor " + std::to_string(i) + " is null");
      return ELASTO_ERR_INVALID_ARG;
    }
  return vit_validate_tables(d, modes, n_modes);
}

// Nested kept sets (Eq. 8: DN_L contains DN_{L-1}): per layer, the modes'
// sets ordered by size form a chain S_1 <= S_2 <= ... Returns the prefix order
// S_1 (ascending), then S_2 \ S_1 (ascending), ..., so that every mode's set
// is a prefix of it; false if some pair of sets is not nested.
bool nested_order(const std::vector<std::vector<int32_t>>& sets, std::vector<int32_t>* order) {
  std::vector<int> by_size(sets.size());
  for (size_t i = 0; i < sets.size(); ++i) by_size[i] = static_cast<int>(i);
  std::stable_sort(by_size.begin(), by_size.end(),
                   [&](int a, int b) { return sets[a].size() < sets[b].size(); });
  order->clear();
  std::vector<int32_t> prev;
  for (int i : by_size) {
    const std::vector<int32_t>& cur = sets[i];  // sorted ascending (validated)
    if (!std::includes(cur.begin(), cur.end(), prev.begin(), prev.end())) return false;
    for (int32_t v : cur)
      if (!std::binary_search(prev.begin(), prev.end(), v)) order->push_back(v);
    prev = cur;
  }
  return true;
}

elasto_status vit_create(const elasto_model_desc* d, const elasto_weights* wts, const elasto_mode_tables* modes,
                         int n_modes, elasto_s* h) {
  elasto_status st = vit_check_inputs(d, wts, modes, n_modes);
  if (st != ELASTO_OK) return st;
  const int L = d->layers, D = d->dim, F = d->mlp, C = d->classes, Bm = d->max_batch;
  const int P = d->patch, np = (d->img_h / P) * (d->img_w / P), n = np + 1, kpe = P * P * d->img_c;
  h->n = n;
  h->np = np;
  h->kpe = kpe;

  // ---------------------------------------------------------------- layout
  GuardedArena& bump = h->guards;  // every buffer followed by a guard zone
  const size_t o_patch_w = bump.take(size_t(D) * kpe * 2, "patch projection weights");
  const size_t o_patch_b = bump.take(D * 4), o_cls = bump.take(D * 4), o_pos = bump.take(size_t(n) * D * 4);
  std::vector<size_t> o_l(6 * L);
  for (int l = 0; l < L; ++l)
    for (int k = 0; k < 6; ++k) o_l[6 * l + k] = bump.take(D * 4);
  const size_t o_norm_w = bump.take(D * 4), o_norm_b = bump.take(D * 4);
  const size_t o_head_w = bump.take(size_t(C) * D * 4, "classifier weights"), o_head_b = bump.take(C * 4, "classifier bias");
  h->shared_bytes = bump.off;

  h->modes.assign(n_modes, VitMode{});
  // fp32-stored models keep each weight as a bf16 pair (hi, lo): ~16 mantissa bits
  const bool split = d->weight_dtype == ELASTO_F32;
  struct Off {
    size_t qkv_w, qkv_b, proj_w, fc1_w, fc1_b, fc2_w;
    size_t qkv_lo = 0, proj_lo = 0, fc1_lo = 0, fc2_lo = 0;
  };
  std::vector<std::vector<Off>> offs(n_modes, std::vector<Off>(L));
  int wmax = 0, fmax = 0;
  // Prefix sharing when every layer's head and MLP sets are nested across the
  // modes and every MLP count is a multiple of 8 (a prefix then needs no
  // padding channels): one packed copy per layer instead of one per mode.
  h->perm_h.assign(L, {});
  h->perm_f.assign(L, {});
  // Embedding width per mode (Section 4.1): kept channels first, zero padding
  // up to a multiple of 64 (the GEMM tile and LayerNorm granularity).
  bool any_emb = false;
  for (int m = 0; m < n_modes; ++m) {
    VitEmbed& em = h->modes[m].emb;
    em.pruned = modes[m].n_embed_kept > 0 && modes[m].n_embed_kept < D;
    em.d = em.pruned ? modes[m].n_embed_kept : D;
    em.d_pad = (em.d + 63) / 64 * 64;
    any_emb = any_emb || em.pruned;
  }
  bool shared = n_modes > 1 && !any_emb;
  {
    std::vector<std::vector<std::vector<int32_t>>> hs(L), fs(L);
    for (int m = 0; m < n_modes; ++m) {
      for (int l = 0; l < L; ++l) {
        size_t a = 0, b = 0;
        for (int k = 0; k < l; ++k) {
          a += modes[m].n_heads_kept[k];
          b += modes[m].n_mlp_kept[k];
        }
        hs[l].emplace_back(modes[m].heads_kept + a, modes[m].heads_kept + a + modes[m].n_heads_kept[l]);
        fs[l].emplace_back(modes[m].mlp_kept + b, modes[m].mlp_kept + b + modes[m].n_mlp_kept[l]);
        if (modes[m].n_mlp_kept[l] % 8 != 0) shared = false;
      }
    }
    for (int l = 0; l < L && shared; ++l)
      shared = nested_order(hs[l], &h->perm_h[l]) && nested_order(fs[l], &h->perm_f[l]);
  }
  h->prefix_shared = shared;
  struct SharedOff {
    size_t qkv_w, qkv_b, proj_w, fc1_w, fc1_b, fc2_w, qkv_lo = 0, proj_lo = 0, fc1_lo = 0, fc2_lo = 0;
  };
  std::vector<SharedOff> soff(L);
  const size_t packed_start = bump.off;
  if (shared) {
    for (int l = 0; l < L; ++l) {
      const size_t hw = 64 * h->perm_h[l].size(), ff = h->perm_f[l].size();
      SharedOff& o = soff[l];
      o.qkv_w = bump.take(3 * hw * D * 2, "packed W_qkv");
      o.qkv_b = bump.take(3 * hw * 4);
      o.proj_w = bump.take(size_t(D) * hw * 2, "packed W_o");
      o.fc1_w = bump.take(ff * D * 2, "packed W1");
      o.fc1_b = bump.take(ff * 4);
      o.fc2_w = bump.take(size_t(D) * ff * 2, "packed W2");
      if (split) {
        o.qkv_lo = bump.take(3 * hw * D * 2);
        o.proj_lo = bump.take(size_t(D) * hw * 2);
        o.fc1_lo = bump.take(ff * D * 2);
        o.fc2_lo = bump.take(size_t(D) * ff * 2);
      }
    }
  }
  const int addend_rows = (1 + (128 + n - 1) / n) * n;
  struct EmbOff {
    size_t patch_w = 0, patch_lo = 0, patch_b = 0, cls = 0, pos = 0, norm_w = 0, norm_b = 0, head_w = 0, addend = 0;
    std::vector<size_t> lvec;  // per layer: ln1_w, ln1_b, ln2_w, ln2_b, proj_b, fc2_b
  };
  std::vector<EmbOff> eoffs(n_modes);
  for (int m = 0; m < n_modes; ++m) {
    const size_t start = bump.off;
    h->modes[m].layers.resize(L);
    const VitEmbed& em = h->modes[m].emb;
    const int Dm = em.d_pad;  // the width every d-axis of this mode's packs has
    if (em.pruned) {
      EmbOff& eo = eoffs[m];
      eo.patch_w = bump.take(size_t(Dm) * kpe * 2);
      if (split) eo.patch_lo = bump.take(size_t(Dm) * kpe * 2);
      eo.patch_b = bump.take(size_t(Dm) * 4);
      eo.cls = bump.take(size_t(Dm) * 4);
      eo.pos = bump.take(size_t(n) * Dm * 4);
      eo.norm_w = bump.take(size_t(Dm) * 4);
      eo.norm_b = bump.take(size_t(Dm) * 4);
      eo.head_w = bump.take(size_t(C) * Dm * 4);
      eo.addend = bump.take(size_t(addend_rows) * Dm * 4);
      for (int k = 0; k < 6 * L; ++k) eo.lvec.push_back(bump.take(size_t(Dm) * 4));
    }
    size_t view = 0;
    for (int l = 0; l < L; ++l) {
      VitLayerPack& lp = h->modes[m].layers[l];
      lp.w = 64 * modes[m].n_heads_kept[l];
      lp.f = modes[m].n_mlp_kept[l];
      // per-mode packs pad the MLP width to 64 channels: the rows of H and W2
      // (and the GELU epilogue's tiles) then start on 128-byte boundaries;
      // a prefix of the shared copy keeps f (a multiple of 8)
      lp.f_pad = shared ? lp.f : (lp.f + 63) / 64 * 64;
      lp.ld_proj = shared ? 64 * static_cast<int>(h->perm_h[l].size()) : lp.w;
      lp.ld_fc2 = shared ? static_cast<int>(h->perm_f[l].size()) : lp.f_pad;
      wmax = std::max(wmax, lp.w);
      fmax = std::max(fmax, lp.f_pad);
      view += (size_t(3) * lp.w * Dm * 2 + size_t(3) * lp.w * 4 + size_t(Dm) * lp.w * 2 + size_t(lp.f_pad) * Dm * 2 +
               size_t(lp.f_pad) * 4 + size_t(Dm) * lp.f_pad * 2) +
              (split ? size_t(3) * lp.w * Dm * 2 + size_t(Dm) * lp.w * 2 + size_t(lp.f_pad) * Dm * 4 : 0);
      if (shared) continue;
      Off& o = offs[m][l];
      o.qkv_w = bump.take(size_t(3) * lp.w * Dm * 2);
      o.qkv_b = bump.take(size_t(3) * lp.w * 4);
      o.proj_w = bump.take(size_t(Dm) * lp.w * 2);
      o.fc1_w = bump.take(size_t(lp.f_pad) * Dm * 2);
      o.fc1_b = bump.take(size_t(lp.f_pad) * 4);
      o.fc2_w = bump.take(size_t(Dm) * lp.f_pad * 2);
      if (split) {
        o.qkv_lo = bump.take(size_t(3) * lp.w * Dm * 2);
        o.proj_lo = bump.take(size_t(Dm) * lp.w * 2);
        o.fc1_lo = bump.take(size_t(lp.f_pad) * Dm * 2);
        o.fc2_lo = bump.take(size_t(Dm) * lp.f_pad * 2);
      }
    }
    h->modes[m].packed_bytes = shared ? view : bump.off - start;
  }
  h->packed_total = bump.off - packed_start;
  const size_t o_patch_lo = split ? bump.take(size_t(D) * kpe * 2) : 0;
  const size_t ws_start = bump.off;
  const size_t rows = size_t(Bm) * n;
  const size_t o_X = bump.take(rows * D * 4, "residual stream X"), o_Y = bump.take(rows * D * 2, "LayerNorm output Y");
  const size_t o_QKV = bump.take(rows * 3 * std::max(wmax, 64) * 2, "QKV"),
               o_O = bump.take(rows * std::max(wmax, 64) * 2, "attention output O");
  const size_t o_H = bump.take(rows * std::max(fmax, 8) * 2, "MLP hidden H"), o_P = bump.take(rows * kpe * 2, "patch rows P");
  // per-token addend of the patch projection: periodic in the token index, so
  // k images' worth (k * n >= n + 128 rows) serve every batch
  h->addend_rows = (1 + (128 + n - 1) / n) * n;
  const size_t o_tok = bump.take(size_t(h->addend_rows) * D * 4, "patch token addend");
  // split-K partial sums of the one-image FC2 (kSplitMax x n x D fp32)
  const size_t o_part = bump.take(size_t(kSplitMax) * n * D * 4, "split-K partial sums");
  const size_t img_bytes = size_t(Bm) * d->img_h * d->img_w * d->img_c * dtype_size(d->weight_dtype);
  const size_t o_img = bump.take(img_bytes, "image staging"), o_logit = bump.take(size_t(Bm) * C * 4, "logit staging");
  const size_t o_status = bump.take(64, "status word");
  const size_t o_pk_sync = bump.take(64, "one-launch barrier words");
  const size_t o_pk_y32 = bump.take(pk_workspace_floats(D) * 4, "one-launch class-token row");
  h->workspace_bytes = bump.off - ws_start;
  h->arena_bytes = bump.off;

  cudaError_t e = cudaMalloc(&h->arena, h->arena_bytes);
  if (e != cudaSuccess) {
    h->arena = nullptr;
    cudaGetLastError();
    set_error("elasto_create: cudaMalloc of " + std::to_string(h->arena_bytes) + " bytes failed");
    return ELASTO_ERR_OOM;
  }
  char* A = h->arena;
  h->patch_w = reinterpret_cast<bf16*>(A + o_patch_w);
  h->patch_w_lo = split ? reinterpret_cast<bf16*>(A + o_patch_lo) : nullptr;
  h->patch_b = reinterpret_cast<float*>(A + o_patch_b);
  h->cls = reinterpret_cast<float*>(A + o_cls);
  h->pos = reinterpret_cast<float*>(A + o_pos);
  for (int l = 0; l < L; ++l) {
    h->ln1_w.push_back(reinterpret_cast<float*>(A + o_l[6 * l + 0]));
    h->ln1_b.push_back(reinterpret_cast<float*>(A + o_l[6 * l + 1]));
    h->proj_b.push_back(reinterpret_cast<float*>(A + o_l[6 * l + 2]));
    h->ln2_w.push_back(reinterpret_cast<float*>(A + o_l[6 * l + 3]));
    h->ln2_b.push_back(reinterpret_cast<float*>(A + o_l[6 * l + 4]));
    h->fc2_b.push_back(reinterpret_cast<float*>(A + o_l[6 * l + 5]));
  }
  h->norm_w = reinterpret_cast<float*>(A + o_norm_w);
  h->norm_b = reinterpret_cast<float*>(A + o_norm_b);
  h->head_w = reinterpret_cast<float*>(A + o_head_w);
  h->head_b = reinterpret_cast<float*>(A + o_head_b);
  h->X = reinterpret_cast<float*>(A + o_X);
  h->splitk_part = reinterpret_cast<float*>(A + o_part);
  h->Y = reinterpret_cast<bf16*>(A + o_Y);
  h->QKV = reinterpret_cast<bf16*>(A + o_QKV);
  h->O = reinterpret_cast<bf16*>(A + o_O);
  h->H = reinterpret_cast<bf16*>(A + o_H);
  h->P = reinterpret_cast<bf16*>(A + o_P);
  h->tok_addend = reinterpret_cast<float*>(A + o_tok);
  h->img_stage = A + o_img;
  h->logit_stage = reinterpret_cast<float*>(A + o_logit);
  h->status = reinterpret_cast<int*>(A + o_status);
  h->pk_sync = reinterpret_cast<unsigned*>(A + o_pk_sync);
  h->pk_y32 = reinterpret_cast<float*>(A + o_pk_y32);
  for (int m = 0; m < n_modes; ++m) {
    VitEmbed& em = h->modes[m].emb;
    if (!em.pruned) {  // the handle's full-width parameters
      em.patch_w = h->patch_w;
      em.patch_w_lo = h->patch_w_lo;
      em.patch_b = h->patch_b;
      em.cls = h->cls;
      em.pos = h->pos;
      em.ln1_w = h->ln1_w;
      em.ln1_b = h->ln1_b;
      em.ln2_w = h->ln2_w;
      em.ln2_b = h->ln2_b;
      em.proj_b = h->proj_b;
      em.fc2_b = h->fc2_b;
      em.norm_w = h->norm_w;
      em.norm_b = h->norm_b;
      em.head_w = h->head_w;
      continue;
    }
    const EmbOff& eo = eoffs[m];
    em.patch_w = reinterpret_cast<bf16*>(A + eo.patch_w);
    em.patch_w_lo = split ? reinterpret_cast<bf16*>(A + eo.patch_lo) : nullptr;
    em.patch_b = reinterpret_cast<float*>(A + eo.patch_b);
    em.cls = reinterpret_cast<float*>(A + eo.cls);
    em.pos = reinterpret_cast<float*>(A + eo.pos);
    em.norm_w = reinterpret_cast<float*>(A + eo.norm_w);
    em.norm_b = reinterpret_cast<float*>(A + eo.norm_b);
    em.head_w = reinterpret_cast<float*>(A + eo.head_w);
    em.addend = reinterpret_cast<float*>(A + eo.addend);
    for (int l = 0; l < L; ++l) {
      em.ln1_w.push_back(reinterpret_cast<float*>(A + eo.lvec[6 * l + 0]));
      em.ln1_b.push_back(reinterpret_cast<float*>(A + eo.lvec[6 * l + 1]));
      em.ln2_w.push_back(reinterpret_cast<float*>(A + eo.lvec[6 * l + 2]));
      em.ln2_b.push_back(reinterpret_cast<float*>(A + eo.lvec[6 * l + 3]));
      em.proj_b.push_back(reinterpret_cast<float*>(A + eo.lvec[6 * l + 4]));
      em.fc2_b.push_back(reinterpret_cast<float*>(A + eo.lvec[6 * l + 5]));
    }
  }
  for (int m = 0; m < n_modes; ++m)
    for (int l = 0; l < L; ++l) {
      VitLayerPack& lp = h->modes[m].layers[l];
      if (shared) {  // every mode points at the one copy of the layer
        const SharedOff& o = soff[l];
        lp.qkv_w = reinterpret_cast<bf16*>(A + o.qkv_w);
        lp.qkv_b = reinterpret_cast<float*>(A + o.qkv_b);
        lp.proj_w = reinterpret_cast<bf16*>(A + o.proj_w);
        lp.fc1_w = reinterpret_cast<bf16*>(A + o.fc1_w);
        lp.fc1_b = reinterpret_cast<float*>(A + o.fc1_b);
        lp.fc2_w = reinterpret_cast<bf16*>(A + o.fc2_w);
        if (split) {
          lp.qkv_w_lo = reinterpret_cast<bf16*>(A + o.qkv_lo);
          lp.proj_w_lo = reinterpret_cast<bf16*>(A + o.proj_lo);
          lp.fc1_w_lo = reinterpret_cast<bf16*>(A + o.fc1_lo);
          lp.fc2_w_lo = reinterpret_cast<bf16*>(A + o.fc2_lo);
        }
        continue;
      }
      const Off& o = offs[m][l];
      lp.qkv_w = reinterpret_cast<bf16*>(A + o.qkv_w);
      lp.qkv_b = reinterpret_cast<float*>(A + o.qkv_b);
      lp.proj_w = reinterpret_cast<bf16*>(A + o.proj_w);
      lp.fc1_w = reinterpret_cast<bf16*>(A + o.fc1_w);
      lp.fc1_b = reinterpret_cast<float*>(A + o.fc1_b);
      lp.fc2_w = reinterpret_cast<bf16*>(A + o.fc2_w);
      if (split) {
        lp.qkv_w_lo = reinterpret_cast<bf16*>(A + o.qkv_lo);
        lp.proj_w_lo = reinterpret_cast<bf16*>(A + o.proj_lo);
        lp.fc1_w_lo = reinterpret_cast<bf16*>(A + o.fc1_lo);
        lp.fc2_w_lo = reinterpret_cast<bf16*>(A + o.fc2_lo);
      }
    }
  ELASTO_CUDA_TRY(cudaMemset(h->arena, 0, h->arena_bytes));
  {
    // guard zones filled right after the arena is cleared, before any
    // create-time kernel writes to it, so that those are checked too
    const elasto_status gs = h->guards.upload(h->arena);
    if (gs != ELASTO_OK) return gs;
  }

  // ---------------------------------------------------------------- upload
  const int dt = d->weight_dtype;
  const size_t es = dtype_size(dt);
  auto W = [&](int i) { return wts->tensors[i]; };
  // temp: raw upload buffer + canonical bf16 + canonical fp32 bias + index list
  const size_t max_mat = std::max({size_t(3) * D * D, size_t(F) * D, size_t(D) * kpe});
  DevTemp raw, canon, canon_lo, canon_b, idxbuf;
  ELASTO_CUDA_TRY(cudaMalloc(&raw.p, max_mat * 4 + size_t(n) * D * 4 + size_t(C) * D * 4));
  ELASTO_CUDA_TRY(cudaMalloc(&canon.p, max_mat * 2));
  if (split) ELASTO_CUDA_TRY(cudaMalloc(&canon_lo.p, max_mat * 2));
  ELASTO_CUDA_TRY(cudaMalloc(&canon_b.p, size_t(std::max(3 * D, F)) * 4));
  ELASTO_CUDA_TRY(cudaMalloc(&idxbuf.p, size_t(std::max(3 * D, F) + 64) * 4));
  // embedding-pruned modes: each mode's kept channels padded with -1 to d_pad
  // (at m * D), and 0, 1, 2, ... for the axes gathered whole
  DevTemp eidx, iota;
  const int n_iota = std::max({kpe, n, C});
  if (any_emb) {
    std::vector<int32_t> host(size_t(n_modes) * D, -1), io(n_iota);
    for (int m = 0; m < n_modes; ++m)
      if (h->modes[m].emb.pruned)
        std::copy(modes[m].embed_kept, modes[m].embed_kept + modes[m].n_embed_kept, host.begin() + size_t(m) * D);
    for (int i = 0; i < n_iota; ++i) io[i] = i;
    ELASTO_CUDA_TRY(cudaMalloc(&eidx.p, host.size() * 4));
    ELASTO_CUDA_TRY(cudaMalloc(&iota.p, io.size() * 4));
    ELASTO_CUDA_TRY(cudaMemcpy(eidx.p, host.data(), host.size() * 4, cudaMemcpyHostToDevice));
    ELASTO_CUDA_TRY(cudaMemcpy(iota.p, io.data(), io.size() * 4, cudaMemcpyHostToDevice));
  }
  auto eix = [&](int m) { return static_cast<const int32_t*>(eidx.p) + size_t(m) * D; };
  const int32_t* iot = static_cast<const int32_t*>(iota.p);
  cudaStream_t s = 0;

  auto up_f32 = [&](const void* src, size_t count, float* dst) -> elasto_status {
    ELASTO_CUDA_TRY(cudaMemcpy(raw.p, src, count * es, cudaMemcpyHostToDevice));
    ELASTO_CUDA_TRY(convert_to_f32(raw.p, dt, count, dst, s));
    return ELASTO_OK;
  };
  auto up_bf16 = [&](const void* src, size_t count, bf16* dst) -> elasto_status {
    ELASTO_CUDA_TRY(cudaMemcpy(raw.p, src, count * es, cudaMemcpyHostToDevice));
    ELASTO_CUDA_TRY(convert_to_bf16(raw.p, dt, count, dst, s));
    return ELASTO_OK;
  };
#define UP(expr)                       \
  do {                                 \
    elasto_status s_ = (expr);         \
    if (s_ != ELASTO_OK) return s_;    \
  } while (0)

  // patch_w [d, C, P, P] -> packed [d, (ky, kx, c)] to match NHWC patch rows
  {
    std::vector<char> re(size_t(D) * kpe * es);
    const char* src = static_cast<const char*>(W(0));
    const int Cc = d->img_c;
    for (int o = 0; o < D; ++o)
      for (int c = 0; c < Cc; ++c)
        for (int ky = 0; ky < P; ++ky)
          for (int kx = 0; kx < P; ++kx) {
            const size_t si = ((size_t(o) * Cc + c) * P + ky) * P + kx;
            const size_t di = size_t(o) * kpe + (size_t(ky) * P + kx) * Cc + c;
            memcpy(re.data() + di * es, src + si * es, es);
          }
    UP(up_bf16(re.data(), size_t(D) * kpe, h->patch_w));
    if (split) ELASTO_CUDA_TRY(convert_to_bf16_lo(raw.p, dt, size_t(D) * kpe, h->patch_w_lo, s));
  }
  UP(up_f32(W(1), D, h->patch_b));
  UP(up_f32(W(2), D, h->cls));
  UP(up_f32(W(3), size_t(n) * D, h->pos));
  const int base_final = 4 + 12 * L;
  UP(up_f32(W(base_final + 0), D, h->norm_w));
  UP(up_f32(W(base_final + 1), D, h->norm_b));
  UP(up_f32(W(base_final + 2), size_t(C) * D, h->head_w));
  UP(up_f32(W(base_final + 3), C, h->head_b));
  for (int m = 0; m < n_modes; ++m) {
    const VitEmbed& em = h->modes[m].emb;
    if (!em.pruned) continue;
    const int Dm = em.d_pad;
    ELASTO_CUDA_TRY(gather2d_bf16(h->patch_w, kpe, eix(m), Dm, iot, kpe, em.patch_w, s));
    if (split) ELASTO_CUDA_TRY(gather2d_bf16(h->patch_w_lo, kpe, eix(m), Dm, iot, kpe, em.patch_w_lo, s));
    ELASTO_CUDA_TRY(gather_f32(h->patch_b, eix(m), Dm, em.patch_b, s));
    ELASTO_CUDA_TRY(gather_f32(h->cls, eix(m), Dm, em.cls, s));
    ELASTO_CUDA_TRY(gather2d_f32(h->pos, D, iot, n, eix(m), Dm, em.pos, s));
    ELASTO_CUDA_TRY(gather_f32(h->norm_w, eix(m), Dm, em.norm_w, s));
    ELASTO_CUDA_TRY(gather_f32(h->norm_b, eix(m), Dm, em.norm_b, s));
    ELASTO_CUDA_TRY(gather2d_f32(h->head_w, D, iot, C, eix(m), Dm, em.head_w, s));
  }

  std::vector<int32_t> idx;
  for (int l = 0; l < L; ++l) {
    const int t0 = 4 + 12 * l;  // ln1_w, ln1_b, qkv_w, qkv_b, proj_w, proj_b, ln2_w, ln2_b, fc1_w, fc1_b, fc2_w, fc2_b
    UP(up_f32(W(t0 + 0), D, h->ln1_w[l]));
    UP(up_f32(W(t0 + 1), D, h->ln1_b[l]));
    UP(up_f32(W(t0 + 5), D, h->proj_b[l]));
    UP(up_f32(W(t0 + 6), D, h->ln2_w[l]));
    UP(up_f32(W(t0 + 7), D, h->ln2_b[l]));
    UP(up_f32(W(t0 + 11), D, h->fc2_b[l]));
    for (int m = 0; m < n_modes; ++m) {
      const VitEmbed& em = h->modes[m].emb;
      if (!em.pruned) continue;
      const std::pair<const float*, float*> v[6] = {{h->ln1_w[l], em.ln1_w[l]}, {h->ln1_b[l], em.ln1_b[l]},
                                                     {h->ln2_w[l], em.ln2_w[l]}, {h->ln2_b[l], em.ln2_b[l]},
                                                     {h->proj_b[l], em.proj_b[l]}, {h->fc2_b[l], em.fc2_b[l]}};
      for (const auto& pr : v) ELASTO_CUDA_TRY(gather_f32(pr.first, eix(m), em.d_pad, pr.second, s));
    }
    bf16* cw = static_cast<bf16*>(canon.p);
    bf16* cwl = static_cast<bf16*>(canon_lo.p);
    float* cb = static_cast<float*>(canon_b.p);
    int32_t* di = static_cast<int32_t*>(idxbuf.p);
    // qkv: rows {blk * d + j * 64 + r}
    UP(up_bf16(W(t0 + 2), size_t(3) * D * D, cw));
    if (split) ELASTO_CUDA_TRY(convert_to_bf16_lo(raw.p, dt, size_t(3) * D * D, cwl, s));
    UP(up_f32(W(t0 + 3), size_t(3) * D, cb));
    // shared copy: head-interleaved rows {p * 192 + blk * 64 + r} <- {blk * d + perm[p] * 64 + r}
    const VitLayerPack& sp = h->modes[0].layers[l];  // its pointers are the shared copy's
    const std::vector<int32_t>& ph = h->perm_h[l];
    const std::vector<int32_t>& pf = h->perm_f[l];
    if (shared && !ph.empty()) {
      idx.clear();
      for (int32_t j : ph)
        for (int blk = 0; blk < 3; ++blk)
          for (int r = 0; r < 64; ++r) idx.push_back(blk * D + j * 64 + r);
      ELASTO_CUDA_TRY(cudaMemcpy(di, idx.data(), idx.size() * 4, cudaMemcpyHostToDevice));
      ELASTO_CUDA_TRY(gather_rows_bf16(cw, D, di, int(idx.size()), sp.qkv_w, s));
      if (split) ELASTO_CUDA_TRY(gather_rows_bf16(cwl, D, di, int(idx.size()), sp.qkv_w_lo, s));
      ELASTO_CUDA_TRY(gather_f32(cb, di, int(idx.size()), sp.qkv_b, s));
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
    for (int m = 0; m < n_modes && !shared; ++m) {
      VitLayerPack& lp = h->modes[m].layers[l];
      if (lp.w == 0) continue;
      size_t ho = 0;
      for (int k = 0; k < l; ++k) ho += modes[m].n_heads_kept[k];
      const int32_t* hk = modes[m].heads_kept + ho;
      idx.clear();
      for (int blk = 0; blk < 3; ++blk)
        for (int j = 0; j < lp.w / 64; ++j)
          for (int r = 0; r < 64; ++r) idx.push_back(blk * D + hk[j] * 64 + r);
      ELASTO_CUDA_TRY(cudaMemcpy(di, idx.data(), idx.size() * 4, cudaMemcpyHostToDevice));
      const VitEmbed& em = h->modes[m].emb;
      if (em.pruned) {  // input columns: the kept embedding channels
        ELASTO_CUDA_TRY(gather2d_bf16(cw, D, di, int(idx.size()), eix(m), em.d_pad, lp.qkv_w, s));
        if (split) ELASTO_CUDA_TRY(gather2d_bf16(cwl, D, di, int(idx.size()), eix(m), em.d_pad, lp.qkv_w_lo, s));
      } else {
        ELASTO_CUDA_TRY(gather_rows_bf16(cw, D, di, int(idx.size()), lp.qkv_w, s));
        if (split) ELASTO_CUDA_TRY(gather_rows_bf16(cwl, D, di, int(idx.size()), lp.qkv_w_lo, s));
      }
      ELASTO_CUDA_TRY(gather_f32(cb, di, int(idx.size()), lp.qkv_b, s));
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
    // proj: columns {j * 64 + r}
    UP(up_bf16(W(t0 + 4), size_t(D) * D, cw));
    if (split) ELASTO_CUDA_TRY(convert_to_bf16_lo(raw.p, dt, size_t(D) * D, cwl, s));
    if (shared && !ph.empty()) {  // columns {perm[p] * 64 + r}
      idx.clear();
      for (int32_t j : ph)
        for (int r = 0; r < 64; ++r) idx.push_back(j * 64 + r);
      ELASTO_CUDA_TRY(cudaMemcpy(di, idx.data(), idx.size() * 4, cudaMemcpyHostToDevice));
      ELASTO_CUDA_TRY(gather_cols_bf16(cw, D, D, di, int(idx.size()), sp.proj_w, s));
      if (split) ELASTO_CUDA_TRY(gather_cols_bf16(cwl, D, D, di, int(idx.size()), sp.proj_w_lo, s));
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
    for (int m = 0; m < n_modes && !shared; ++m) {
      VitLayerPack& lp = h->modes[m].layers[l];
      if (lp.w == 0) continue;
      size_t ho = 0;
      for (int k = 0; k < l; ++k) ho += modes[m].n_heads_kept[k];
      const int32_t* hk = modes[m].heads_kept + ho;
      idx.clear();
      for (int j = 0; j < lp.w / 64; ++j)
        for (int r = 0; r < 64; ++r) idx.push_back(hk[j] * 64 + r);
      ELASTO_CUDA_TRY(cudaMemcpy(di, idx.data(), idx.size() * 4, cudaMemcpyHostToDevice));
      const VitEmbed& em = h->modes[m].emb;
      if (em.pruned) {  // output rows: the kept embedding channels
        ELASTO_CUDA_TRY(gather2d_bf16(cw, D, eix(m), em.d_pad, di, int(idx.size()), lp.proj_w, s));
        if (split) ELASTO_CUDA_TRY(gather2d_bf16(cwl, D, eix(m), em.d_pad, di, int(idx.size()), lp.proj_w_lo, s));
      } else {
        ELASTO_CUDA_TRY(gather_cols_bf16(cw, D, D, di, int(idx.size()), lp.proj_w, s));
        if (split) ELASTO_CUDA_TRY(gather_cols_bf16(cwl, D, D, di, int(idx.size()), lp.proj_w_lo, s));
      }
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
    // fc1: rows F (padding rows stay zero), b1 entries F
    UP(up_bf16(W(t0 + 8), size_t(F) * D, cw));
    if (split) ELASTO_CUDA_TRY(convert_to_bf16_lo(raw.p, dt, size_t(F) * D, cwl, s));
    UP(up_f32(W(t0 + 9), F, cb));
    if (shared && !pf.empty()) {  // rows perm_f
      ELASTO_CUDA_TRY(cudaMemcpy(di, pf.data(), pf.size() * 4, cudaMemcpyHostToDevice));
      ELASTO_CUDA_TRY(gather_rows_bf16(cw, D, di, int(pf.size()), sp.fc1_w, s));
      if (split) ELASTO_CUDA_TRY(gather_rows_bf16(cwl, D, di, int(pf.size()), sp.fc1_w_lo, s));
      ELASTO_CUDA_TRY(gather_f32(cb, di, int(pf.size()), sp.fc1_b, s));
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
    for (int m = 0; m < n_modes && !shared; ++m) {
      VitLayerPack& lp = h->modes[m].layers[l];
      if (lp.f == 0) continue;
      size_t fo = 0;
      for (int k = 0; k < l; ++k) fo += modes[m].n_mlp_kept[k];
      ELASTO_CUDA_TRY(cudaMemcpy(di, modes[m].mlp_kept + fo, size_t(lp.f) * 4, cudaMemcpyHostToDevice));
      const VitEmbed& em = h->modes[m].emb;
      if (em.pruned) {  // input columns: the kept embedding channels
        ELASTO_CUDA_TRY(gather2d_bf16(cw, D, di, lp.f, eix(m), em.d_pad, lp.fc1_w, s));
        if (split) ELASTO_CUDA_TRY(gather2d_bf16(cwl, D, di, lp.f, eix(m), em.d_pad, lp.fc1_w_lo, s));
      } else {
        ELASTO_CUDA_TRY(gather_rows_bf16(cw, D, di, lp.f, lp.fc1_w, s));
        if (split) ELASTO_CUDA_TRY(gather_rows_bf16(cwl, D, di, lp.f, lp.fc1_w_lo, s));
      }
      ELASTO_CUDA_TRY(gather_f32(cb, di, lp.f, lp.fc1_b, s));
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
    // fc2: columns F into [d, f_pad] (padding columns zero)
    UP(up_bf16(W(t0 + 10), size_t(D) * F, cw));
    if (split) ELASTO_CUDA_TRY(convert_to_bf16_lo(raw.p, dt, size_t(D) * F, cwl, s));
    if (shared && !pf.empty()) {  // columns perm_f
      ELASTO_CUDA_TRY(cudaMemcpy(di, pf.data(), pf.size() * 4, cudaMemcpyHostToDevice));
      ELASTO_CUDA_TRY(gather_cols_bf16(cw, D, F, di, int(pf.size()), sp.fc2_w, s));
      if (split) ELASTO_CUDA_TRY(gather_cols_bf16(cwl, D, F, di, int(pf.size()), sp.fc2_w_lo, s));
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
    for (int m = 0; m < n_modes && !shared; ++m) {
      VitLayerPack& lp = h->modes[m].layers[l];
      if (lp.f == 0) continue;
      size_t fo = 0;
      for (int k = 0; k < l; ++k) fo += modes[m].n_mlp_kept[k];
      idx.assign(modes[m].mlp_kept + fo, modes[m].mlp_kept + fo + lp.f);
      for (int k = lp.f; k < lp.f_pad; ++k) idx.push_back(-1);
      ELASTO_CUDA_TRY(cudaMemcpy(di, idx.data(), idx.size() * 4, cudaMemcpyHostToDevice));
      const VitEmbed& em = h->modes[m].emb;
      if (em.pruned) {  // output rows: the kept embedding channels
        ELASTO_CUDA_TRY(gather2d_bf16(cw, F, eix(m), em.d_pad, di, lp.f_pad, lp.fc2_w, s));
        if (split) ELASTO_CUDA_TRY(gather2d_bf16(cwl, F, eix(m), em.d_pad, di, lp.f_pad, lp.fc2_w_lo, s));
      } else {
        ELASTO_CUDA_TRY(gather_cols_bf16(cw, D, F, di, lp.f_pad, lp.fc2_w, s));
        if (split) ELASTO_CUDA_TRY(gather_cols_bf16(cwl, D, F, di, lp.f_pad, lp.fc2_w_lo, s));
      }
      ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
    }
  }
#undef UP
  ELASTO_CUDA_TRY(cudaDeviceSynchronize());

  // ---------------------------------------------------------------- plans
  const int Mcap = Bm * n;
  // Patch projection over token-ordered rows (class-token slots are zero
  // rows): X = addend + P W_pe^T, addend = cls + pos[0] on class tokens and
  // pos[t] + b_pe on patch tokens (Section 4.1: N = HW/P^2 patches, n = N + 1).
  ELASTO_CUDA_TRY(token_addend_launch(h->cls, h->pos, h->patch_b, n, D, h->addend_rows / n, h->tok_addend, 0));
  for (int m = 0; m < n_modes; ++m) {
    const VitEmbed& em = h->modes[m].emb;
    if (em.pruned)
      ELASTO_CUDA_TRY(
          token_addend_launch(em.cls, em.pos, em.patch_b, n, em.d_pad, h->addend_rows / n, em.addend, 0));
  }
  // plan variants for 1, 8 and 32 images (those below max_batch) and max_batch
  h->n_plan_rows = 0;
  for (int b : {1, 8, 32})
    if (b < Bm) h->plan_rows[h->n_plan_rows++] = b * n;
  h->plan_rows[h->n_plan_rows++] = Mcap;
  // One GemmPlanSet filled with a plan per bucket by `make(plan, rows)`.
  auto plan_set = [&](GemmPlanSet& set, auto&& make) -> elasto_status {
    set.n = h->n_plan_rows;
    for (int i = 0; i < set.n; ++i) {
      set.rows[i] = h->plan_rows[i];
      const elasto_status r = make(set.plan[i], set.rows[i]);
      if (r != ELASTO_OK) return r;
    }
    return ELASTO_OK;
  };
  st = plan_set(h->patch, [&](GemmPlan& gp, int rows) {
    elasto_status r = gemm_plan(&gp, h->P, Mcap, h->patch_w, D, kpe, nullptr, h->X, D, EPI_BIAS_RESID_F32,
                                h->status, h->patch_w_lo, rows);
    return r != ELASTO_OK ? r : gemm_set_residual_source(&gp, h->tok_addend, h->addend_rows, n);
  });
  if (st != ELASTO_OK) return st;
  ELASTO_CUDA_TRY(cudaDeviceSynchronize());
  for (int m = 0; m < n_modes; ++m) {
    VitMode& vm = h->modes[m];
    VitEmbed& em = vm.emb;
    const int Dm = em.d_pad, dm = em.d;  // padded and kept embedding width
    vm.macs = int64_t(np) * dm * kpe + int64_t(dm) * C;
    vm.launches = 3;  // patchify, patch GEMM, head
    if (em.pruned) {  // the patch projection at this mode's width, its own addend
      st = plan_set(em.patch, [&](GemmPlan& gp, int rows) {
        elasto_status r = gemm_plan(&gp, h->P, Mcap, em.patch_w, Dm, kpe, nullptr, h->X, Dm, EPI_BIAS_RESID_F32,
                                    h->status, em.patch_w_lo, rows);
        return r != ELASTO_OK ? r : gemm_set_residual_source(&gp, em.addend, h->addend_rows, n);
      });
      if (st != ELASTO_OK) return st;
    }
    for (int l = 0; l < L; ++l) {
      VitLayerPack& lp = vm.layers[l];
      vm.macs += int64_t(n) * dm * 3 * lp.w + 2 * int64_t(n) * n * lp.w + int64_t(n) * lp.w * dm +
                 2 * int64_t(n) * dm * lp.f;
      vm.launches += 2;  // two LayerNorms
      if (lp.w > 0) {
        st = plan_set(lp.qkv, [&](GemmPlan& gp, int rows) {
          return gemm_plan(&gp, h->Y, Mcap, lp.qkv_w, 3 * lp.w, Dm, lp.qkv_b, h->QKV, 3 * lp.w, EPI_BIAS_BF16,
                           h->status, lp.qkv_w_lo, rows);
        });
        if (st != ELASTO_OK) return st;
        st = attn_plan(&lp.attn, h->QKV, h->O, Bm, n, lp.w / 64, h->status, shared);
        if (st != ELASTO_OK) return st;
        vm.launches += 2;
      }
      st = plan_set(lp.proj, [&](GemmPlan& gp, int rows) {
        // one image: the reduction split over idle SMs, and LN2 computed by
        // the launch that adds the partial sums
        if (rows <= n) {
          const elasto_status r = gemm_plan_split_resid(&gp, h->O, Mcap, lp.proj_w, Dm, lp.w, em.proj_b[l], h->X, Dm,
                                                        h->status, lp.proj_w_lo, rows, lp.ld_proj, h->splitk_part);
          if (r == ELASTO_OK) gemm_split_fuse_layernorm(&gp, em.ln2_w[l], em.ln2_b[l], h->Y, em.d);
          return r;
        }
        return gemm_plan(&gp, h->O, Mcap, lp.proj_w, Dm, lp.w, em.proj_b[l], h->X, Dm, EPI_BIAS_RESID_F32, h->status,
                         lp.proj_w_lo, rows, lp.ld_proj);
      });
      if (st != ELASTO_OK) return st;
      if (lp.f > 0) {
        st = plan_set(lp.fc1, [&](GemmPlan& gp, int rows) {
          return gemm_plan(&gp, h->Y, Mcap, lp.fc1_w, lp.f_pad, Dm, lp.fc1_b, h->H, lp.f_pad, EPI_BIAS_GELU_BF16,
                           h->status, lp.fc1_w_lo, rows);
        });
        if (st != ELASTO_OK) return st;
        vm.launches += 1;
      }
      st = plan_set(lp.fc2, [&](GemmPlan& gp, int rows) {
        // one image: the 3072-long reduction split over the idle SMs, and
        // the next layer's LN1 computed by the launch that adds the partials
        if (rows <= n) {
          const elasto_status r = gemm_plan_split_resid(&gp, h->H, Mcap, lp.fc2_w, Dm, lp.f_pad, em.fc2_b[l], h->X,
                                                        Dm, h->status, lp.fc2_w_lo, rows, lp.ld_fc2, h->splitk_part);
          if (r == ELASTO_OK && l + 1 < L) gemm_split_fuse_layernorm(&gp, em.ln1_w[l + 1], em.ln1_b[l + 1], h->Y, em.d);
          return r;
        }
        return gemm_plan(&gp, h->H, Mcap, lp.fc2_w, Dm, lp.f_pad, em.fc2_b[l], h->X, Dm, EPI_BIAS_RESID_F32, h->status,
                         lp.fc2_w_lo, rows, lp.ld_fc2);
      });
      if (st != ELASTO_OK) return st;
      vm.launches += 2;
    }
  }
  // one-image forwards as one persistent launch, where the mode allows it
  return pk_build(h, h->pk_sync, h->pk_y32, &h->pk);
}

elasto_launch_record make_rec(int kind, int layer, int m, int n, int k, double macs, double bytes) {
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

// GEMM record: A [M,K] and W [N,K] bf16 read once, out [M,N] written (and
// read too for a residual epilogue).
elasto_launch_record gemm_rec(int layer, int M, int N, int K, int out_bytes, bool resid) {
  const double mn = double(M) * N;
  return make_rec(ELASTO_K_GEMM, layer, M, N, K, mn * K,
                  2.0 * M * K + 2.0 * N * K + mn * out_bytes * (resid ? 2 : 1));
}

#define ELASTO_LAUNCH(rec, expr)                 \
  do {                                           \
    ELASTO_CUDA_TRY(h->prof.before(s));          \
    ELASTO_CUDA_TRY(expr);                       \
    ELASTO_CUDA_TRY(h->prof.after(s, (rec)));    \
  } while (0)

elasto_status vit_forward(elasto_s* h, cudaStream_t s, const void* images, int batch, float* logits) {
  const elasto_model_desc& d = h->d;
  const int mode = h->cur.load(std::memory_order_acquire);
  const VitMode& vm = h->modes[mode];
  const int n = h->n, D = d.dim, M = batch * n, Mp = batch * h->np, C = d.classes;
  const double img_elt = d.weight_dtype == ELASTO_BF16 ? 2 : 4;
  const VitEmbed& em = vm.emb;
  const int Dm = em.d_pad;  // residual-stream width (kept embedding channels, zero-padded)
  h->prof.begin();
  if (batch == 1 && pk_ready(h->pk, mode)) {
    // the whole forward as one persistent launch (csrc/persistent.cu);
    // algorithmic bytes: the mode's weights, the image and the logits
    ELASTO_LAUNCH(make_rec(ELASTO_K_ONE_LAUNCH, -1, n, Dm, 0, double(vm.macs),
                           double(vm.packed_bytes + h->shared_bytes) + double(h->np) * h->kpe * img_elt +
                               double(C) * 4),
                  pk_launch(h->pk, mode, n, images, logits, h->status, s));
    return ELASTO_OK;
  }
  ELASTO_LAUNCH(make_rec(ELASTO_K_PATCHIFY, -1, M, h->kpe, 0, 0, double(Mp) * h->kpe * img_elt + double(M) * h->kpe * 2),
                patch_rows_launch(images, d.weight_dtype, batch, d.img_h, d.img_w, d.img_c, d.patch, h->P, s));
  // patch projection; the addend (class token / position embedding / b_pe)
  // is periodic in the token and read from L2
  ELASTO_LAUNCH(gemm_rec(-1, M, Dm, h->kpe, 4, false),
                gemm_launch((em.pruned ? em.patch : h->patch).pick(M), M, s));
  const double ln_bytes = double(M) * Dm * (4 + 2);
  for (int l = 0; l < d.layers; ++l) {
    const VitLayerPack& lp = vm.layers[l];
    // LN1 / LN2 are skipped where the previous GEMM's split-K sum computed them
    if (l == 0 || !vm.layers[l - 1].fc2.pick(M).ln_y)
      ELASTO_LAUNCH(make_rec(ELASTO_K_LAYERNORM, l, M, Dm, 0, 0, ln_bytes),
                    layernorm_launch(h->X, em.ln1_w[l], em.ln1_b[l], h->Y, M, Dm, em.d, s));
    if (lp.w > 0) {
      ELASTO_LAUNCH(gemm_rec(l, M, 3 * lp.w, Dm, 2, false), gemm_launch(lp.qkv.pick(M), M, s));
      ELASTO_LAUNCH(make_rec(ELASTO_K_ATTENTION, l, M, lp.w, n, 2.0 * batch * n * n * lp.w,
                             double(M) * lp.w * 2 * 4),
                    attn_launch(lp.attn, batch, s));
    }
    ELASTO_LAUNCH(gemm_rec(l, M, Dm, lp.w, 4, true), gemm_launch(lp.proj.pick(M), M, s));
    if (!lp.proj.pick(M).ln_y)
      ELASTO_LAUNCH(make_rec(ELASTO_K_LAYERNORM, l, M, Dm, 0, 0, ln_bytes),
                    layernorm_launch(h->X, em.ln2_w[l], em.ln2_b[l], h->Y, M, Dm, em.d, s));
    if (lp.f > 0) ELASTO_LAUNCH(gemm_rec(l, M, lp.f_pad, Dm, 2, false), gemm_launch(lp.fc1.pick(M), M, s));
    ELASTO_LAUNCH(gemm_rec(l, M, Dm, lp.f_pad, 4, true), gemm_launch(lp.fc2.pick(M), M, s));
  }
  ELASTO_LAUNCH(make_rec(ELASTO_K_HEAD, -1, batch, C, Dm, double(batch) * C * em.d,
                         double(batch) * Dm * 4 + double(C) * Dm * 4 + double(batch) * C * 4),
                head_launch(h->X, batch, n, Dm, em.d, em.norm_w, em.norm_b, em.head_w, h->head_b, C, logits, s));
  return ELASTO_OK;
}

}  // namespace

// ============================================================================
// Exported C-ABI
// ============================================================================
extern "C" {

elasto_status elasto_create(const elasto_model_desc* desc, const elasto_weights* weights,
                            const elasto_mode_tables* modes, int n_modes, elasto_t* out) {
  clear_error();
  if (!desc || !weights || !weights->tensors || !modes || n_modes <= 0 || !out) {
    set_error("elasto_create: null argument or n_modes <= 0");
    return ELASTO_ERR_INVALID_ARG;
  }
  *out = nullptr;
  if (desc->max_batch <= 0 || (desc->weight_dtype != ELASTO_F32 && desc->weight_dtype != ELASTO_BF16)) {
    set_error("elasto_create: max_batch must be >= 1 and weight_dtype ELASTO_F32 or ELASTO_BF16");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (desc->arch != ELASTO_ARCH_VIT && desc->arch != ELASTO_ARCH_RESNET50) {
    set_error("elasto_create: unknown arch");
    return ELASTO_ERR_INVALID_ARG;
  }
  elasto_status st = desc->arch == ELASTO_ARCH_VIT ? vit_check_inputs(desc, weights, modes, n_modes)
                                                   : cnn_check_inputs(desc, weights, modes, n_modes);
  if (st != ELASTO_OK) return st;
  st = check_device();
  if (st != ELASTO_OK) return st;
  std::unique_ptr<elasto_s> h(new elasto_s());
  h->d = *desc;
  cudaGetDevice(&h->dev);
  if (desc->arch == ELASTO_ARCH_VIT) {
    st = vit_create(desc, weights, modes, n_modes, h.get());
  } else {
    h->cnn = cnn_new();
    st = cnn_create(desc, weights, modes, n_modes, h->cnn);
  }
  if (st != ELASTO_OK) {
    cudaDeviceSynchronize();
    if (h->arena) cudaFree(h->arena);
    h->guards.release();
    pk_free(h->pk);
    if (h->cnn) cnn_destroy(h->cnn);
    return st;
  }
  h->cur.store(0);
  *out = h.release();
  return ELASTO_OK;
}

elasto_status elasto_set_mode(elasto_t h, int mode) {
  if (!h) {
    set_error("elasto_set_mode: null handle");
    return ELASTO_ERR_INVALID_ARG;
  }
  const int nm = h->cnn ? cnn_n_modes(h->cnn) : static_cast<int>(h->modes.size());
  if (mode < 0 || mode >= nm) {
    set_error("elasto_set_mode: mode " + std::to_string(mode) + " out of range [0, " + std::to_string(nm) + ")");
    return ELASTO_ERR_BAD_MODE;
  }
  h->cur.store(mode, std::memory_order_release);
  return ELASTO_OK;
}

elasto_status elasto_get_mode(elasto_t h, int* mode) {
  if (!h || !mode) {
    set_error("elasto_get_mode: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  *mode = h->cur.load(std::memory_order_acquire);
  return ELASTO_OK;
}

elasto_status elasto_forward(elasto_t h, void* stream, const void* images, int batch, float* logits) {
  if (!h || !images || !logits) {
    set_error("elasto_forward: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (batch < 1 || batch > h->d.max_batch) {
    set_error("elasto_forward: batch " + std::to_string(batch) + " outside [1, max_batch]");
    return ELASTO_ERR_INVALID_ARG;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (h->cnn) return cnn_forward(h->cnn, h->cur.load(std::memory_order_acquire), s, images, batch, logits);
  return vit_forward(h, s, images, batch, logits);
}

elasto_status elasto_forward_host(elasto_t h, void* stream, const void* images_host, int batch,
                                  float* logits_host) {
  if (!h || !images_host || !logits_host) {
    set_error("elasto_forward_host: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (batch < 1 || batch > h->d.max_batch) {
    set_error("elasto_forward_host: batch outside [1, max_batch]");
    return ELASTO_ERR_INVALID_ARG;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void* img_dev = h->cnn ? cnn_image_stage(h->cnn) : h->img_stage;
  float* logit_dev = h->cnn ? cnn_logit_stage(h->cnn) : h->logit_stage;
  const size_t ib = size_t(batch) * h->d.img_h * h->d.img_w * h->d.img_c * dtype_size(h->d.weight_dtype);
  ELASTO_CUDA_TRY(cudaMemcpyAsync(img_dev, images_host, ib, cudaMemcpyHostToDevice, s));
  elasto_status st = elasto_forward(h, stream, img_dev, batch, logit_dev);
  if (st != ELASTO_OK) return st;
  ELASTO_CUDA_TRY(cudaMemcpyAsync(logits_host, logit_dev, size_t(batch) * h->d.classes * 4, cudaMemcpyDeviceToHost, s));
  ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
  return ELASTO_OK;
}

elasto_status elasto_forward_host_batches(elasto_t h, void* stream, int n_batches, int batch,
                                          const void* const* images_host, float* const* logits_host) {
  if (!h || !images_host || !logits_host || n_batches < 1) {
    set_error("elasto_forward_host_batches: null argument or n_batches < 1");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (batch < 1 || batch > h->d.max_batch) {
    set_error("elasto_forward_host_batches: batch outside [1, max_batch]");
    return ELASTO_ERR_INVALID_ARG;
  }
  for (int i = 0; i < n_batches; ++i)
    if (!images_host[i] || !logits_host[i]) {
      set_error("elasto_forward_host_batches: null buffer for batch " + std::to_string(i));
      return ELASTO_ERR_INVALID_ARG;
    }
  const size_t img_cap = size_t(h->d.max_batch) * h->d.img_h * h->d.img_w * h->d.img_c * dtype_size(h->d.weight_dtype);
  const size_t logit_cap = size_t(h->d.max_batch) * h->d.classes * 4;
  if (!h->stage2) {  // first call: the second staging pair, streams and events
    cudaError_t e = cudaMalloc(&h->stage2, img_cap + 256 + logit_cap);
    if (e != cudaSuccess) {
      h->stage2 = nullptr;
      cudaGetLastError();
      set_error("elasto_forward_host_batches: cudaMalloc of the second staging pair failed");
      return ELASTO_ERR_OOM;
    }
    ELASTO_CUDA_TRY(cudaStreamCreateWithFlags(&h->h2d, cudaStreamNonBlocking));
    ELASTO_CUDA_TRY(cudaStreamCreateWithFlags(&h->d2h, cudaStreamNonBlocking));
    for (int k = 0; k < 2; ++k) {
      ELASTO_CUDA_TRY(cudaEventCreateWithFlags(&h->ev_h2d[k], cudaEventDisableTiming));
      ELASTO_CUDA_TRY(cudaEventCreateWithFlags(&h->ev_fwd[k], cudaEventDisableTiming));
      ELASTO_CUDA_TRY(cudaEventCreateWithFlags(&h->ev_d2h[k], cudaEventDisableTiming));
    }
  }
  void* img[2] = {h->cnn ? cnn_image_stage(h->cnn) : h->img_stage, h->stage2};
  float* lg[2] = {h->cnn ? cnn_logit_stage(h->cnn) : h->logit_stage,
                  reinterpret_cast<float*>(h->stage2 + (img_cap + 255) / 256 * 256)};
  const size_t ib = size_t(batch) * h->d.img_h * h->d.img_w * h->d.img_c * dtype_size(h->d.weight_dtype);
  const size_t lb = size_t(batch) * h->d.classes * 4;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the copy streams start after the work already on `stream` (which may
  // still be using the staging buffers)
  ELASTO_CUDA_TRY(cudaEventRecord(h->ev_fwd[0], s));
  ELASTO_CUDA_TRY(cudaEventRecord(h->ev_fwd[1], s));
  ELASTO_CUDA_TRY(cudaEventRecord(h->ev_d2h[0], s));
  ELASTO_CUDA_TRY(cudaEventRecord(h->ev_d2h[1], s));
  // batch 0's images
  ELASTO_CUDA_TRY(cudaStreamWaitEvent(h->h2d, h->ev_fwd[0], 0));
  ELASTO_CUDA_TRY(cudaMemcpyAsync(img[0], images_host[0], ib, cudaMemcpyHostToDevice, h->h2d));
  ELASTO_CUDA_TRY(cudaEventRecord(h->ev_h2d[0], h->h2d));
  for (int i = 0; i < n_batches; ++i) {
    const int cb = i & 1, nb = cb ^ 1;
    if (i + 1 < n_batches) {
      // batch i+1's images into the other staging buffer once the forward
      // that last read it (batch i-1) is done
      ELASTO_CUDA_TRY(cudaStreamWaitEvent(h->h2d, h->ev_fwd[nb], 0));
      ELASTO_CUDA_TRY(cudaMemcpyAsync(img[nb], images_host[i + 1], ib, cudaMemcpyHostToDevice, h->h2d));
      ELASTO_CUDA_TRY(cudaEventRecord(h->ev_h2d[nb], h->h2d));
    }
    // batch i: its images are in, and batch i-2's logits have left lg[cb]
    ELASTO_CUDA_TRY(cudaStreamWaitEvent(s, h->ev_h2d[cb], 0));
    ELASTO_CUDA_TRY(cudaStreamWaitEvent(s, h->ev_d2h[cb], 0));
    const elasto_status st = elasto_forward(h, stream, img[cb], batch, lg[cb]);
    if (st != ELASTO_OK) return st;
    ELASTO_CUDA_TRY(cudaEventRecord(h->ev_fwd[cb], s));
    ELASTO_CUDA_TRY(cudaStreamWaitEvent(h->d2h, h->ev_fwd[cb], 0));
    ELASTO_CUDA_TRY(cudaMemcpyAsync(logits_host[i], lg[cb], lb, cudaMemcpyDeviceToHost, h->d2h));
    ELASTO_CUDA_TRY(cudaEventRecord(h->ev_d2h[cb], h->d2h));
  }
  ELASTO_CUDA_TRY(cudaStreamSynchronize(h->d2h));
  ELASTO_CUDA_TRY(cudaStreamSynchronize(s));
  return ELASTO_OK;
}

elasto_status elasto_sync_status(elasto_t h, void* stream) {
  if (!h) {
    set_error("elasto_sync_status: null handle");
    return ELASTO_ERR_INVALID_ARG;
  }
  ELASTO_CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int* sw = h->cnn ? cnn_status_word(h->cnn) : h->status;
  int v = 0;
  ELASTO_CUDA_TRY(cudaMemcpy(&v, sw, sizeof v, cudaMemcpyDeviceToHost));
  if (v != 0) {
    ELASTO_CUDA_TRY(cudaMemset(sw, 0, sizeof v));
    set_error("device status word: a bounded device-side wait gave up");
    return static_cast<elasto_status>(v);
  }
  return ELASTO_OK;
}

elasto_status elasto_destroy(elasto_t h) {
  if (!h) {
    set_error("elasto_destroy: null handle");
    return ELASTO_ERR_INVALID_ARG;
  }
  cudaDeviceSynchronize();
  if (h->arena) cudaFree(h->arena);
  if (h->cnn) cnn_destroy(h->cnn);
  noalloc_cache_free(h->noalloc);
  pk_free(h->pk);
  if (h->stage2) cudaFree(h->stage2);
  if (h->h2d) cudaStreamDestroy(h->h2d);
  if (h->d2h) cudaStreamDestroy(h->d2h);
  for (int k = 0; k < 2; ++k) {
    if (h->ev_h2d[k]) cudaEventDestroy(h->ev_h2d[k]);
    if (h->ev_fwd[k]) cudaEventDestroy(h->ev_fwd[k]);
    if (h->ev_d2h[k]) cudaEventDestroy(h->ev_d2h[k]);
  }
  h->guards.release();
  h->prof.release();
  delete h;
  return ELASTO_OK;
}

const char* elasto_last_error(void) { return last_error_cstr(); }

elasto_status elasto_check_guards(elasto_t h, void* stream, int* n_bad) {
  if (!h) {
    set_error("elasto_check_guards: null handle");
    return ELASTO_ERR_INVALID_ARG;
  }
  char* base = h->arena;
  GuardedArena* g = &h->guards;
  if (h->cnn) g = cnn_guards(h->cnn, &base);
  std::string first;
  const int bad = g->check(base, static_cast<cudaStream_t>(stream), &first);
  if (n_bad) *n_bad = bad > 0 ? bad : 0;
  if (bad < 0) {
    set_error("elasto_check_guards: CUDA error while checking: " + std::string(cudaGetErrorString(cudaGetLastError())));
    return ELASTO_ERR_CUDA;
  }
  if (bad > 0) {
    set_error("elasto_check_guards: " + std::to_string(bad) + " guard zone(s) overwritten; first after " + first);
    return ELASTO_ERR_GUARD;
  }
  return ELASTO_OK;
}

elasto_status elasto_debug_damage_guard(elasto_t h, int zone) {
  if (!h) {
    set_error("elasto_debug_damage_guard: null handle");
    return ELASTO_ERR_INVALID_ARG;
  }
  char* base = h->arena;
  GuardedArena* g = &h->guards;
  if (h->cnn) g = cnn_guards(h->cnn, &base);
  if (zone < 0 || zone >= static_cast<int>(g->zones.size()) || !base) {
    set_error("elasto_debug_damage_guard: zone out of range");
    return ELASTO_ERR_INVALID_ARG;
  }
  ELASTO_CUDA_TRY(cudaDeviceSynchronize());
  ELASTO_CUDA_TRY(cudaMemset(base + g->zones[zone].off, 0x5A, 1));
  ELASTO_CUDA_TRY(cudaDeviceSynchronize());
  return ELASTO_OK;
}

elasto_status elasto_query(elasto_t h, int what, int mode, int64_t* value) {
  if (!h || !value) {
    set_error("elasto_query: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (h->cnn) return cnn_query(h->cnn, what, mode, value);
  const int nm = static_cast<int>(h->modes.size());
  const bool needs_mode = what == ELASTO_Q_PACKED_BYTES || what == ELASTO_Q_MODE_MACS || what == ELASTO_Q_LAUNCHES ||
                          what == ELASTO_Q_ONE_LAUNCH;
  if (needs_mode && (mode < 0 || mode >= nm)) {
    set_error("elasto_query: bad mode");
    return ELASTO_ERR_BAD_MODE;
  }
  switch (what) {
    case ELASTO_Q_N_MODES: *value = nm; break;
    case ELASTO_Q_PACKED_BYTES: *value = int64_t(h->modes[mode].packed_bytes); break;
    case ELASTO_Q_SHARED_BYTES: *value = int64_t(h->shared_bytes); break;
    case ELASTO_Q_WORKSPACE_BYTES: *value = int64_t(h->workspace_bytes); break;
    case ELASTO_Q_ARENA_BYTES: *value = int64_t(h->arena_bytes); break;
    case ELASTO_Q_MODE_MACS: *value = h->modes[mode].macs; break;
    case ELASTO_Q_LAUNCHES: *value = h->modes[mode].launches; break;
    case ELASTO_Q_PACKED_TOTAL: *value = int64_t(h->packed_total); break;
    case ELASTO_Q_PREFIX_SHARED: *value = h->prefix_shared ? 1 : 0; break;
    case ELASTO_Q_GUARD_ZONES: *value = int64_t(h->guards.zones.size()); break;
    case ELASTO_Q_ONE_LAUNCH: *value = pk_ready(h->pk, mode) ? 1 : 0; break;
    default: set_error("elasto_query: unknown query"); return ELASTO_ERR_INVALID_ARG;
  }
  return ELASTO_OK;
}

elasto_status elasto_set_one_launch(elasto_t h, int enable) {
  if (!h) {
    set_error("elasto_set_one_launch: null handle");
    return ELASTO_ERR_INVALID_ARG;
  }
  pk_enable(h->pk, enable != 0);  // ResNet-50 handles have no plan: nothing changes
  return ELASTO_OK;
}

elasto_status elasto_profile_enable(elasto_t h, int enable) {
  if (!h) {
    set_error("elasto_profile_enable: null handle");
    return ELASTO_ERR_INVALID_ARG;
  }
  Profiler& p = h->cnn ? *cnn_profiler(h->cnn) : h->prof;
  ELASTO_CUDA_TRY(p.enable(enable != 0));
  return ELASTO_OK;
}

elasto_status elasto_profile_read(elasto_t h, elasto_launch_record* out, int capacity, int* count) {
  if (!h || !out || !count || capacity < 0) {
    set_error("elasto_profile_read: invalid arguments");
    return ELASTO_ERR_INVALID_ARG;
  }
  Profiler& p = h->cnn ? *cnn_profiler(h->cnn) : h->prof;
  return p.read(out, capacity, count);
}

elasto_status elasto_profile_dns(elasto_t h, void* stream, int batch, int trials, elasto_dn_profile* out) {
  if (!h || !out || trials < 1) {
    set_error("elasto_profile_dns: null argument or trials < 1");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (batch < 1 || batch > h->d.max_batch) {
    set_error("elasto_profile_dns: batch outside [1, max_batch]");
    return ELASTO_ERR_INVALID_ARG;
  }
  const int nm = h->cnn ? cnn_n_modes(h->cnn) : static_cast<int>(h->modes.size());
  const int saved = h->cur.load(std::memory_order_acquire);
  void* img = h->cnn ? cnn_image_stage(h->cnn) : h->img_stage;
  float* logits = h->cnn ? cnn_logit_stage(h->cnn) : h->logit_stage;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  ELASTO_CUDA_TRY(cudaEventCreate(&e0));
  cudaError_t ce = cudaEventCreate(&e1);
  if (ce != cudaSuccess) {
    cudaEventDestroy(e0);
    return cuda_fail(ce, "cudaEventCreate");
  }
  elasto_status st = ELASTO_OK;
  std::vector<float> ts(trials);
  for (int m = 0; m < nm && st == ELASTO_OK; ++m) {
    h->cur.store(m, std::memory_order_release);
    for (int i = 0; i < 3 && st == ELASTO_OK; ++i) st = elasto_forward(h, stream, img, batch, logits);
    for (int i = 0; i < trials && st == ELASTO_OK; ++i) {
      if ((ce = cudaEventRecord(e0, s)) != cudaSuccess) break;
      st = elasto_forward(h, stream, img, batch, logits);
      if (st != ELASTO_OK || (ce = cudaEventRecord(e1, s)) != cudaSuccess || (ce = cudaEventSynchronize(e1)) != cudaSuccess ||
          (ce = cudaEventElapsedTime(&ts[i], e0, e1)) != cudaSuccess)
        break;
    }
    if (st == ELASTO_OK && ce != cudaSuccess) st = cuda_fail(ce, "elasto_profile_dns: timing");
    if (st != ELASTO_OK) break;
    std::vector<float> sorted = ts;
    std::sort(sorted.begin(), sorted.end());
    int64_t packed = 0, shared = 0, macs = 0;
    elasto_query(h, ELASTO_Q_PACKED_BYTES, m, &packed);
    elasto_query(h, ELASTO_Q_SHARED_BYTES, m, &shared);
    elasto_query(h, ELASTO_Q_MODE_MACS, m, &macs);
    out[m].latency_ms = sorted[trials / 2];
    out[m].memory_bytes = double(packed + shared);
    out[m].gflops = 2.0 * double(macs) * batch / 1e9;
    out[m].accuracy = std::numeric_limits<float>::quiet_NaN();
  }
  h->cur.store(saved, std::memory_order_release);
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  return st;
}

elasto_status elasto_select_dn(const elasto_dn_profile* lut, int n, float max_latency_ms, double max_memory_bytes,
                               float min_accuracy, int* mode) {
  if (!lut || !mode || n <= 0) {
    set_error("elasto_select_dn: null argument or empty table");
    return ELASTO_ERR_INVALID_ARG;
  }
  int best = -1;
  for (int i = 0; i < n; ++i) {
    const elasto_dn_profile& e = lut[i];
    if (!std::isnan(max_latency_ms) && !(e.latency_ms <= max_latency_ms)) continue;
    if (!std::isnan(max_memory_bytes) && !(e.memory_bytes <= max_memory_bytes)) continue;
    if (!std::isnan(min_accuracy) && !(e.accuracy >= min_accuracy)) continue;  // NaN accuracy fails
    if (best < 0 || e.gflops < lut[best].gflops ||
        (e.gflops == lut[best].gflops && e.latency_ms < lut[best].latency_ms))
      best = i;
  }
  if (best < 0) {
    set_error("elasto_select_dn: no descendant network satisfies the constraints");
    return ELASTO_ERR_BAD_MODE;
  }
  *mode = best;
  return ELASTO_OK;
}

elasto_status elasto_debug_export_packed(elasto_t h, int mode, int layer, int which, void* host_dst, size_t bytes) {
  if (!h || !host_dst) {
    set_error("elasto_debug_export_packed: null argument");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (h->cnn) return cnn_export_packed(h->cnn, mode, layer, which, host_dst, bytes);
  if (mode < 0 || mode >= static_cast<int>(h->modes.size())) {
    set_error("elasto_debug_export_packed: bad mode");
    return ELASTO_ERR_BAD_MODE;
  }
  if (layer < 0 || layer >= h->d.layers || which < 0 || which > 5) {
    set_error("elasto_debug_export_packed: bad layer or buffer index");
    return ELASTO_ERR_INVALID_ARG;
  }
  const VitLayerPack& lp = h->modes[mode].layers[layer];
  const VitEmbed& em = h->modes[mode].emb;
  const size_t D = em.d, Dm = em.d_pad;  // kept embedding width; stored rows have Dm entries
  size_t need = 0;
  const void* src = nullptr;
  switch (which) {
    case 0: need = size_t(3) * lp.w * D * 2; src = lp.qkv_w; break;
    case 1: need = size_t(3) * lp.w * 4; src = lp.qkv_b; break;
    case 2: need = D * lp.w * 2; src = lp.proj_w; break;
    case 3: need = size_t(lp.f) * D * 2; src = lp.fc1_w; break;
    case 4: need = size_t(lp.f) * 4; src = lp.fc1_b; break;
    case 5: need = D * lp.f * 2; src = lp.fc2_w; break;
  }
  if (bytes != need) {
    set_error("elasto_debug_export_packed: expected " + std::to_string(need) + " bytes");
    return ELASTO_ERR_INVALID_ARG;
  }
  if (need == 0) return ELASTO_OK;
  if (h->prefix_shared) {
    // The mode's heads / channels are the first k entries of the layer's
    // prefix order; the export lists them ascending (and q | k | v blocks
    // apart), so copy the prefix and permute on the host (exact).
    const bool heads = which <= 2;
    const std::vector<int32_t>& perm = heads ? h->perm_h[layer] : h->perm_f[layer];
    const int k = heads ? lp.w / 64 : lp.f;
    std::vector<int> pos(k);  // pos[q] = prefix position of the q-th smallest kept index
    for (int i = 0; i < k; ++i) pos[i] = i;
    std::sort(pos.begin(), pos.end(), [&](int a, int b) { return perm[a] < perm[b]; });
    const size_t es = (which == 1 || which == 4) ? 4 : 2;
    std::vector<char> tmp;
    char* out = static_cast<char*>(host_dst);
    if (which == 0 || which == 1) {  // rows (or entries) p * 192 + blk * 64 + r -> (blk * k + q) * 64 + r
      const size_t row = which == 0 ? D * 2 : 4;
      tmp.resize(size_t(3) * lp.w * row);
      ELASTO_CUDA_TRY(cudaMemcpy(tmp.data(), src, tmp.size(), cudaMemcpyDeviceToHost));
      for (int blk = 0; blk < 3; ++blk)
        for (int q = 0; q < k; ++q)
          memcpy(out + (size_t(blk) * k + q) * 64 * row, tmp.data() + (size_t(pos[q]) * 3 + blk) * 64 * row, 64 * row);
    } else if (which == 2 || which == 5) {  // [D, ld] columns of the prefix -> [D, k * width]
      const int width = which == 2 ? 64 : 1, ld = which == 2 ? lp.ld_proj : lp.ld_fc2;
      tmp.resize(D * size_t(ld) * es);
      ELASTO_CUDA_TRY(cudaMemcpy(tmp.data(), src, tmp.size(), cudaMemcpyDeviceToHost));
      for (size_t r = 0; r < D; ++r)
        for (int q = 0; q < k; ++q)
          memcpy(out + (r * k + q) * width * es, tmp.data() + (r * ld + size_t(pos[q]) * width) * es, width * es);
    } else {  // which 3 / 4: rows (or entries) of FC1 in prefix order
      const size_t row = which == 3 ? D * 2 : 4;
      tmp.resize(size_t(k) * row);
      ELASTO_CUDA_TRY(cudaMemcpy(tmp.data(), src, tmp.size(), cudaMemcpyDeviceToHost));
      for (int q = 0; q < k; ++q) memcpy(out + size_t(q) * row, tmp.data() + size_t(pos[q]) * row, row);
    }
    return ELASTO_OK;
  }
  if (which == 5) {
    // stored [d_pad, f_pad]; export [d, f]
    ELASTO_CUDA_TRY(cudaMemcpy2D(host_dst, size_t(lp.f) * 2, src, size_t(lp.f_pad) * 2, size_t(lp.f) * 2, D,
                                 cudaMemcpyDeviceToHost));
  } else if (which == 0 || which == 3) {
    // stored [rows, d_pad]; export [rows, d]
    const size_t rows = which == 0 ? size_t(3) * lp.w : size_t(lp.f);
    ELASTO_CUDA_TRY(cudaMemcpy2D(host_dst, D * 2, src, Dm * 2, D * 2, rows, cudaMemcpyDeviceToHost));
  } else {
    ELASTO_CUDA_TRY(cudaMemcpy(host_dst, src, need, cudaMemcpyDeviceToHost));
  }
  return ELASTO_OK;
}

}  // extern "C"
