// Layout of an elastic-model handle (shared by the C-ABI translation units).
#pragma once
#include <atomic>
#include <vector>

#include "common.h"
#include "elasto_internal.h"
#include "guard.h"

namespace elasto {

// One layer of one mode: kept widths, packed weights, launch plans.
struct VitLayerPack {
  int w = 0;       // kept heads * 64
  int f = 0;       // kept MLP channels
  int f_pad = 0;   // f, or f rounded up to 64 in a per-mode pack (zero rows/cols; GELU(0) = 0)
  int ld_proj = 0; // row stride of proj_w (w, or 64 x heads of the shared copy)
  int ld_fc2 = 0;  // row stride of fc2_w (f_pad, or the shared copy's channels)
  bf16* qkv_w = nullptr;
  float* qkv_b = nullptr;
  bf16* proj_w = nullptr;
  bf16* fc1_w = nullptr;
  float* fc1_b = nullptr;
  bf16* fc2_w = nullptr;
  // low bf16 planes (fp32-stored models only; W = hi + lo)
  bf16 *qkv_w_lo = nullptr, *proj_w_lo = nullptr, *fc1_w_lo = nullptr, *fc2_w_lo = nullptr;
  GemmPlanSet qkv, proj, fc1, fc2;  // one plan per batch bucket
  AttnPlan attn;
};

// The parameters that carry the embedding width. A mode that keeps every
// channel points at the handle's copies; an embedding-pruned mode (Section
// 4.1) has its own, holding the kept channels E first and zero padding up to
// d_pad (a multiple of 64), so the residual stream X is [rows, d_pad] with
// zeros past d.
struct VitEmbed {
  int d = 0, d_pad = 0;  // kept channels, padded width
  bool pruned = false;
  bf16 *patch_w = nullptr, *patch_w_lo = nullptr;  // [d_pad, P*P*C]
  float *patch_b = nullptr, *cls = nullptr, *pos = nullptr;  // [d_pad], [d_pad], [n, d_pad]
  std::vector<float*> ln1_w, ln1_b, ln2_w, ln2_b, proj_b, fc2_b;  // per layer, [d_pad]
  float *norm_w = nullptr, *norm_b = nullptr, *head_w = nullptr;  // [d_pad], [d_pad], [C, d_pad]
  float* addend = nullptr;  // per-token addend of the patch projection, [k * n, d_pad] (see elasto_s::tok_addend)
  GemmPlanSet patch;        // pruned modes: the patch projection at width d_pad
};

// Launch plans of elasto_forward_noalloc (csrc/noalloc.cu), cached per
// (mode, batch); host memory only.
struct NoallocCache;
void noalloc_cache_free(NoallocCache* c);

// One-launch plans of the one-image forward (csrc/persistent.cu), one per
// mode; device memory of their own.
struct PkPlan;
void pk_free(PkPlan* p);

struct VitMode {
  std::vector<VitLayerPack> layers;
  VitEmbed emb;
  size_t packed_bytes = 0;  // bytes of packed weights this mode reads
  int64_t macs = 0;
  int launches = 0;
};

}  // namespace elasto

struct elasto_s {
  elasto_model_desc d{};
  int dev = 0;
  int n = 0, np = 0, kpe = 0;
  char* arena = nullptr;
  elasto::GuardedArena guards;  // guard zone after every arena buffer
  size_t arena_bytes = 0, shared_bytes = 0, workspace_bytes = 0;
  // shared (mode-independent) parameters
  elasto::bf16* patch_w = nullptr;
  elasto::bf16* patch_w_lo = nullptr;  // low plane for fp32-stored models
  float *patch_b = nullptr, *cls = nullptr, *pos = nullptr, *norm_w = nullptr, *norm_b = nullptr;
  float *head_w = nullptr, *head_b = nullptr;
  std::vector<float*> ln1_w, ln1_b, proj_b, ln2_w, ln2_b, fc2_b;
  // workspace
  float* X = nullptr;
  float* splitk_part = nullptr;  // split-K partial sums of the one-image FC2
  elasto::bf16 *Y = nullptr, *QKV = nullptr, *O = nullptr, *H = nullptr, *P = nullptr;
  // Per-token addend of the patch projection (cls + pos[0] on class tokens,
  // pos[t] + b_pe on patch tokens) for k = 1 + ceil(128 / n) images: it is
  // the same for every image, and the patch GEMM reads row r mod n of it.
  float* tok_addend = nullptr;  // [k * n, d]
  int addend_rows = 0;          // k * n
  void* img_stage = nullptr;
  float* logit_stage = nullptr;
  int* status = nullptr;
  elasto::GemmPlanSet patch;
  int plan_rows[elasto::GemmPlanSet::kMax] = {};  // the row counts the plan variants are made for
  int n_plan_rows = 0;
  std::vector<elasto::VitMode> modes;
  // Prefix sharing (nested kept sets, Eq. 8): one packed copy per layer with
  // heads and MLP channels ordered "kept by the smallest mode first"; every
  // mode uses a prefix of it. perm_h[l] / perm_f[l] give that order.
  bool prefix_shared = false;
  std::vector<std::vector<int32_t>> perm_h, perm_f;
  size_t packed_total = 0;  // device bytes of all modes' packed weights
  std::atomic<int> cur{0};
  // elasto_forward_host_batches: a second device staging pair (images, then
  // logits) and the copy streams / events, made by its first call
  char* stage2 = nullptr;
  cudaStream_t h2d = nullptr, d2h = nullptr;
  cudaEvent_t ev_h2d[2] = {}, ev_fwd[2] = {}, ev_d2h[2] = {};
  elasto::NoallocCache* noalloc = nullptr;  // built by the first elasto_forward_noalloc call
  elasto::PkPlan* pk = nullptr;             // one-launch plans of the one-image forward (null: none)
  unsigned* pk_sync = nullptr;              // their grid-barrier counter and abort flag
  float* pk_y32 = nullptr;                  // their final-norm class-token row [d]
  // CNN state lives behind this pointer (null for ViT)
  elasto::CnnModel* cnn = nullptr;
  elasto::Profiler prof;
};

namespace elasto {

// csrc/persistent.cu. pk_build makes every mode's plan it can (a mode without
// one keeps the kernel-by-kernel forward) and leaves *out null when the
// device cannot run cooperative launches of the kernel.
cudaError_t pk_init_attributes();
size_t pk_workspace_floats(int d);  // floats of the class-token row buffer for width d
elasto_status pk_build(elasto_s* h, unsigned* sync, float* y32, PkPlan** out);
bool pk_ready(const PkPlan* p, int mode);
void pk_enable(PkPlan* p, bool on);
cudaError_t pk_launch(const PkPlan* p, int mode, int n, const void* images, float* logits, int* status,
                      cudaStream_t s);
// Self-test of the one-launch forward's grid barrier (elasto_op_grid_barrier).
cudaError_t pk_barrier_selftest(cudaStream_t s, int unreachable, unsigned* sync, int* status,
                                unsigned long long* elapsed_ns);

}  // namespace elasto
