// Internal interface between the C-ABI layer and the ResNet-50 (CNN) path.
#pragma once
#include "common.h"

namespace elasto {

// Records an event pair around each launch of a forward while enabled.
struct Profiler {
  static constexpr int kSlots = 1024;
  bool on = false;
  cudaEvent_t ev[2 * kSlots] = {};
  elasto_launch_record rec[kSlots] = {};
  int count = 0;
  bool overflow = false;
  cudaError_t enable(bool e);
  void begin() {
    count = 0;
    overflow = false;
  }
  // Call before/after one launch on stream s.
  cudaError_t before(cudaStream_t s);
  cudaError_t after(cudaStream_t s, const elasto_launch_record& r);
  elasto_status read(elasto_launch_record* out, int capacity, int* n);
  void release();
};

struct CnnModel;  // defined in cnn.cu

// Host-side validation of descriptor, weights and tables (no CUDA calls).
elasto_status cnn_check_inputs(const elasto_model_desc* d, const elasto_weights* w, const elasto_mode_tables* modes,
                               int n_modes);
CnnModel* cnn_new();
elasto_status cnn_create(const elasto_model_desc* d, const elasto_weights* w, const elasto_mode_tables* modes,
                         int n_modes, CnnModel* m);
elasto_status cnn_forward(CnnModel* m, int mode, cudaStream_t s, const void* images, int batch, float* logits);
int cnn_n_modes(const CnnModel* m);
void* cnn_image_stage(CnnModel* m);
float* cnn_logit_stage(CnnModel* m);
int* cnn_status_word(CnnModel* m);
Profiler* cnn_profiler(CnnModel* m);
void cnn_destroy(CnnModel* m);  // frees the model and its device memory
elasto_status cnn_query(CnnModel* m, int what, int mode, int64_t* value);
elasto_status cnn_export_packed(CnnModel* m, int mode, int block, int which, void* host_dst, size_t bytes);

struct GuardedArena;  // guard.h
GuardedArena* cnn_guards(CnnModel* m, char** base);  // the CNN arena's guard zones and base

cudaError_t ensure_kernel_attributes();
elasto_status check_device();

}  // namespace elasto
