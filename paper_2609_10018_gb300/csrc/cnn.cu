// ResNet-50 descendant networks (Eq. 7): placeholder until the implicit-GEMM
// convolution path lands; elasto_create reports ELASTO_ERR_UNSUPPORTED.
#include "elasto_internal.h"

namespace elasto {

struct CnnModel {
  int n_modes = 0;
  Profiler prof;
};

elasto_status cnn_check_inputs(const elasto_model_desc*, const elasto_weights*, const elasto_mode_tables*, int) {
  set_error("elasto_create: the ResNet-50 path is not available in this build");
  return ELASTO_ERR_UNSUPPORTED;
}
CnnModel* cnn_new() { return new CnnModel(); }
elasto_status cnn_create(const elasto_model_desc*, const elasto_weights*, const elasto_mode_tables*, int,
                         CnnModel*) {
  set_error("elasto_create: the ResNet-50 path is not available in this build");
  return ELASTO_ERR_UNSUPPORTED;
}
elasto_status cnn_forward(CnnModel*, int, cudaStream_t, const void*, int, float*) { return ELASTO_ERR_UNSUPPORTED; }
int cnn_n_modes(const CnnModel* m) { return m->n_modes; }
void* cnn_image_stage(CnnModel*) { return nullptr; }
float* cnn_logit_stage(CnnModel*) { return nullptr; }
int* cnn_status_word(CnnModel*) { return nullptr; }
Profiler* cnn_profiler(CnnModel* m) { return &m->prof; }
void cnn_destroy(CnnModel* m) {
  m->prof.release();
  delete m;
}
elasto_status cnn_query(CnnModel*, int, int, int64_t*) { return ELASTO_ERR_UNSUPPORTED; }
elasto_status cnn_export_packed(CnnModel*, int, int, int, void*, size_t) { return ELASTO_ERR_UNSUPPORTED; }

}  // namespace elasto
