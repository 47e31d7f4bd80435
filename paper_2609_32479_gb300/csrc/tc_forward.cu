// tcgen05 path placeholder (filled in by the fused kernel).
#include "trackfit_internal.h"

bool tf_tc_supported(const tf_shape&) { return false; }
int tf_tc_create(trackfit_ctx*, const float*) { return TRACKFIT_ERR_UNSUPPORTED; }
void tf_tc_destroy(trackfit_ctx*) {}
int tf_tc_forward(trackfit_ctx*, const float*, const int32_t*, int64_t, float*, float*, float*, cudaStream_t) {
  return TRACKFIT_ERR_UNSUPPORTED;
}
