// Prefill GEMM entry points (tensor-core kernel lands here).
#include <cuda_runtime.h>

#include "polyq.h"
#include "polyq_internal.h"

extern "C" int polyq_gemm_workspace_bytes(const polyq_dev_layer* L, int64_t M, size_t* bytes) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_gemm_workspace_bytes");
  if (rc) return rc;
  (void)M;
  (void)bytes;
  return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_gemm_workspace_bytes: GEMM not built yet");
}

extern "C" int polyq_linear_gemm(const polyq_dev_layer* L, const void* X, int64_t M, float* Y,
                                 void* workspace, size_t ws_bytes, void* stream) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_linear_gemm");
  if (rc) return rc;
  (void)X; (void)M; (void)Y; (void)workspace; (void)ws_bytes; (void)stream;
  return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_linear_gemm: GEMM not built yet");
}
