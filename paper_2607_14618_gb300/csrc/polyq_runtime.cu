// Host runtime helpers: device properties and a cache of TMA tensor maps.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstring>
#include <map>
#include <mutex>
#include <tuple>

#include "polyq_dev.cuh"
#include "polyq_internal.h"

namespace {

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                              const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                              const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

std::mutex g_mu;
EncodeFn g_encode = nullptr;
std::map<int, int> g_sms;
using Key = std::tuple<uintptr_t, int, uint64_t, uint64_t, uint64_t, uint32_t, uint32_t, int>;
std::map<Key, CUtensorMap> g_maps;

int get_encode(EncodeFn* fn) {
  if (!g_encode) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                                     cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !p)
      return polyq_set_error(POLYQ_ECUDA, "cuTensorMapEncodeTiled unavailable: %s",
                             cudaGetErrorString(e));
    g_encode = (EncodeFn)p;
  }
  *fn = g_encode;
  return POLYQ_OK;
}

}  // namespace

int polyq_sm_count(int* out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return polyq_set_error(POLYQ_ECUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_sms.find(dev);
  if (it == g_sms.end()) {
    int n = 0;
    e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess || n <= 0)
      return polyq_set_error(POLYQ_ECUDA, "SM count: %s", cudaGetErrorString(e));
    it = g_sms.emplace(dev, n).first;
  }
  *out = it->second;
  return POLYQ_OK;
}

int polyq_tensor_map_2d(CUtensorMap* out, const void* base, int elem_bytes, uint64_t cols,
                        uint64_t rows, uint64_t row_stride_bytes, uint32_t box_cols,
                        uint32_t box_rows, int swizzle_bytes) {
  Key k{(uintptr_t)base, elem_bytes, cols, rows, row_stride_bytes, box_cols, box_rows, swizzle_bytes};
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_maps.find(k);
  if (it != g_maps.end()) {
    *out = it->second;
    return POLYQ_OK;
  }
  EncodeFn enc;
  int rc = get_encode(&enc);
  if (rc) return rc;
  CUtensorMapDataType dt = elem_bytes == 1   ? CU_TENSOR_MAP_DATA_TYPE_UINT8
                           : elem_bytes == 2 ? CU_TENSOR_MAP_DATA_TYPE_UINT16
                                             : CU_TENSOR_MAP_DATA_TYPE_UINT32;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUtensorMap m;
  std::memset(&m, 0, sizeof m);
  CUresult r = enc(&m, dt, 2, const_cast<void*>(base), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE,
                   swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                   : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                         : CU_TENSOR_MAP_SWIZZLE_NONE,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return polyq_set_error(POLYQ_ECUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  if (g_maps.size() > 4096) g_maps.clear();
  g_maps.emplace(k, m);
  *out = m;
  return POLYQ_OK;
}

extern "C" int polyq_workspace_status(const void* workspace, int* status, void* stream) {
  polyq_clear_error();
  if (!workspace || !status)
    return polyq_set_error(POLYQ_EINVAL, "polyq_workspace_status: NULL argument");
  cudaStream_t st = (cudaStream_t)stream;
  int v = 0;
  cudaError_t e = cudaMemcpyAsync(&v, workspace, sizeof v, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_workspace_status: %s", cudaGetErrorString(e));
  *status = v;
  if (v == 0) return POLYQ_OK;
  static const char* what[] = {"?", "a consumer's wait for a stage's data",
                               "a producer's wait for a free stage",
                               "a chained launch's grid barrier",
                               "a chained launch's wait for a phase's records"};
  return polyq_set_error(POLYQ_ETIMEOUT, "a bounded device wait gave up: %s (status %d)",
                         what[(v >= 1 && v <= 4) ? v : 0], v);
}
