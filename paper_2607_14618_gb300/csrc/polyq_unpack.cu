// Unpack kernel (test aid): reads every code of the packed layer with plain
// per-element bit arithmetic, independent of the GEMV/GEMM decoders.
#include <cuda_runtime.h>

#include "polyq.h"
#include "polyq_internal.h"

namespace {

__global__ void unpack_codes_kernel(polyq_dev_layer L, uint16_t* __restrict__ codes) {
  const int64_t total = L.N * L.K;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t n = i / L.K;
    const int32_t p = (int32_t)(i - n * L.K);
    int bi = 0;
    while (bi + 1 < L.n_blocks && p >= L.blocks[bi + 1].pos0) ++bi;
    const polyq_block& B = L.blocks[bi];
    const uint8_t* seg = L.packed + n * L.row_stride + B.seg_off;
    const int32_t j = p - B.pos0;
    uint32_t v;
    if (B.bits == 16) {
      v = (uint32_t)seg[2 * j] | ((uint32_t)seg[2 * j + 1] << 8);
    } else {
      const int64_t bit = (int64_t)j * B.bits;
      const int64_t byte = bit >> 3;
      const int sh = (int)(bit & 7);
      uint32_t w = seg[byte];
      if (sh + B.bits > 8) w |= (uint32_t)seg[byte + 1] << 8;
      v = (w >> sh) & ((1u << B.bits) - 1u);
    }
    codes[i] = (uint16_t)v;
  }
}

}  // namespace

extern "C" int polyq_unpack_codes(const polyq_dev_layer* L, uint16_t* codes, void* stream) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_unpack_codes");
  if (rc) return rc;
  if (!codes) return polyq_set_error(POLYQ_EINVAL, "polyq_unpack_codes: codes is NULL");
  const int64_t total = L->N * L->K;
  int grid = (int)std::min<int64_t>((total + 255) / 256, 152 * 16);
  unpack_codes_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>(*L, codes);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_unpack_codes: %s", cudaGetErrorString(e));
  return POLYQ_OK;
}
