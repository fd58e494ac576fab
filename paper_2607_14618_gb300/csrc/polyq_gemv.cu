// Decode GEMV for the PolyQ mixed-bit layer (one launch over all blocks).
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "polyq.h"
#include "polyq_internal.h"

namespace {

// One warp per output row; lanes stride over the clustered positions.
__global__ void gemv_rowwarp_kernel(polyq_dev_layer L, const __nv_bfloat16* __restrict__ x,
                                    int batch, float* __restrict__ y,
                                    const float* __restrict__ residual) {
  const int warps = blockDim.x >> 5;
  const int64_t n = (int64_t)blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (n >= L.N) return;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  const uint8_t* row = L.packed + n * L.row_stride;
  const uint32_t* mrow = L.meta + n * L.n_groups;
  for (int bi = 0; bi < L.n_blocks; ++bi) {
    const polyq_block B = L.blocks[bi];
    const uint8_t* seg = row + B.seg_off;
    for (int32_t j = lane; j < B.n_ch; j += 32) {
      float w;
      if (B.bits == 16) {
        uint16_t h = (uint16_t)seg[2 * j] | ((uint16_t)seg[2 * j + 1] << 8);
        w = __half2float(__ushort_as_half(h));
      } else {
        const int64_t bit = (int64_t)j * B.bits;
        const int sh = (int)(bit & 7);
        uint32_t v = seg[bit >> 3];
        if (sh + B.bits > 8) v |= (uint32_t)seg[(bit >> 3) + 1] << 8;
        const uint32_t q = (v >> sh) & ((1u << B.bits) - 1u);
        const uint32_t m = mrow[B.grp_off + j / POLYQ_GROUP];
        const float s = __half2float(__ushort_as_half((uint16_t)(m & 0xFFFF)));
        const float z = __half2float(__ushort_as_half((uint16_t)(m >> 16)));
        w = ((float)q - z) * s;
      }
      const int32_t p = B.pos0 + j;
      const int32_t src = L.gather ? L.gather[p] : p;
      for (int b = 0; b < batch; ++b) acc[b] += w * __bfloat162float(x[(int64_t)b * L.K + src]);
    }
  }
  for (int b = 0; b < batch; ++b) {
    float v = acc[b];
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) {
      const int64_t idx = (int64_t)b * L.N + n;
      y[idx] = v + (residual ? residual[idx] : 0.f);
    }
  }
}

}  // namespace

extern "C" int polyq_gemv_workspace_bytes(const polyq_dev_layer* L, int batch, size_t* bytes) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_gemv_workspace_bytes");
  if (rc) return rc;
  if (!bytes) return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_workspace_bytes: bytes is NULL");
  if (batch < 1 || batch > 4)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_gemv_workspace_bytes: batch %d", batch);
  *bytes = 0;
  return POLYQ_OK;
}

extern "C" int polyq_linear_gemv(const polyq_dev_layer* L, const void* x, int batch, float* y,
                                 const float* residual, void* workspace, size_t ws_bytes,
                                 void* stream) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_linear_gemv");
  if (rc) return rc;
  (void)workspace;
  (void)ws_bytes;
  if (!x || !y) return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemv: x or y is NULL");
  if (batch < 1 || batch > 4)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_linear_gemv: batch %d not in 1..4", batch);
  const int threads = 256;
  const int64_t blocks = (L->N + threads / 32 - 1) / (threads / 32);
  gemv_rowwarp_kernel<<<(unsigned)blocks, threads, 0, (cudaStream_t)stream>>>(
      *L, (const __nv_bfloat16*)x, batch, y, residual);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemv: %s", cudaGetErrorString(e));
  return POLYQ_OK;
}
