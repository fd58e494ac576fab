/*
 * polyq_debug.h - test aids of the debug build of the PolyQ library
 * (libpolyq_debug.so, compiled from the same sources with -DPOLYQ_DEBUG; the
 * product library libpolyq.so does not export these).
 *
 * They run the real decode GEMV and prefill GEMM kernels and, in addition,
 * write out what those kernels' decoders produce, so that a test can compare
 * the decoders with the packed format of Section 4.2 (include/polyq.h: the
 * LSB-first bitstreams, the fp16 scale/zero metadata, dequantised weight
 * (q - zero) * scale) bit for bit.  Arguments and errors as for the calls
 * they wrap.  Each call sets a device-global output pointer, runs the
 * kernels and clears it again, synchronising `stream` around the kernels:
 * do not run two of them at once.
 */
#ifndef POLYQ_DEBUG_H
#define POLYQ_DEBUG_H

#include <stddef.h>
#include <stdint.h>

#include "polyq.h"

#ifdef __cplusplus
extern "C" {
#endif

/* polyq_linear_gemv (no residual); codes_out: device uint16 [N][K], the
 * code of every (row, clustered position) as the streaming kernel's MMA
 * steps decoded it from the TMA-staged packed rows (for 16-bit positions the
 * fp16 bit pattern).  Positions the kernel does not decode keep their
 * contents. */
int polyq_debug_gemv_codes(const polyq_dev_layer* layer, const void* x, int batch, float* y,
                           void* workspace, size_t workspace_bytes, uint16_t* codes_out,
                           void* stream);

/* polyq_linear_gemm; w_out: device uint16 [N][K], the fp16 weight of every
 * (row, clustered position) as the GEMM's dequantisers wrote it into the
 * tensor cores' B operand tile (for 16-bit blocks, as TMA loaded it),
 * fp16_rn((q - zero) * scale) for b < 16. */
int polyq_debug_gemm_weights(const polyq_dev_layer* layer, const void* X, int64_t M, float* Y,
                             void* workspace, size_t workspace_bytes, uint16_t* w_out,
                             void* stream);

#ifdef __cplusplus
}
#endif
#endif /* POLYQ_DEBUG_H */
