// Prefill GEMM of the PolyQ mixed-bit layer on the 5th-generation tensor
// cores (tcgen05, tensor memory):
//
//   Y[m][n] = sum_p X[m][gather[p]] * W'[n][p]        (Section 4.1 product)
//
// The contraction runs over 32-wide K tiles (half a quantisation group); every
// tile lies inside one bit block (Section 4.2) and one group, so each weight
// row of a tile has one (scale, zero).
//  1. gemm_prep gathers X through `gather` into a clustered fp16 matrix Xg
//     (workspace), zero-padded at block ends, with the K order inside each
//     tile permuted the same way the dequantiser emits codes.  Xg is stored
//     as the shared-memory images of the producer's copies: one 16 KB block
//     per (pair of M tiles, K tile), 256 rows of 64 bytes in the 64-byte
//     swizzle, so that one contiguous bulk copy fetches a stage's X.
//     Each row m is scaled by the power of two 2^-e_m that brings its largest
//     |x * t| into [2^14, 2^15), so that any finite bf16 row rounds to fp16
//     without overflow and without dropping small values into subnormals;
//     the epilogue multiplies row m of Y by 2^e_m.
//  2. gemm_main: one persistent CTA per SM, 10 warps.
//       warp 0      TMA producer: Xg blocks (bulk copies), packed code
//                   bytes and meta of 256 weight rows, or for 16-bit blocks the
//                   fp16 weights straight into the operand buffer;
//       warp 1      allocates 512 TMEM columns and issues tcgen05.mma
//                   (M=128, N=256, K=16, fp16 in, fp32 accumulate): the
//                   weights are the A operand, 128 rows per MMA, and the
//                   256 tokens of an M pair the B operand, so a TMEM lane
//                   holds one output column;
//       warps 2..9  dequantise: (q - z) * s in fp16 via magic-number decode,
//                   written in the UMMA 64-byte-swizzle K-major layout.  Warps
//                   2-5 take the even stages and 6-9 the odd ones, two weight
//                   rows per thread; afterwards all eight drain the
//                   accumulator with tcgen05.ld and store fp32 Y, each warp
//                   store covering 32 consecutive columns of one row.
//     Five pipeline stages.  When the (M, N) tiles cannot fill the GPU the K
//     range is split, uniformly or stream-K (each CTA an equal contiguous
//     share of all (tile, K tile) pairs), and the pieces are added into a
//     zeroed Y (so the order of those additions varies); otherwise Y is
//     stored directly.  Every wait is bounded and reports through the
//     workspace status word.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "polyq.h"
#ifdef POLYQ_DEBUG
#include "polyq_debug.h"
#endif
#include "polyq_dev.cuh"
#include "polyq_internal.h"

namespace {

using namespace polyq;

constexpr int BM = 128;           // rows per MMA
constexpr int MT = 2;             // M tiles per work unit (share one weight tile)
constexpr int BN = 256;           // weight rows per work unit
constexpr int BK = 32;            // K per tile: half a quantisation group
constexpr int kStagesG = 5;
constexpr int kCodeBox = 32;      // code bytes per row loaded per tile: the tile's codes from a
                                  // 16-byte aligned start (offset <= 12 with at most 16 bytes of
                                  // codes, or 32 bytes of 8-bit codes at offset 0), one TMA
                                  // row request each (48-byte rows take two)
constexpr int kATile = BM * BK * 2;             // 8 KB (64-byte rows)
constexpr int kBTile = BN * BK * 2;             // 16 KB
constexpr int kCodes = BN * kCodeBox;           // 8 KB
constexpr int kMeta = BN * 16;                  // 4 KB
constexpr int kStageG = MT * kATile + kBTile + kCodes + kMeta;  // 44 KB
constexpr int kThreadsG = 320;
constexpr int kDqWarps = 8;
constexpr double kUnitCostTiles = 12.0;  // per-piece overhead, in K-tile stages, of the split model
constexpr double kStageSeconds = 0.6e-6;  // one K-tile stage of a CTA, measured
constexpr double kZeroBytesPerS = 5e12;   // the pre-pass zeroing Y
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kIdesc = umma_idesc_f16(BM, BN);

struct GmBlock {
  int bits, n_ch, pos0, seg_off, grp_off, n_grp;
  int kt0, n_kt;  // K-tile range of the block
};

struct GmParams {
  CUtensorMap tm_codes;  // packed [N][S] u8, box {kCodeBox, 256}
  CUtensorMap tm_meta;   // meta [N][meta_stride] u32, box {4, 256}
  CUtensorMap tm_w16;    // packed [N][S/2] u16, box {32, 256}, 64B swizzle
  GmBlock blk[POLYQ_MAX_BLOCKS];
  int n_blocks;
  int M, N, K, KT;
  int units_m, units_n, ksplit, units;  // work units: (M pair, N tile, K split)
  int streamk;  // 1: each CTA takes an equal contiguous range of (unit, K tile) pairs
  int has_meta;
  int prep_staged;  // 1: the pre-pass stages each row of X in shared memory
  const __nv_bfloat16* x;
  const int32_t* gather;
  const float* xscale;  // Section 3.4 activation factors (clustered order) or NULL
  __half* xg;
  float* rowscale;      // [M]: 2^e_m, the power of two row m of Xg was divided by
  float* y;
  int* status;
};

// try_wait that lets the hardware suspend the thread for up to `hint_ns`
// (it wakes when the phase completes) instead of returning at once.
__device__ __forceinline__ bool mbar_try_wait_hint(uint32_t bar, uint32_t parity,
                                                   uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

// Bounded waits that also give up once another role of the CTA has failed:
// 0 when the phase completed, 1 on a timeout, 2 when `abort` was raised.  The
// flag is read only after a poll has failed, so that a stage whose barrier
// has already completed costs one poll and no shared load.  The lone producer
// and MMA threads poll with a suspend hint of up to 1 us, so that their
// polling does not take issue slots from the dequantisation warps that share
// their schedulers: at most 2^22 such polls, a few seconds.
constexpr uint32_t kWaitLimitSleep = 1u << 22;
constexpr uint32_t kSuspendHintNs = 1000;
constexpr int kWaitOk = 0, kWaitTimeout = 1, kWaitAborted = 2;
__device__ __forceinline__ int wait_ab(uint32_t bar, uint32_t parity, const volatile int* abort) {
  for (uint32_t it = 0; it < kWaitLimit; ++it) {
    if (mbar_try_wait(bar, parity)) return kWaitOk;
    if (*abort) return kWaitAborted;
  }
  return kWaitTimeout;
}
__device__ __forceinline__ int wait_sleep_ab(uint32_t bar, uint32_t parity,
                                             const volatile int* abort) {
  for (uint32_t it = 0; it < kWaitLimitSleep; ++it) {
    if (mbar_try_wait_hint(bar, parity, kSuspendHintNs)) return kWaitOk;
    if (*abort) return kWaitAborted;
  }
  return kWaitTimeout;
}

// The pieces of work a CTA takes, in order: an output tile (um, un) and a
// range [kt_lo, kt_hi) of its K tiles.  Units are strided over the grid, each
// with its K split's range; with `streamk`, a CTA takes the K tiles
// [T*b/C, T*(b+1)/C) of the T = units * KT (unit, K tile) pairs in unit-major
// order, which cuts at most two units per CTA short.  Every role of a CTA
// walks the same sequence.
struct Pieces {
  long long g, g_hi;
  int u;
  __device__ __forceinline__ void init(const GmParams& P) {
    if (P.streamk) {
      const long long T = (long long)P.units * P.KT;
      g = T * blockIdx.x / gridDim.x;
      g_hi = T * (blockIdx.x + 1) / gridDim.x;
    } else {
      u = blockIdx.x;
    }
  }
  __device__ __forceinline__ bool next(const GmParams& P, int& um, int& un, int& kt_lo,
                                       int& kt_hi) {
    int uu;
    if (P.streamk) {
      if (g >= g_hi) return false;
      uu = (int)(g / P.KT);
      kt_lo = (int)(g - (long long)uu * P.KT);
      kt_hi = (int)min((long long)P.KT, (long long)kt_lo + (g_hi - g));
      g += kt_hi - kt_lo;
    } else {
      if (u >= P.units) return false;
      uu = u;
      u += gridDim.x;
      const int ks = uu / (P.units_m * P.units_n);
      kt_lo = (int)((long long)ks * P.KT / P.ksplit);
      kt_hi = (int)((long long)(ks + 1) * P.KT / P.ksplit);
    }
    um = uu % P.units_m;
    un = (uu / P.units_m) % P.units_n;
    return true;
  }
};

__device__ __forceinline__ int find_kblock(const GmBlock* blk, int nblk, int kt) {
  int b = 0;
  while (b + 1 < nblk && kt >= blk[b + 1].kt0) ++b;
  return b;
}

// The block of the current K tile with its fields in registers.  K tiles
// only increase within a piece, so after a seek at the piece's first tile the
// cursor advances with one comparison per tile instead of a search through
// the block table in shared memory.
struct BlockCursor {
  int bi, kt0, next_kt0, bits, seg_off, grp_off;
  __device__ __forceinline__ void load(const GmBlock* sblk, int nblk) {
    const GmBlock& B = sblk[bi];
    kt0 = B.kt0;
    bits = B.bits;
    seg_off = B.seg_off;
    grp_off = B.grp_off;
    next_kt0 = bi + 1 < nblk ? sblk[bi + 1].kt0 : 0x7FFFFFFF;
  }
  __device__ __forceinline__ void seek(const GmBlock* sblk, int nblk, int kt) {
    bi = find_kblock(sblk, nblk, kt);
    load(sblk, nblk);
  }
  __device__ __forceinline__ void advance(const GmBlock* sblk, int nblk, int kt) {
    while (kt >= next_kt0) {
      ++bi;
      load(sblk, nblk);
    }
  }
};

// Position inside a 32-code half group of the code that fills K slot `s`
// (0..31) of a tile (the order in which the dequantiser emits its fp16 pairs).
__host__ __device__ inline int slot_code(int bits, int s) {
  const int h = s & 1;
  switch (bits) {
    case 2: return 16 * (s >> 4) + ((s & 15) >> 1) + 8 * h;
    case 3: return (s >> 1) + 16 * h;
    case 4: return 8 * (s >> 3) + ((s & 7) >> 1) + 4 * h;
    default: return s;  // 8- and 16-bit: natural order
  }
}

// ---------------------------------------------------------------------------
// pre-pass: Xg(m, kt*32 + s) = fp16(X[m][gather[p]] * xscale[p] * 2^-e_m) with
// p = pos0 + 32 h + slot_code(s)
// for the h-th 32-code half group of the block (tile kt).  Each CTA first
// builds, in shared memory, the map from a clustered slot to the source
// channel it reads (and its activation factor); then, one row at a time, it
// copies the row of X into shared memory with 16-byte loads (finding the
// row's largest magnitude on the way) and gathers from there.  Rows up to
// 16384 wide are held in registers, the next row's loads in flight while the
// current row is gathered.  Global reads and writes are so coalesced whatever
// the permutation.  Layers too wide for shared memory (see prep_smem_bytes)
// gather from global memory instead.  Y is zeroed when the K range is split
// over CTAs.
// ---------------------------------------------------------------------------
constexpr int kRowExp = 14;       // a row's largest magnitude becomes [2^14, 2^15)
constexpr int kRowExpMin = -126;  // 2^e stays a normal float
constexpr int kPrepThreads = 256;
constexpr int kPrepMaxSmem = 200 * 1024;
constexpr int kRowVec = 8;  // 16-byte pieces of a row a thread holds (rows up to 16384 wide)

// Element offset of Xg(m, k) in the blocked layout: block (m / 256, k / 32)
// of 256 rows x 32 fp16, row m % 256 at 64 bytes each, its 16-byte chunks
// in the 64-byte swizzle (chunk index XOR bits 7..8 of the byte address).
__device__ __forceinline__ size_t xg_off(int m, int k, int KT) {
  const int r = m & (MT * BM - 1), c = (k >> 3) & 3;
  return (((size_t)(m / (MT * BM)) * KT + (k >> 5)) * (MT * BM) + r) * BK +
         ((c ^ ((r >> 1) & 3)) << 3) + (k & 7);
}

// Clustered K slot k of a row: the position p it takes its value from, or -1
// past the end of a block.
__device__ __forceinline__ int slot_pos(const GmBlock* sblk, int nblk, int k) {
  const int kt = k / BK, s = k % BK;
  const GmBlock& B = sblk[find_kblock(sblk, nblk, kt)];
  const int w = 32 * (kt - B.kt0) + slot_code(B.bits, s);
  return w < B.n_ch ? B.pos0 + w : -1;
}

// Shared memory of the staged pre-pass: the slot -> source map (int32 [Kp]),
// the slot factors (fp32 [Kp], scaled layers only) and one row of X (bf16
// [K]); 0 when it does not fit.
size_t prep_smem_bytes(int K, int Kp, bool xscale) {
  const size_t b = (size_t)Kp * 4 * (xscale ? 2 : 1) + ((size_t)K * 2 + 15) / 16 * 16;
  return b <= (size_t)kPrepMaxSmem ? b : 0;
}

__global__ void __launch_bounds__(kPrepThreads) gemm_prep(const __grid_constant__ GmParams P) {
  extern __shared__ __align__(16) uint8_t psm[];
  pdl_trigger();
  __shared__ GmBlock sblk[POLYQ_MAX_BLOCKS];
  __shared__ uint32_t s_wmax[kPrepThreads / 32];
  if (threadIdx.x < POLYQ_MAX_BLOCKS) {
    switch (threadIdx.x) {
      case 0: sblk[0] = P.blk[0]; break;
      case 1: sblk[1] = P.blk[1]; break;
      case 2: sblk[2] = P.blk[2]; break;
      case 3: sblk[3] = P.blk[3]; break;
      default: sblk[4] = P.blk[4]; break;
    }
  }
  __syncthreads();
  const int Kp = P.KT * BK, half = Kp / 2;  // slots and fp16 pairs per row of Xg
  const bool staged = P.prep_staged != 0;
  int* s_src = reinterpret_cast<int*>(psm);
  float* s_fac = reinterpret_cast<float*>(psm + (size_t)Kp * 4);
  uint16_t* s_row = reinterpret_cast<uint16_t*>(psm + (size_t)Kp * 4 * (P.xscale ? 2 : 1));
  if (staged) {
    // static layer data, built before the wait for the previous kernel; a
    // thread's loads of 16 slots are issued together
    constexpr int U = 16;
    for (int k0 = threadIdx.x; k0 < Kp; k0 += kPrepThreads * U) {
      int pos[U], src[U];
      float fac[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int k = k0 + u * kPrepThreads;
        pos[u] = k < Kp ? slot_pos(sblk, P.n_blocks, k) : -1;
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        src[u] = pos[u] < 0 ? -1 : (P.gather ? __ldg(P.gather + pos[u]) : pos[u]);
        fac[u] = (P.xscale && pos[u] >= 0) ? __ldg(P.xscale + pos[u]) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int k = k0 + u * kPrepThreads;
        if (k < Kp) {
          s_src[k] = src[u];
          if (P.xscale) s_fac[k] = fac[u];
        }
      }
    }
  }
  pdl_wait();  // X comes from the previous kernel; Y and the workspace may still be in use
  if (blockIdx.x == 0 && threadIdx.x == 0) *P.status = 0;
  if (P.ksplit > 1 || P.streamk) {
    const long long total4 = (long long)P.M * P.N / 4;
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total4;
         e += (long long)gridDim.x * blockDim.x)
      reinterpret_cast<float4*>(P.y)[e] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  // the value at clustered slot k of row m
  auto value = [&](int m, int k) -> float {
    int src;
    float f = 1.f;
    if (staged) {
      src = s_src[k];
      if (src < 0) return 0.f;
      if (P.xscale) f = s_fac[k];
    } else {
      const int p = slot_pos(sblk, P.n_blocks, k);
      if (p < 0) return 0.f;
      src = P.gather ? __ldg(P.gather + p) : p;
      if (P.xscale) f = __ldg(P.xscale + p);
    }
    const uint16_t b = staged ? s_row[src]
                              : __ldg(reinterpret_cast<const uint16_t*>(P.x) + (size_t)m * P.K + src);
    return __uint_as_float((uint32_t)b << 16) * f;
  };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Row scale of row m from its largest magnitude bits mx (fp32 bit pattern,
  // per thread): e_m = floor(log2(max)) - kRowExp, an fp32 subnormal maximum
  // counting as 2^-127.  2^e and 2^-e are normal floats (-126 <= e <= 113),
  // so the products with 2^-e are exact scalings (rounded like any product
  // where they fall below the normal range).  Returns 2^-e_m.
  // The rows of the last M pair past M are zero (their MMA columns are not
  // stored, but they must be finite).
  auto zero_pad_rows = [&]() {
    const int Mp = P.units_m * (MT * BM);
    for (int m = P.M + blockIdx.x; m < Mp; m += gridDim.x)
      for (int i = threadIdx.x; i < Kp / 4; i += kPrepThreads)
        *reinterpret_cast<uint2*>(P.xg + xg_off(m, 4 * i, P.KT)) = make_uint2(0u, 0u);
  };
  auto row_scale = [&](int m, uint32_t mx) -> float {
    if (P.xscale) {
      mx = 0;
      for (int k = threadIdx.x; k < Kp; k += kPrepThreads)
        mx = max(mx, __float_as_uint(fabsf(value(m, k))));
    }
    mx = __reduce_max_sync(0xffffffffu, mx);
    if (lane == 0) s_wmax[warp] = mx;
    __syncthreads();
#pragma unroll
    for (int w = 0; w < kPrepThreads / 32; ++w) mx = max(mx, s_wmax[w]);
    const int e = mx ? max((int)(mx >> 23) - 127 - kRowExp, kRowExpMin) : 0;
    if (threadIdx.x == 0) P.rowscale[m] = __int_as_float((127 + e) << 23);
    return __int_as_float((127 - e) << 23);
  };
  const int n8 = P.K / 8;  // 16-byte pieces of a row
  const bool vec = staged && (P.K & 7) == 0 && (reinterpret_cast<uintptr_t>(P.x) & 15) == 0 &&
                   n8 <= kRowVec * kPrepThreads;
  if (vec) {
    // A thread holds its pieces of a row in registers: the next row's loads
    // are issued before the current row is gathered, so they are in flight
    // meanwhile.
    auto load_row = [&](int m, uint4 (&v)[kRowVec]) {
      const uint4* row = reinterpret_cast<const uint4*>(P.x) + (size_t)m * n8;
#pragma unroll
      for (int u = 0; u < kRowVec; ++u) {
        const int i = threadIdx.x + u * kPrepThreads;
        v[u] = i < n8 ? __ldg(row + i) : make_uint4(0u, 0u, 0u, 0u);
      }
    };
    uint4 v[kRowVec];
    if ((int)blockIdx.x < P.M) load_row(blockIdx.x, v);
    for (int m = blockIdx.x; m < P.M; m += gridDim.x) {
      uint32_t mx = 0;
#pragma unroll
      for (int u = 0; u < kRowVec; ++u) {
        const int i = threadIdx.x + u * kPrepThreads;
        if (i < n8) {
          reinterpret_cast<uint4*>(s_row)[i] = v[u];
          const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
          for (int q = 0; q < 4; ++q) mx = max(mx, max(w[q] & 0x7FFFu, (w[q] >> 16) & 0x7FFFu));
        }
      }
      mx <<= 16;  // bf16 magnitude bits -> fp32 bits
      __syncthreads();  // the staged row (and, on the first row, the map) is complete
      const float inv = row_scale(m, mx);
      if (m + (int)gridDim.x < P.M) load_row(m + gridDim.x, v);
      // four consecutive slots per thread and 8-byte store (with eight, the
      // row reads of a warp's threads collide in shared-memory banks more)
      for (int i = threadIdx.x; i < Kp / 4; i += kPrepThreads) {
        uint32_t w[2];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const __half2 h = __halves2half2(__float2half_rn(value(m, 4 * i + 2 * q) * inv),
                                           __float2half_rn(value(m, 4 * i + 2 * q + 1) * inv));
          w[q] = *reinterpret_cast<const uint32_t*>(&h);
        }
        *reinterpret_cast<uint2*>(P.xg + xg_off(m, 4 * i, P.KT)) = make_uint2(w[0], w[1]);
      }
      __syncthreads();  // the row buffer and s_wmax are reused by the next row
    }
    zero_pad_rows();
    return;
  }
  for (int m = blockIdx.x; m < P.M; m += gridDim.x) {
    // largest magnitude of the row's values (bit patterns of non-negative
    // floats order as integers); without activation factors that is the
    // largest |X[m][k]| over the raw row, since the gather is a permutation
    const uint16_t* row = reinterpret_cast<const uint16_t*>(P.x) + (size_t)m * P.K;
    uint32_t mx = 0;
    if ((P.K & 7) == 0 && (reinterpret_cast<uintptr_t>(row) & 15) == 0) {
      for (int i = threadIdx.x; i < P.K / 8; i += kPrepThreads) {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(row) + i);
        if (staged) reinterpret_cast<uint4*>(s_row)[i] = v;
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) mx = max(mx, max(w[q] & 0x7FFFu, (w[q] >> 16) & 0x7FFFu));
      }
    } else {
      for (int i = threadIdx.x; i < P.K; i += kPrepThreads) {
        const uint16_t v = __ldg(row + i);
        if (staged) s_row[i] = v;
        mx = max(mx, (uint32_t)(v & 0x7FFFu));
      }
    }
    mx <<= 16;  // bf16 magnitude bits -> fp32 bits
    __syncthreads();  // the staged row (and, on the first row, the map) is complete
    const float inv = row_scale(m, mx);
    for (int i = threadIdx.x; i < half; i += kPrepThreads)
      *reinterpret_cast<__half2*>(P.xg + xg_off(m, 2 * i, P.KT)) =
          __halves2half2(__float2half_rn(value(m, 2 * i) * inv),
                         __float2half_rn(value(m, 2 * i + 1) * inv));
    __syncthreads();  // the row buffer and s_wmax are reused by the next row
  }
  zero_pad_rows();
}

// ---------------------------------------------------------------------------
// dequantisation of one weight row of one tile into the swizzled B operand
// ---------------------------------------------------------------------------
// Row r, 16-byte chunk c (0..3) of a K-major tile with 64-byte rows and the
// 64-byte swizzle (chunk index XOR bits 7..8 of the address).
__device__ __forceinline__ void store_pairs_sw64(uint8_t* btile, int r, int chunk,
                                                 const uint32_t (&p)[4]) {
  uint8_t* dst = btile + r * 64 + ((chunk ^ ((r >> 1) & 3)) << 4);
  *reinterpret_cast<uint4*>(dst) = make_uint4(p[0], p[1], p[2], p[3]);
}

__device__ __forceinline__ void red_add_f32(float* p, float a) {
  asm volatile("red.global.add.f32 [%0], %1;" ::"l"(p), "f"(a) : "memory");
}

__device__ __forceinline__ uint32_t dq_pair(uint32_t raw, __half2 zz, __half2 ss) {
  // raw holds fp16 (1024 + q) in each half: (q - z) is exact, the product
  // (q - z) * s is rounded once to fp16.
  const __half2 d = __hsub2(*reinterpret_cast<const __half2*>(&raw), zz);
  const __half2 w = __hmul2(d, ss);
  return *reinterpret_cast<const uint32_t*>(&w);
}

// Dequantise 32 codes of weight row r.  `w` holds the row's code words
// starting at the first code (2-bit: 2 words, 3-bit: 3, 4-bit: 4, 8-bit: 8).
__device__ __forceinline__ void dequant_row(int bits, const uint32_t (&w)[8], uint32_t meta,
                                            uint8_t* btile, int r) {
  const uint32_t magic = 0x64006400u;
  const __half s = __ushort_as_half((uint16_t)(meta & 0xFFFFu));
  const __half z = __ushort_as_half((uint16_t)(meta >> 16));
  const __half2 ss = __halves2half2(s, s);
  const __half zz1 = __hadd(z, __float2half(1024.f));
  const __half2 zz = __halves2half2(zz1, zz1);
  if (bits == 2) {
#pragma unroll
    for (int wd = 0; wd < 2; ++wd) {
#pragma unroll
      for (int c2 = 0; c2 < 2; ++c2) {
        uint32_t p[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int ii = 4 * c2 + i;
          p[i] = dq_pair(((w[wd] >> (2 * ii)) & 0x00030003u) | magic, zz, ss);
        }
        store_pairs_sw64(btile, r, 2 * wd + c2, p);
      }
    }
  } else if (bits == 3) {
    const uint32_t a = w[0], b = w[1], c = w[2];
#pragma unroll
    for (int c4 = 0; c4 < 4; ++c4) {
      uint32_t p[4];
#pragma unroll
      for (int i4 = 0; i4 < 4; ++i4) {
        const int i = 4 * c4 + i4;  // codes i and i + 16
        const int o = 3 * i;
        const uint32_t lo = o < 32 ? __funnelshift_r(a, b, o) : __funnelshift_r(b, c, o - 32);
        const uint32_t hi = o < 32 ? __funnelshift_r(b, c, o) : (c >> (o - 32));
        p[i4] = dq_pair((__byte_perm(lo, hi, 0x7610) & 0x00070007u) | magic, zz, ss);
      }
      store_pairs_sw64(btile, r, c4, p);
    }
  } else if (bits == 4) {
#pragma unroll
    for (int wd = 0; wd < 4; ++wd) {
      uint32_t p[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) p[i] = dq_pair(((w[wd] >> (4 * i)) & 0x000F000Fu) | magic, zz, ss);
      store_pairs_sw64(btile, r, wd, p);
    }
  } else {  // 8-bit
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      uint32_t p[4];
      p[0] = dq_pair(__byte_perm(w[2 * c], 0x64646464u, 0x4140), zz, ss);
      p[1] = dq_pair(__byte_perm(w[2 * c], 0x64646464u, 0x4342), zz, ss);
      p[2] = dq_pair(__byte_perm(w[2 * c + 1], 0x64646464u, 0x4140), zz, ss);
      p[3] = dq_pair(__byte_perm(w[2 * c + 1], 0x64646464u, 0x4342), zz, ss);
      store_pairs_sw64(btile, r, c, p);
    }
  }
}

#ifdef POLYQ_DEBUG
// Debug build only: every fp16 weight the dequantisers (or, for 16-bit
// blocks, TMA) place in a B tile is written to g_dbg_w[n][position] (the
// layer's clustered order), read back from the swizzled tile.
__device__ uint16_t* g_dbg_w;
__device__ long long g_dbg_wK;

__device__ __forceinline__ void dbg_row(const uint8_t* btile, int r, int n, int N,
                                        const GmBlock& B, int hg) {
  uint16_t* out = g_dbg_w;
  if (!out || n >= N) return;
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    const uint16_t* src =
        reinterpret_cast<const uint16_t*>(btile + r * 64 + ((c ^ ((r >> 1) & 3)) << 4));
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int w = 32 * hg + slot_code(B.bits, 8 * c + e);
      if (w < B.n_ch) out[(long long)n * g_dbg_wK + B.pos0 + w] = src[e];
    }
  }
}
#endif

__global__ void __launch_bounds__(kThreadsG, 1) gemm_main(const __grid_constant__ GmParams P) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment of the operand tiles (128-byte swizzle atoms)
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  __shared__ uint64_t bar_full[kStagesG], bar_bready[kStagesG], bar_sfree[kStagesG];
  __shared__ uint64_t bar_accf, bar_acce;
  __shared__ uint32_t tmem_base_slot;
  __shared__ GmBlock sblk[POLYQ_MAX_BLOCKS];
  __shared__ volatile int s_abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x < POLYQ_MAX_BLOCKS) {
    switch (threadIdx.x) {
      case 0: sblk[0] = P.blk[0]; break;
      case 1: sblk[1] = P.blk[1]; break;
      case 2: sblk[2] = P.blk[2]; break;
      case 3: sblk[3] = P.blk[3]; break;
      default: sblk[4] = P.blk[4]; break;
    }
  }
  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int s = 0; s < kStagesG; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);
      mbar_init(smem_u32(&bar_bready[s]), kDqWarps / 2);  // one group of four warps per stage
      mbar_init(smem_u32(&bar_sfree[s]), 1);
    }
    mbar_init(smem_u32(&bar_accf), 1);
    mbar_init(smem_u32(&bar_acce), kDqWarps);
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_slot;
  pdl_trigger();

  const int nblk = P.n_blocks;
  auto stage_ptr = [&](int s) { return smem + s * kStageG; };
  auto fail = [&](int code) {
    s_abort = 1;
    atomicExch(P.status, code);
  };

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      prefetch_tmap(&P.tm_codes);
      if (P.has_meta) prefetch_tmap(&P.tm_meta);
      prefetch_tmap(&P.tm_w16);
      pdl_wait();  // Xg comes from the pre-pass
      int kg = 0;
      Pieces pc;
      pc.init(P);
      int um, un, kt_lo, kt_hi;
      BlockCursor B;
      while (!s_abort && pc.next(P, um, un, kt_lo, kt_hi)) {
        B.seek(sblk, nblk, kt_lo);
        for (int kt = kt_lo; kt < kt_hi; ++kt, ++kg) {
          const int s = kg % kStagesG, use = kg / kStagesG;
          if (use > 0) {
            const int w = wait_sleep_ab(smem_u32(&bar_sfree[s]), (use - 1) & 1, &s_abort);
            if (w != kWaitOk) {
              if (w == kWaitTimeout) fail(kStatusTimeoutEmpty);
              break;
            }
          }
          B.advance(sblk, nblk, kt);
          const int hg = kt - B.kt0;  // half group
          uint8_t* st = stage_ptr(s);
          const uint32_t bar = smem_u32(&bar_full[s]);
          const bool w16 = B.bits == 16;
          mbar_expect_tx(bar, MT * kATile + (w16 ? kBTile : kCodes + kMeta));
          // both M tiles of X: one 16 KB block of Xg, already in the
          // swizzled shared-memory layout
          bulk_load(smem_u32(st), P.xg + ((size_t)um * P.KT + kt) * (MT * BM * BK), MT * kATile,
                    bar);
          if (w16) {
            tma_load_2d(smem_u32(st + MT * kATile), &P.tm_w16, (B.seg_off + 64 * hg) / 2, un * BN,
                        bar);
          } else {
            const int start = B.seg_off + 4 * B.bits * hg;
            tma_load_2d(smem_u32(st + MT * kATile + kBTile), &P.tm_codes, start & ~15, un * BN,
                        bar);
            tma_load_2d(smem_u32(st + MT * kATile + kBTile + kCodes), &P.tm_meta,
                        (B.grp_off + hg / 2) & ~3, un * BN, bar);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int uc = 0, s = 0;
      uint32_t ph = 0;
      const uint64_t dx0 = umma_desc_sw64(smem_u32(smem));
      const uint64_t dw0 = umma_desc_sw64(smem_u32(smem + MT * kATile));
      Pieces pc;
      pc.init(P);
      int um, un, kt_lo, kt_hi;
      for (; !s_abort && pc.next(P, um, un, kt_lo, kt_hi); ++uc) {
        if (uc > 0) {
          const int w = wait_sleep_ab(smem_u32(&bar_acce), (uc - 1) & 1, &s_abort);
          if (w != kWaitOk) {
            if (w == kWaitTimeout) fail(kStatusTimeoutEmpty);
            break;
          }
        }
        tc_fence_after();
        for (int kt = kt_lo; kt < kt_hi; ++kt) {
          // Every dequantiser warp of the stage's group waits for the
          // stage's copies (bar_full) before it arrives on bar_bready, so
          // bar_bready alone orders the MMAs after the X tile and the weights.
          const int w = wait_sleep_ab(smem_u32(&bar_bready[s]), ph, &s_abort);
          if (w != kWaitOk) {
            if (w == kWaitTimeout) fail(kStatusTimeoutFull);
            break;
          }
          tc_fence_after();
          // A: 128 of the tile's 256 weight rows; B: all 256 tokens of the M
          // pair (one 256-row box).  Accumulator t holds weight rows 128 t..
          // in its TMEM lanes and the tokens in its 256 columns.  The slot's
          // descriptors are those of slot 0 plus its offset (address >> 4).
          const uint64_t so = (uint64_t)((s * kStageG) >> 4);
          const uint64_t dx = dx0 + so, dw = dw0 + so;
#pragma unroll
          for (int t = 0; t < MT; ++t)
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              tc_mma_f16(tmem + t * BN, dw + (uint64_t)((t * BM * BK * 2) >> 4) + 2 * kk, dx + 2 * kk,
                         kIdesc, (kt > kt_lo || kk > 0) ? 1u : 0u);
          tc_commit(smem_u32(&bar_sfree[s]));
          if (++s == kStagesG) {
            s = 0;
            ph ^= 1u;
          }
        }
        tc_commit(smem_u32(&bar_accf));
      }
    }
  } else {
    // ---------------- dequantisation + epilogue (8 warps) ----------------
    // Two groups of four warps take alternate stages (group g the stages
    // with kg % 2 == g); a thread dequantises rows r0 and r0 + 128 of its
    // group's stages.  Each group so has two stage periods for its
    // latency-bound work, and each thread two independent rows.
    const int dq = threadIdx.x - 64;  // 0..255
    const int grp = dq >> 7;
    const int r0 = dq & 127;
    const int q = warp & 3;          // TMEM lane quarter this warp may access
    const int half = (warp - 2) >> 2;
    int kg = 0, uc = 0;
    Pieces pc;
    pc.init(P);
    int um, un, kt_lo, kt_hi;
    BlockCursor B;
    for (; !s_abort && pc.next(P, um, un, kt_lo, kt_hi); ++uc) {
      B.seek(sblk, nblk, kt_lo);
      for (int kt = kt_lo; kt < kt_hi; ++kt, ++kg) {
        if ((kg & 1) != grp) continue;
        const int s = kg % kStagesG, use = kg / kStagesG;
        // The producer issues a slot's copies only after the MMAs of its
        // previous use are done, so once they have landed the weight tile
        // may be overwritten too.
        const int w = wait_ab(smem_u32(&bar_full[s]), use & 1, &s_abort);
        if (w != kWaitOk) {
          if (w == kWaitTimeout) fail(kStatusTimeoutFull);
          break;
        }
        B.advance(sblk, nblk, kt);
        if (B.bits != 16) {
          const int hg = kt - B.kt0;
          uint8_t* st = stage_ptr(s);
          const int start = B.seg_off + 4 * B.bits * hg;
          const int mslot = (B.grp_off + hg / 2) & 3;
          const int sh = (start & 15) >> 2;  // uniform over the CTA
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int r = r0 + 128 * h;
            // the row's code bytes start at offset (start & 15) of a 16-byte
            // aligned window; two conflict-free 16-byte reads cover them
            const uint4* rp =
                reinterpret_cast<const uint4*>(st + MT * kATile + kBTile + r * kCodeBox);
            const uint4 c0 = rp[0], c1 = rp[1];
            const uint32_t cw[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
            uint32_t w[8];
            switch (sh) {
              case 0:
#pragma unroll
                for (int k = 0; k < 8; ++k) w[k] = cw[k];
                break;
              case 1:
#pragma unroll
                for (int k = 0; k < 7; ++k) w[k] = cw[k + 1];
                w[7] = 0;
                break;
              case 2:
#pragma unroll
                for (int k = 0; k < 6; ++k) w[k] = cw[k + 2];
                w[6] = w[7] = 0;
                break;
              default:
#pragma unroll
                for (int k = 0; k < 5; ++k) w[k] = cw[k + 3];
                w[5] = w[6] = w[7] = 0;
                break;
            }
            const uint32_t meta = reinterpret_cast<const uint32_t*>(
                st + MT * kATile + kBTile + kCodes)[r * 4 + mslot];
            dequant_row(B.bits, w, meta, st + MT * kATile, r);
#ifdef POLYQ_DEBUG
            dbg_row(st + MT * kATile, r, un * BN + r, P.N, sblk[B.bi], hg);
#endif
          }
          fence_proxy_async_smem();
        }
#ifdef POLYQ_DEBUG
        else {
          for (int h = 0; h < 2; ++h)
            dbg_row(stage_ptr(s) + MT * kATile, r0 + 128 * h, un * BN + r0 + 128 * h, P.N,
                    sblk[B.bi], kt - B.kt0);
        }
#endif
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bar_bready[s]));
      }
      if (s_abort) break;
      // epilogue: lane i of a warp owns output column n = weight row
      // 128 t + 32 q + i of the tile, and each TMEM column one token of the
      // M pair, so every store of a warp writes 32 consecutive floats of one
      // row of Y.  Tokens [128 half, +128) of the pair, 32 at a time.  The
      // 2^e_m of the pre-pass (one token per lane, broadcast by shuffles) are
      // loaded together, and both accumulators' TMEM loads of a chunk share
      // one wait.  (The loads follow the accumulator's barrier, which orders
      // them after the pre-pass even for a warp that took no stage.)
      {
        const int w = wait_ab(smem_u32(&bar_accf), uc & 1, &s_abort);
        if (w != kWaitOk) {
          if (w == kWaitTimeout) fail(kStatusTimeoutFull);
          break;
        }
      }
      tc_fence_after();
      const int mh = um * (MT * BM) + 128 * half;
      float rs_l[4];
#pragma unroll
      for (int c4 = 0; c4 < 4; ++c4)
        rs_l[c4] = mh + 32 * c4 + lane < P.M ? P.rowscale[mh + 32 * c4 + lane] : 0.f;
      const bool add = P.ksplit > 1 || P.streamk;  // Y was zeroed by the pre-pass
      const int n0 = un * BN + 32 * q + lane;       // + BM for the second accumulator
#pragma unroll
      for (int c4 = 0; c4 < 4; ++c4) {
        const int m0 = mh + 32 * c4;
        const int jn = min(32, P.M - m0);  // tokens of this chunk inside M
        if (jn <= 0) break;
        uint32_t v0[32], v1[32];
        const uint32_t ta = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(128 * half + 32 * c4);
        tc_ld_32x32b_x32(ta, v0);
        tc_ld_32x32b_x32(ta + BN, v1);
        tc_wait_ld();
        tc_regs_ready(v0);
        tc_regs_ready(v1);
        float* dst = P.y + (size_t)m0 * P.N + n0;
        const bool ok0 = n0 < P.N, ok1 = n0 + BM < P.N;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float rs = __shfl_sync(0xffffffffu, rs_l[c4], j);
          if (j < jn) {
            const float f0 = __uint_as_float(v0[j]) * rs, f1 = __uint_as_float(v1[j]) * rs;
            if (add) {
              if (ok0) red_add_f32(dst, f0);
              if (ok1) red_add_f32(dst + BM, f1);
            } else {
              if (ok0) dst[0] = f0;
              if (ok1) dst[BM] = f1;
            }
          }
          dst += P.N;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bar_acce));
    }
  }

  // all roles done (or aborted): wait for the last tensor-core work, free TMEM
  __syncthreads();
  if (warp == 1) {
    if (lane == 0) {
      // the last commit of this CTA went to bar_accf; its completion means all
      // MMAs have finished reading shared memory and writing TMEM
      int uc = 0;
      Pieces pc;
      pc.init(P);
      int um, un, kt_lo, kt_hi;
      while (pc.next(P, um, un, kt_lo, kt_hi)) ++uc;
      if (uc > 0) mbar_wait(smem_u32(&bar_accf), (uc - 1) & 1);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int k_tiles(const polyq_dev_layer* L, GmBlock* blk) {
  int kt = 0;
  for (int i = 0; i < L->n_blocks; ++i) {
    const polyq_block& b = L->blocks[i];
    GmBlock g;
    g.bits = b.bits;
    g.n_ch = b.n_ch;
    g.pos0 = b.pos0;
    g.seg_off = b.seg_off;
    g.grp_off = b.grp_off;
    g.n_grp = b.n_grp;
    g.kt0 = kt;
    g.n_kt = (b.n_ch + BK - 1) / BK;  // half groups
    kt += g.n_kt;
    if (blk) blk[i] = g;
  }
  return kt;
}

// Workspace: Xg (16 KB blocks, M rounded up to a pair of M tiles) fp16, the
// row scales [M] fp32, then 256 bytes holding the status word; each part
// starts on a 256-byte boundary.
size_t gemm_xg_bytes(const polyq_dev_layer* L, int64_t M) {
  const size_t Mp = (size_t)((M + MT * BM - 1) / (MT * BM)) * (MT * BM);
  return (Mp * k_tiles(L, nullptr) * BK * 2 + 255) / 256 * 256;
}
size_t gemm_workspace(const polyq_dev_layer* L, int64_t M) {
  return gemm_xg_bytes(L, M) + ((size_t)M * 4 + 255) / 256 * 256 + 256;
}

}  // namespace

extern "C" int polyq_gemm_workspace_bytes(const polyq_dev_layer* L, int64_t M, size_t* bytes) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_gemm_workspace_bytes");
  if (rc) return rc;
  if (!bytes) return polyq_set_error(POLYQ_EINVAL, "polyq_gemm_workspace_bytes: bytes is NULL");
  if (M < 1 || M > (1 << 24))
    return polyq_set_error(POLYQ_EINVAL, "polyq_gemm_workspace_bytes: M=%lld", (long long)M);
  *bytes = gemm_workspace(L, M);
  return POLYQ_OK;
}

#ifdef POLYQ_DEBUG
// Debug build only: polyq_linear_gemm with every weight placed in a B tile
// written to w_out [N][K] (fp16 bits, clustered order).
extern "C" int polyq_debug_gemm_weights(const polyq_dev_layer* L, const void* X, int64_t M,
                                        float* Y, void* workspace, size_t ws_bytes,
                                        uint16_t* w_out, void* stream) {
  polyq_clear_error();
  cudaStream_t st = (cudaStream_t)stream;
  const long long K = L ? L->K : 0;
  cudaError_t e = cudaMemcpyToSymbolAsync(g_dbg_w, &w_out, sizeof w_out, 0,
                                          cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyToSymbolAsync(g_dbg_wK, &K, sizeof K, 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return polyq_set_error(POLYQ_ECUDA, "debug: %s", cudaGetErrorString(e));
  const int rc = polyq_linear_gemm(L, X, M, Y, workspace, ws_bytes, stream);
  uint16_t* none = nullptr;
  cudaMemcpyToSymbolAsync(g_dbg_w, &none, sizeof none, 0, cudaMemcpyHostToDevice, st);
  cudaStreamSynchronize(st);
  return rc;
}
#endif

extern "C" int polyq_linear_gemm(const polyq_dev_layer* L, const void* X, int64_t M, float* Y,
                                 void* workspace, size_t ws_bytes, void* stream) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_linear_gemm");
  if (rc) return rc;
  if (!X || !Y) return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemm: X or Y is NULL");
  if ((uintptr_t)Y % 16)  // Y is zeroed for split K with 16-byte stores
    return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemm: Y must be 16-byte aligned");
  if (M < 1 || M > (1 << 24))
    return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemm: M=%lld", (long long)M);
  const size_t need = gemm_workspace(L, M);
  if (!workspace || ws_bytes < need)
    return polyq_set_error(POLYQ_ENOMEM, "polyq_linear_gemm: workspace needs %zu bytes, got %zu",
                           need, ws_bytes);
  if ((uintptr_t)workspace % 256)
    return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemm: workspace must be 256-byte aligned");
  if (L->row_stride % 16)
    return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemm: row_stride must be a multiple of 16");

  GmParams P;
  memset(&P, 0, sizeof P);
  const int KT = k_tiles(L, P.blk);
  P.n_blocks = L->n_blocks;
  P.M = (int)M;
  P.N = (int)L->N;
  P.K = (int)L->K;
  P.KT = KT;
  P.units_m = (int)((M + MT * BM - 1) / (MT * BM));
  P.units_n = (int)((L->N + BN - 1) / BN);
  P.x = (const __nv_bfloat16*)X;
  P.gather = L->gather;
  P.xscale = L->xscale;
  P.xg = (__half*)workspace;
  P.rowscale = (float*)((uint8_t*)workspace + gemm_xg_bytes(L, M));
  P.y = Y;
  P.status = (int*)((uint8_t*)workspace + need - 256);
  rc = polyq_tensor_map_2d(&P.tm_codes, L->packed, 1, (uint64_t)L->row_stride, (uint64_t)L->N,
                           (uint64_t)L->row_stride, kCodeBox, BN);
  if (rc) return rc;
  rc = polyq_tensor_map_2d(&P.tm_w16, L->packed, 2, (uint64_t)L->row_stride / 2, (uint64_t)L->N,
                           (uint64_t)L->row_stride, BK, BN, 64);
  if (rc) return rc;
  if (L->n_groups > 0) {
    rc = polyq_tensor_map_2d(&P.tm_meta, L->meta, 4, (uint64_t)L->meta_stride, (uint64_t)L->N,
                             (uint64_t)L->meta_stride * 4, 4, BN);
    if (rc) return rc;
    P.has_meta = 1;
  }

  cudaStream_t st = (cudaStream_t)stream;
  int sms = 0;
  rc = polyq_sm_count(&sms);
  if (rc) return rc;
  // Split K when the (M, N) tiles fill the SMs poorly.  The modelled time, in
  // K-tile stages of one CTA, is for a uniform split into k ranges: whole
  // waves of units times (K tiles per unit + a per-piece cost for filling the
  // pipeline and adding the tile into Y); for stream-K: the K tiles of one
  // CTA's equal share plus the per-piece cost of the (at most three) pieces
  // it touches.  Both add the zeroing of Y when they split.  Each uniform
  // split keeps at least 16 K tiles; near ties go to the simpler choice.
  {
    const int mn = P.units_m * P.units_n;
    const bool can_split = (P.N % 4) == 0;  // zeroing writes float4
    const double zero = (double)M * P.N * 4.0 / kZeroBytesPerS / kStageSeconds;
    int ks = 1;
    double best = 1e300;
    const int kmax = can_split ? std::max(1, std::min(64, KT / 16)) : 1;
    for (int k = 1; k <= kmax; ++k) {
      const long long waves = ((long long)mn * k + sms - 1) / sms;
      const double t = (double)waves * ((double)KT / k + kUnitCostTiles) + (k > 1 ? zero : 0.0);
      if (t < 0.98 * best) {
        best = t;
        ks = k;
      }
    }
    const double share = std::ceil((double)mn * KT / sms);
    const double t_sk = share + kUnitCostTiles * (std::ceil(share / KT) + 1.0) + zero;
    if (can_split && (long long)mn * KT >= sms && t_sk < 0.98 * best) {
      P.streamk = 1;
      P.ksplit = 1;
      P.units = mn;
    } else {
      P.ksplit = ks;
      P.units = mn * ks;
    }
  }
  static bool attr_done[8] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  const size_t smem = (size_t)kStagesG * kStageG + 1024;
  if (!attr_done[dev & 7]) {
    cudaError_t e = cudaFuncSetAttribute(gemm_main, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess)
      return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemm: smem attribute: %s",
                             cudaGetErrorString(e));
    attr_done[dev & 7] = true;
  }
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  const size_t prep_smem = prep_smem_bytes(P.K, KT * BK, P.xscale != nullptr);
  P.prep_staged = prep_smem > 0;
  static bool prep_attr_done[8] = {false};
  if (!prep_attr_done[dev & 7]) {
    cudaError_t ea = cudaFuncSetAttribute(gemm_prep, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          kPrepMaxSmem);
    if (ea != cudaSuccess)
      return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemm: prep smem attribute: %s",
                             cudaGetErrorString(ea));
    prep_attr_done[dev & 7] = true;
  }
  {
    // as many CTAs as are resident at once (registers and shared memory),
    // each taking rows m = b, b + grid, ...
    int per_sm = 0;
    cudaError_t eo =
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gemm_prep, kPrepThreads, prep_smem);
    if (eo != cudaSuccess || per_sm < 1)
      return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemm: prep occupancy: %s",
                             cudaGetErrorString(eo));
    per_sm = std::min(8, per_sm);
    cfg.gridDim = dim3((unsigned)std::min<long long>(M, (long long)sms * per_sm));
  }
  cfg.blockDim = dim3(kPrepThreads);
  cfg.dynamicSmemBytes = prep_smem;
  cudaError_t e = cudaLaunchKernelEx(&cfg, gemm_prep, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemm: prep launch: %s", cudaGetErrorString(e));
  // The main kernel may launch while the pre-pass runs (programmatic
  // dependent launch): its set-up overlaps the pre-pass, and its producer
  // waits for the pre-pass before the first load of Xg.  It allocates all of
  // an SM's tensor memory, which is safe because two of its CTAs (197 KB of
  // shared memory each) never share an SM.
  cfg.gridDim = dim3((unsigned)(P.streamk ? sms : std::min(P.units, sms)));
  cfg.blockDim = dim3(kThreadsG);
  cfg.dynamicSmemBytes = smem;
  e = cudaLaunchKernelEx(&cfg, gemm_main, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemm: launch: %s", cudaGetErrorString(e));
  return POLYQ_OK;
}
