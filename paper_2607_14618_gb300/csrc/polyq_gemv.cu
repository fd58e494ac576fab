// Decode GEMV of the PolyQ mixed-bit layer (Section 4.1 factorisation with
// the Section 4.2 bit blocks), one pass over all blocks:
//
//   y[b][n] = residual[b][n] + sum_p x[b][gather[p]] * W'[n][p]
//
// Two kernels per call:
//  1. gemv_prep: for every step of every block, gathers the activations
//     through `gather`, lays them out in the order the main kernel decodes the
//     codes (scaled by the powers of two the decoder leaves on each code), and
//     sums them per chunk for the zero-point and magic-number corrections.
//  2. gemv_main: persistent CTAs; one producer warp streams 64-row tiles of
//     packed codes and scale/zero metadata with TMA into a 4-stage
//     shared-memory ring; four consumer warps turn each code pair into two
//     exact bf16 values 128 + q*2^p with a single LOP3 and multiply them with
//     the activations on the tensor cores (mma.sync m16n8k16, fp32
//     accumulation).  Each MMA column holds one 64-code chunk, so a chunk's
//     dot product is exact and its scale/zero are applied once:
//        y += s * (D - 128*sum(x') - z*sum(x)).
//     Every (tile, step) item writes a partial sum; the last item of a tile
//     to finish adds the partials in step order, so results do not depend on
//     scheduling or on where a row sits in the matrix.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "polyq.h"
#include "polyq_dev.cuh"
#include "polyq_gemv_layout.cuh"
#include "polyq_internal.h"

namespace {

using namespace polyq;
using namespace polyq::gv;

struct GvBlock {
  int bits, n_ch, pos0, seg_off, grp_off, n_grp;
  int step0, n_steps;  // global step range of this block
};

struct GvParams {
  CUtensorMap tm_codes[POLYQ_MAX_BLOCKS];
  CUtensorMap tm_meta;
  GvBlock blk[POLYQ_MAX_BLOCKS];
  int n_blocks;
  int N, K, S, G;
  int steps;       // steps per row (all blocks)
  int tiles;       // ceil(N / 64)
  int items;       // tiles * steps
  int batch;
  const __nv_bfloat16* x;
  const int32_t* gather;
  uint8_t* rec;          // steps * rec_bytes(NB)
  float* partial;        // items * 64 * NB
  uint32_t* counters;    // tiles * 4
  int* status;
  float* y;
  const float* residual;
};

__device__ __forceinline__ int find_block(const GvParams& P, int s) {
  int b = 0;
  while (b + 1 < P.n_blocks && s >= P.blk[b + 1].step0) ++b;
  return b;
}


__device__ __forceinline__ uint32_t float_to_bf16_bits(float f) {
  // values here are bf16 values scaled by powers of two: exact
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(f));
}

// ---------------------------------------------------------------------------
// pre-pass
// ---------------------------------------------------------------------------
template <int NB>
__global__ void __launch_bounds__(256) gemv_prep(const __grid_constant__ GvParams P) {
  pdl_trigger();
  pdl_wait();  // x comes from the previous kernel; the workspace may still be in use
  constexpr int CPL = cpl_of(NB);
  constexpr int NG = ng_of(NB);
  constexpr int U = units_of(NB);
  constexpr int LW = rec_lane_words(NB);
  __shared__ float xs_scaled[NB][U];
  __shared__ float xs_plain[NB][U];
  const int s = blockIdx.x;
  // zero the per-tile arrival counters (a grid-stride slice per CTA)
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < P.tiles * kWarps;
       i += gridDim.x * blockDim.x)
    P.counters[i] = 0u;
  if (blockIdx.x == 0 && threadIdx.x == 0) *P.status = 0;
  if (s >= P.steps) return;
  const int bi = find_block(P, s);
  const GvBlock B = P.blk[bi];
  const int j = s - B.step0;
  uint32_t* rec = reinterpret_cast<uint32_t*>(P.rec + (size_t)s * rec_bytes(NB));
  const int batch = P.batch;

  auto xval = [&](int b, int w) -> float {  // activation of block weight w
    if (b >= batch || w >= B.n_ch) return 0.f;
    const int p = B.pos0 + w;
    const int src = P.gather ? P.gather[p] : p;
    return __bfloat162float(P.x[(size_t)b * P.K + src]);
  };

  if (B.bits == 16) {
    for (int e = threadIdx.x; e < NB * 4 * 16; e += blockDim.x) {
      const int b = e / 64, t = (e / 16) % 4, k = e % 16;
      const int w0 = j * kU16 + lane_weight16(t, 2 * k);
      const int w1 = j * kU16 + lane_weight16(t, 2 * k + 1);
      const uint32_t lo = float_to_bf16_bits(xval(b, w0));
      const uint32_t hi = float_to_bf16_bits(xval(b, w1));
      rec[(b * 4 + t) * LW + k] = lo | (hi << 16);
    }
    return;
  }
  const bool nib = B.bits == 8;
  const int ub = ubits(B.bits);
  // one thread per (lane t, pair j) of the step
  for (int e = threadIdx.x; e < 4 * (CPL / 2); e += blockDim.x) {
    const int t = e / (CPL / 2), jp = e % (CPL / 2);
    int ulo, plo, uhi, phi;
    pair_units(ub, jp, &ulo, &plo, &uhi, &phi);
    const int su_lo = lane_unit(B.bits, NB, t, ulo);
    const int su_hi = lane_unit(B.bits, NB, t, uhi);
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      float v[2];
      const int su[2] = {su_lo, su_hi};
      const int pp[2] = {plo, phi};
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int gu = j * U + su[h];  // unit index inside the block
        float xv, scale = ldexpf(1.f, -pp[h]);
        if (nib) {
          xv = xval(b, gu >> 1);
          if (gu & 1) scale *= 16.f;
          xs_plain[b][su[h]] = (gu & 1) ? 0.f : xv;
        } else {
          xv = xval(b, gu);
          xs_plain[b][su[h]] = xv;
        }
        v[h] = xv * scale;
        xs_scaled[b][su[h]] = v[h];
      }
      rec[(b * 4 + t) * LW + jp] = float_to_bf16_bits(v[0]) | (float_to_bf16_bits(v[1]) << 16);
    }
  }
  __syncthreads();
  // per-chunk sums in a fixed order: C1 = 128 * sum x', X = sum x
  const int pw = rec_pair_words(NB);
  float* recf = reinterpret_cast<float*>(rec);
  for (int e = threadIdx.x; e < NB * NG; e += blockDim.x) {
    const int b = e / NG, c = e % NG;
    float c1 = 0.f, xx = 0.f;
    for (int u = 64 * c; u < 64 * c + 64; ++u) {
      c1 += xs_scaled[b][u];
      xx += xs_plain[b][u];
    }
    recf[pw + b * NG + c] = 128.f * c1;
    recf[pw + NB * NG + b * NG + c] = xx;
  }
}

// ---------------------------------------------------------------------------
// main kernel
// ---------------------------------------------------------------------------
template <int UB>
__device__ __forceinline__ uint32_t window(const uint32_t* w, int off) {
  // bits [off, off+32) of the little-endian stream held in w[]
  if (off < 0) return w[0] << (-off);
  const int k = off >> 5, r = off & 31;
  if (r == 0) return w[k];
  return __funnelshift_r(w[k], w[k + 1], r);
}

template <>
__device__ __forceinline__ uint32_t window<3>(const uint32_t* w, int off) {
  if (off < 0) return w[0] << (-off);
  const int k = off >> 5, r = off & 31;
  if (r == 0) return w[k];
  if (k == 2) return w[2] >> r;
  return __funnelshift_r(w[k], w[k + 1], r);
}

// Pair register for lane pair j from the lane's words of one row.
template <int UB>
__device__ __forceinline__ uint32_t make_pair(const uint32_t* words, int j) {
  constexpr int GP = group_pairs(UB);
  constexpr int GW = group_words(UB);
  const PairDef d = pair_def(UB, j % GP);
  const uint32_t* g = words + (j / GP) * GW;
  uint32_t win;
  if (UB == 3) {
    win = window<3>(g, d.win);
  } else {
    win = d.win ? (g[0] >> d.win) : g[0];
  }
  const uint32_t m = (((1u << UB) - 1u) << d.plo) | ((((1u << UB) - 1u) << d.phi) << 16);
  return lop3_and_or(win, m, 0x43004300u);
}

// Load the lane's words of tile row r from the stage's codes area.
template <int BITS, int NB>
__device__ __forceinline__ void load_words(uint32_t* w, const uint8_t* codes, int r, int t) {
  constexpr int H = halves(BITS, NB);
  constexpr int SB = step_bytes(BITS, NB);
  constexpr int NW = lane_words(BITS, NB);
  if (H) {
#pragma unroll
    for (int h = 0; h < H; ++h) {
      const uint4* p = reinterpret_cast<const uint4*>(codes + h * kRows * kPitchSplit +
                                                      r * kPitchSplit + 32 * t);
      const uint4 a = p[0], b = p[1];
      w[8 * h + 0] = a.x; w[8 * h + 1] = a.y; w[8 * h + 2] = a.z; w[8 * h + 3] = a.w;
      w[8 * h + 4] = b.x; w[8 * h + 5] = b.y; w[8 * h + 6] = b.z; w[8 * h + 7] = b.w;
    }
  } else {
    const uint8_t* p = codes + r * SB + t * (SB / 4);
    if constexpr ((SB / 4) % 16 == 0) {
#pragma unroll
      for (int k = 0; k < NW / 4; ++k) {
        const uint4 a = reinterpret_cast<const uint4*>(p)[k];
        w[4 * k] = a.x; w[4 * k + 1] = a.y; w[4 * k + 2] = a.z; w[4 * k + 3] = a.w;
      }
    } else if constexpr ((SB / 4) % 8 == 0) {
#pragma unroll
      for (int k = 0; k < NW / 2; ++k) {
        const uint2 a = reinterpret_cast<const uint2*>(p)[k];
        w[2 * k] = a.x; w[2 * k + 1] = a.y;
      }
    } else {
#pragma unroll
      for (int k = 0; k < NW; ++k) w[k] = reinterpret_cast<const uint32_t*>(p)[k];
    }
  }
}

// One MMA step of a b<16 block for this warp's 16 rows; adds the chunk
// results into acc[row][batch].
template <int NB, int BITS>
__device__ __forceinline__ void step_mma(const GvParams& P, const GvBlock& B, int j,
                                         const uint8_t* stage, const uint32_t* zero16,
                                         int warp, int lane, float (&acc)[2][NB]) {
  constexpr int UB = ubits(BITS);
  constexpr int CPL = cpl_of(NB);
  constexpr int NG = ng_of(NB);
  constexpr int NW = lane_words(BITS, NB);
  constexpr int NMMA = CPL / 4;
  constexpr int LW = rec_lane_words(NB);
  const int g = lane >> 2, t = lane & 3;
  const int rA = warp * 16 + g, rB = rA + 8;
  const uint8_t* codes = stage;
  const uint32_t* meta_s = reinterpret_cast<const uint32_t*>(stage + kCodesBytes);
  const uint32_t* rec = reinterpret_cast<const uint32_t*>(stage + kCodesBytes + kMetaBytes);

  uint32_t wa[NW], wb[NW];
  load_words<BITS, NB>(wa, codes, rA, t);
  load_words<BITS, NB>(wb, codes, rB, t);

  // B fragment source: this lane holds column n = g of B for k-slots of lane
  // t; it is non-zero only when column n is the chunk (and batch) that lane
  // t's pairs belong to.
  const int my_b = g / NG, my_c = g % NG;
  const bool b_ok = my_b < P.batch;
  const uint32_t* brow = rec + (my_b * 4 + t) * LW;

  float d[4][4];
#pragma unroll
  for (int q = 0; q < 4; ++q) d[q][0] = d[q][1] = d[q][2] = d[q][3] = 0.f;

#pragma unroll
  for (int i2 = 0; i2 < NMMA / 2; ++i2) {
    // two MMAs share one 16-byte activation load
    const int chunk = pair_chunk(BITS, NB, t, 4 * i2);
    const bool act = b_ok && (my_c == chunk);
    const uint4 bv = *reinterpret_cast<const uint4*>(act ? (brow + 4 * i2) : zero16);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = 2 * i2 + h;
      const uint32_t a0 = make_pair<UB>(wa, 2 * i);
      const uint32_t a1 = make_pair<UB>(wb, 2 * i);
      const uint32_t a2 = make_pair<UB>(wa, 2 * i + 1);
      const uint32_t a3 = make_pair<UB>(wb, 2 * i + 1);
      mma_bf16_16816(d[i & 3], a0, a1, a2, a3, h ? bv.z : bv.x, h ? bv.w : bv.y);
    }
  }
  float D[4];
#pragma unroll
  for (int v = 0; v < 4; ++v) D[v] = (d[0][v] + d[1][v]) + (d[2][v] + d[3][v]);

  // epilogue: columns 2t, 2t+1 -> batch be, chunks c0, c0+1
  const int be = (2 * t) / NG;
  if (be < P.batch) {
    const int c0 = (2 * t) % NG;
    const bool nib = BITS == 8;
    const int gfirst = B.grp_off + (nib ? (j * NG) / 2 : j * NG);
    const int x0 = gfirst & ~3;
    const float* recf = reinterpret_cast<const float*>(rec);
    constexpr int PW = rec_pair_words(NB);
#pragma unroll
    for (int cc = 0; cc < 2; ++cc) {
      const int c = c0 + cc;
      const int gi = B.grp_off + (nib ? (j * NG + c) / 2 : j * NG + c);
      const float C1 = recf[PW + be * NG + c];
      const float X = recf[PW + NB * NG + be * NG + c];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const uint32_t m = meta_s[(r ? rB : rA) * kMetaBox + (gi - x0)];
        const float sc = __half2float(__ushort_as_half((uint16_t)(m & 0xFFFFu)));
        const float ze = __half2float(__ushort_as_half((uint16_t)(m >> 16)));
        const float dot = D[2 * r + cc] - C1;
        const float v = sc * fmaf(-ze, X, dot);
#pragma unroll
        for (int b = 0; b < NB; ++b)
          if (b == be) acc[r][b] += v;
      }
    }
  }
}

// One 16-bit step (fp16 weights, CUDA-core FMAs).
template <int NB>
__device__ __forceinline__ void step_16(const GvParams& P, const uint8_t* stage, int warp,
                                        int lane, float (&acc)[2][NB]) {
  constexpr int LW = rec_lane_words(NB);
  const int g = lane >> 2, t = lane & 3;
  const int rA = warp * 16 + g, rB = rA + 8;
  const uint32_t* rec = reinterpret_cast<const uint32_t*>(stage + kCodesBytes + kMetaBytes);
  uint32_t wa[16], wb[16];
  load_words<16, NB>(wa, stage, rA, t);
  load_words<16, NB>(wb, stage, rB, t);
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    if (b >= P.batch) break;
    const uint32_t* xr = rec + (b * 4 + t) * LW;
    float sa = 0.f, sb = 0.f;
#pragma unroll
    for (int k4 = 0; k4 < 4; ++k4) {
      const uint4 xv = reinterpret_cast<const uint4*>(xr)[k4];
      const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int k = 4 * k4 + q;
        const float x0 = bf16_lo(xw[q]), x1 = bf16_hi(xw[q]);
        const float2 fa = __half22float2(*reinterpret_cast<const __half2*>(&wa[k]));
        const float2 fb = __half22float2(*reinterpret_cast<const __half2*>(&wb[k]));
        sa = fmaf(fa.x, x0, sa);
        sa = fmaf(fa.y, x1, sa);
        sb = fmaf(fb.x, x0, sb);
        sb = fmaf(fb.y, x1, sb);
      }
    }
    acc[0][b] += sa;
    acc[1][b] += sb;
  }
}

template <int NB>
__global__ void __launch_bounds__(160, 2) gemv_main(const __grid_constant__ GvParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* stages = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint32_t* zero16 = reinterpret_cast<uint32_t*>(bars + 2 * kStages);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kWarps);
    }
    mbar_fence_init();
  }
  if (threadIdx.x < 4) zero16[threadIdx.x] = 0u;
  __syncthreads();
  pdl_trigger();

  const int n_mine = P.items > (int)blockIdx.x
                         ? (P.items - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                         : 0;
  constexpr int RB = rec_bytes(NB);

  if (warp == kWarps) {
    // ---------------- producer ----------------
    if (lane != 0) return;
    for (int b = 0; b < P.n_blocks; ++b) prefetch_tmap(&P.tm_codes[b]);
    prefetch_tmap(&P.tm_meta);
    auto issue_weights = [&](int k, int slot) {
      const int item = blockIdx.x + k * gridDim.x;
      const int tile = item / P.steps, s = item % P.steps;
      const int bi = find_block(P, s);
      const GvBlock& B = P.blk[bi];
      const int j = s - B.step0;
      const uint32_t dst = smem_u32(stages + slot * kStageBytes);
      const uint32_t bar = full0 + 8 * slot;
      int sb, h;
      switch (B.bits) {
        case 2: sb = step_bytes(2, NB); h = halves(2, NB); break;
        case 3: sb = step_bytes(3, NB); h = halves(3, NB); break;
        case 4: sb = step_bytes(4, NB); h = halves(4, NB); break;
        case 8: sb = step_bytes(8, NB); h = halves(8, NB); break;
        default: sb = step_bytes(16, NB); h = halves(16, NB); break;
      }
      const int nbox = h ? h : 1;
      const int bw = h ? kPitchSplit : sb;
      uint32_t bytes = nbox * bw * kRows + RB;
      if (B.bits < 16) bytes += kMetaBytes;
      mbar_expect_tx(bar, bytes);
      for (int q = 0; q < nbox; ++q)
        tma_load_2d(dst + q * kRows * kPitchSplit, &P.tm_codes[bi], B.seg_off + j * sb + 128 * q,
                    tile * kRows, bar);
      if (B.bits < 16) {
        const int ngs = B.bits == 8 ? ng_of(NB) / 2 : ng_of(NB);
        const int x0 = (B.grp_off + j * ngs) & ~3;
        tma_load_2d(dst + kCodesBytes, &P.tm_meta, x0, tile * kRows, bar);
      }
    };
    auto issue_rec = [&](int k, int slot) {
      const int item = blockIdx.x + k * gridDim.x;
      const int s = item % P.steps;
      const uint32_t dst = smem_u32(stages + slot * kStageBytes + kCodesBytes + kMetaBytes);
      bulk_load(dst, P.rec + (size_t)s * RB, RB, full0 + 8 * slot);
    };
    const int pre = min(n_mine, kStages);
    for (int k = 0; k < pre; ++k) issue_weights(k, k);
    pdl_wait();  // activation records come from the pre-pass
    for (int k = 0; k < pre; ++k) issue_rec(k, k);
    for (int k = kStages; k < n_mine; ++k) {
      const int slot = k % kStages;
      const uint32_t par = ((k / kStages) - 1) & 1;
      if (!mbar_wait(empty0 + 8 * slot, par)) {
        atomicExch(P.status, kStatusTimeoutEmpty);
        break;
      }
      issue_weights(k, slot);
      issue_rec(k, slot);
    }
    return;
  }

  // ---------------- consumers ----------------
  pdl_wait();
  for (int k = 0; k < n_mine; ++k) {
    const int slot = k % kStages;
    const uint32_t par = (k / kStages) & 1;
    if (!mbar_wait(full0 + 8 * slot, par)) {
      if (lane == 0) atomicExch(P.status, kStatusTimeoutFull);
      return;
    }
    const int item = blockIdx.x + k * gridDim.x;
    const int tile = item / P.steps, s = item % P.steps;
    const int bi = find_block(P, s);
    const GvBlock B = P.blk[bi];
    const int j = s - B.step0;
    const uint8_t* stage = stages + slot * kStageBytes;
    float acc[2][NB];
#pragma unroll
    for (int r = 0; r < 2; ++r)
#pragma unroll
      for (int b = 0; b < NB; ++b) acc[r][b] = 0.f;
    switch (B.bits) {
      case 2: step_mma<NB, 2>(P, B, j, stage, zero16, warp, lane, acc); break;
      case 3: step_mma<NB, 3>(P, B, j, stage, zero16, warp, lane, acc); break;
      case 4: step_mma<NB, 4>(P, B, j, stage, zero16, warp, lane, acc); break;
      case 8: step_mma<NB, 8>(P, B, j, stage, zero16, warp, lane, acc); break;
      default: step_16<NB>(P, stage, warp, lane, acc); break;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty0 + 8 * slot);

    // sum over the four lanes of a row group
#pragma unroll
    for (int r = 0; r < 2; ++r)
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        float v = acc[r][b];
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 2);
        acc[r][b] = v;
      }
    const int g = lane >> 2, t = lane & 3;
    float* part = P.partial + ((size_t)item * kRows + warp * 16) * NB;
#pragma unroll
    for (int r = 0; r < 2; ++r)
#pragma unroll
      for (int b = 0; b < NB; ++b)
        if (b == t) part[(g + 8 * r) * NB + b] = acc[r][b];
    __threadfence();
    __syncwarp();
    uint32_t prev = 0;
    if (lane == 0) prev = atomicAdd(&P.counters[tile * kWarps + warp], 1u);
    prev = __shfl_sync(0xffffffffu, prev, 0);
    if (prev == (uint32_t)P.steps - 1) {
      // last step of this tile for this warp's rows: reduce in step order
      __threadfence();
      for (int e = lane; e < 16 * NB; e += 32) {
        const int row = e / NB, b = e % NB;
        const int n = tile * kRows + warp * 16 + row;
        float v = 0.f;
        for (int s2 = 0; s2 < P.steps; ++s2) {
          const size_t it = (size_t)tile * P.steps + s2;
          v += __ldcg(P.partial + (it * kRows + warp * 16 + row) * NB + b);
        }
        if (n < P.N && b < P.batch) {
          const size_t o = (size_t)b * P.N + n;
          P.y[o] = v + (P.residual ? P.residual[o] : 0.f);
        }
      }
      if (lane == 0) P.counters[tile * kWarps + warp] = 0u;
    }
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int nb_of(int batch) { return batch == 1 ? 1 : batch == 2 ? 2 : 4; }

struct Geometry {
  int steps = 0, tiles = 0, items = 0, nb = 1;
  GvBlock blk[POLYQ_MAX_BLOCKS];
  size_t rec_off = 0, part_off = 0, cnt_off = 0, status_off = 0, total = 0;
};

int geometry(const polyq_dev_layer* L, int batch, Geometry* G) {
  G->nb = nb_of(batch);
  const int nb = G->nb;
  int s = 0;
  for (int i = 0; i < L->n_blocks; ++i) {
    const polyq_block& b = L->blocks[i];
    GvBlock& g = G->blk[i];
    g.bits = b.bits;
    g.n_ch = b.n_ch;
    g.pos0 = b.pos0;
    g.seg_off = b.seg_off;
    g.grp_off = b.grp_off;
    g.n_grp = b.n_grp;
    g.step0 = s;
    const int per = b.bits == 16 ? kU16 : (b.bits == 8 ? units_of(nb) / 2 : units_of(nb));
    g.n_steps = (b.n_ch + per - 1) / per;
    s += g.n_steps;
  }
  G->steps = s;
  G->tiles = (int)((L->N + kRows - 1) / kRows);
  G->items = G->tiles * s;
  auto al = [](size_t v) { return (v + 255) / 256 * 256; };
  G->rec_off = 0;
  G->part_off = al((size_t)s * rec_bytes(nb));
  G->cnt_off = al(G->part_off + (size_t)G->items * kRows * nb * 4);
  G->status_off = al(G->cnt_off + (size_t)G->tiles * kWarps * 4);
  G->total = G->status_off + 256;
  return POLYQ_OK;
}

template <int NB>
int launch(const polyq_dev_layer* L, const Geometry& G, GvParams& P, cudaStream_t st) {
  static bool attr_done[8] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  const size_t smem = (size_t)kStages * kStageBytes + 2 * kStages * 8 + 16;
  if (!attr_done[dev & 7]) {
    cudaError_t e = cudaFuncSetAttribute(gemv_main<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess)
      return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemv: smem attribute: %s",
                             cudaGetErrorString(e));
    attr_done[dev & 7] = true;
  }
  int sms = 0;
  int rc = polyq_sm_count(&sms);
  if (rc) return rc;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;

  cudaLaunchConfig_t cfg = {};
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3((unsigned)std::max(G.steps, 1));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, gemv_prep<NB>, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemv: prep launch: %s", cudaGetErrorString(e));

  cfg.gridDim = dim3((unsigned)std::min(G.items, 2 * sms));
  cfg.blockDim = dim3(32 * (kWarps + 1));
  cfg.dynamicSmemBytes = smem;
  e = cudaLaunchKernelEx(&cfg, gemv_main<NB>, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemv: launch: %s", cudaGetErrorString(e));
  return POLYQ_OK;
}

}  // namespace

extern "C" int polyq_gemv_workspace_bytes(const polyq_dev_layer* L, int batch, size_t* bytes) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_gemv_workspace_bytes");
  if (rc) return rc;
  if (!bytes) return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_workspace_bytes: bytes is NULL");
  if (batch < 1 || batch > 4)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_gemv_workspace_bytes: batch %d", batch);
  Geometry G;
  geometry(L, batch, &G);
  *bytes = G.total;
  return POLYQ_OK;
}

extern "C" int polyq_linear_gemv(const polyq_dev_layer* L, const void* x, int batch, float* y,
                                 const float* residual, void* workspace, size_t ws_bytes,
                                 void* stream) {
  polyq_clear_error();
  int rc = polyq_check_dev_layer(L, "polyq_linear_gemv");
  if (rc) return rc;
  if (!x || !y) return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemv: x or y is NULL");
  if (batch < 1 || batch > 4)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_linear_gemv: batch %d not in 1..4", batch);
  Geometry G;
  geometry(L, batch, &G);
  if (!workspace || ws_bytes < G.total)
    return polyq_set_error(POLYQ_ENOMEM, "polyq_linear_gemv: workspace needs %zu bytes, got %zu",
                           G.total, ws_bytes);
  if ((uintptr_t)workspace % 256)
    return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemv: workspace must be 256-byte aligned");

  GvParams P;
  memset(&P, 0, sizeof P);
  for (int i = 0; i < L->n_blocks; ++i) {
    const int bits = L->blocks[i].bits;
    const int nb = G.nb;
    const int h = halves(bits, nb);
    const int bw = h ? kPitchSplit : step_bytes(bits, nb);
    rc = polyq_tensor_map_2d(&P.tm_codes[i], L->packed, 1, (uint64_t)L->row_stride,
                             (uint64_t)L->N, (uint64_t)L->row_stride, (uint32_t)bw, kRows);
    if (rc) return rc;
    P.blk[i] = G.blk[i];
  }
  if (L->n_groups > 0) {
    rc = polyq_tensor_map_2d(&P.tm_meta, L->meta, 4, (uint64_t)L->meta_stride, (uint64_t)L->N,
                             (uint64_t)L->meta_stride * 4, kMetaBox, kRows);
    if (rc) return rc;
  }
  P.n_blocks = L->n_blocks;
  P.N = (int)L->N;
  P.K = (int)L->K;
  P.S = (int)L->row_stride;
  P.G = (int)L->n_groups;
  P.steps = G.steps;
  P.tiles = G.tiles;
  P.items = G.items;
  P.batch = batch;
  P.x = (const __nv_bfloat16*)x;
  P.gather = L->gather;
  uint8_t* ws = (uint8_t*)workspace;
  P.rec = ws + G.rec_off;
  P.partial = (float*)(ws + G.part_off);
  P.counters = (uint32_t*)(ws + G.cnt_off);
  P.status = (int*)(ws + G.status_off);
  P.y = y;
  P.residual = residual;
  cudaStream_t st = (cudaStream_t)stream;
  switch (G.nb) {
    case 1: return launch<1>(L, G, P, st);
    case 2: return launch<2>(L, G, P, st);
    default: return launch<4>(L, G, P, st);
  }
}
