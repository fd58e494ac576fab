// Decode GEMV of the PolyQ mixed-bit layer (Section 4.1 factorisation with
// the Section 4.2 bit blocks), one pass over all blocks of one or several
// independent layers:
//
//   y[b][n] = residual[b][n] + sum_p x[b][gather[p]] * W'[n][p]
//
// Two kernels per call:
//  1. gemv_prep: for every step of every block, gathers the activations
//     through `gather`, lays them out in the order the main kernel decodes the
//     codes (scaled by the powers of two the decoder leaves on each code), sums
//     them per chunk for the zero-point and magic-number corrections, and sets
//     y to the residual (or zero).
//  2. gemv_main: persistent CTAs; one producer warp streams 64-row tiles of
//     packed codes and scale/zero metadata with TMA into a 3-stage
//     shared-memory ring; four consumer warps turn each code pair into two
//     exact bf16 values 128 + q*2^p with a single LOP3 and multiply them with
//     the activations on the tensor cores (mma.sync m16n8k16, fp32
//     accumulation).  Each MMA column holds one 64-code chunk, so a chunk's
//     dot product is exact and its scale/zero are applied once:
//        y += s * (D - 128*sum(x') - z*sum(x)).
//     The (layer, tile, step) items of all layers of a call form one list;
//     each CTA takes a contiguous range and keeps row sums in registers across
//     a tile's steps.  A tile split between CTAs gets one fp32 atomic addition
//     per piece into y, so the order of those few additions is not fixed from
//     run to run.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "polyq.h"
#include "polyq_dev.cuh"
#include "polyq_gemv_layout.cuh"
#include "polyq_internal.h"

namespace {

using namespace polyq;
using namespace polyq::gv;

constexpr int kCtasPerSm = 3;
constexpr int kMaxGrid = 1024;  // persistent CTAs at most

struct GvBlock {
  int bits, n_ch, pos0, seg_off, grp_off, n_grp;
  int step0, n_steps;  // step range of this block inside its layer
};

// One layer of a call.  Tensor maps first (64-byte aligned).
struct GvLayer {
  CUtensorMap tm_codes[POLYQ_MAX_BLOCKS];
  CUtensorMap tm_meta;
  GvBlock blk[POLYQ_MAX_BLOCKS];
  int n_blocks;
  int N, K;
  int steps;      // steps per row
  int items;      // tiles * steps
  int item0;      // first item of this layer in the call's list
  int rec0;       // first record of this layer
  const __nv_bfloat16* x;
  const int32_t* gather;
  float* y;
  const float* residual;
};

struct GvParams {
  GvLayer L[POLYQ_MAX_GROUP];
  int n_layers;
  int items;       // all layers
  int recs;        // all layers' steps
  int batch;
  uint32_t magic;  // 0x43004300 (two bf16 128.0), kept in a register
  uint8_t* rec;    // recs * rec_bytes(NB)
  int* status;
};

// Per-CTA shared copy of the scalars and block tables (runtime-indexed reads
// of kernel parameters would become slow generic loads).
struct GvShared {
  GvBlock blk[POLYQ_MAX_GROUP][POLYQ_MAX_BLOCKS];
  int n_blocks[POLYQ_MAX_GROUP];
  int N[POLYQ_MAX_GROUP];
  int steps[POLYQ_MAX_GROUP];
  int item0[POLYQ_MAX_GROUP + 1];
  int rec0[POLYQ_MAX_GROUP];
};

__device__ __forceinline__ void load_shared(const GvParams& P, GvShared* S) {
  // constant-offset parameter reads only
#pragma unroll
  for (int l = 0; l < POLYQ_MAX_GROUP; ++l) {
    if (l >= P.n_layers) break;
    if (threadIdx.x < POLYQ_MAX_BLOCKS) {
#pragma unroll
      for (int b = 0; b < POLYQ_MAX_BLOCKS; ++b)
        if (b == (int)threadIdx.x) S->blk[l][b] = P.L[l].blk[b];
    }
    if (threadIdx.x == 0) {
      S->n_blocks[l] = P.L[l].n_blocks;
      S->N[l] = P.L[l].N;
      S->steps[l] = P.L[l].steps;
      S->item0[l] = P.L[l].item0;
      S->rec0[l] = P.L[l].rec0;
    }
  }
  if (threadIdx.x == 0) S->item0[P.n_layers] = P.items;
}

__device__ __forceinline__ int find_block(const GvBlock* blk, int nblk, int s) {
  int b = 0;
  while (b + 1 < nblk && s >= blk[b + 1].step0) ++b;
  return b;
}

__device__ __forceinline__ int find_layer(const int* starts, int nl, int v) {
  int l = 0;
  while (l + 1 < nl && v >= starts[l + 1]) ++l;
  return l;
}

__device__ __forceinline__ uint32_t float_to_bf16_bits(float f) {
  // values here are bf16 values scaled by powers of two: exact
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(f));
}

// ---------------------------------------------------------------------------
// pre-pass: one CTA per step of every layer
// ---------------------------------------------------------------------------
template <int NB>
__global__ void __launch_bounds__(256) gemv_prep(const __grid_constant__ GvParams P) {
  pdl_trigger();
  pdl_wait();  // x comes from the previous kernel; y and the workspace may still be in use
  constexpr int CPL = cpl_of(NB);
  constexpr int NG = ng_of(NB);
  constexpr int U = units_of(NB);
  constexpr int LW = rec_lane_words(NB);
  __shared__ float xs_scaled[NB][U];
  __shared__ float xs_plain[NB][U];
  __shared__ GvShared S;
  load_shared(P, &S);
  __syncthreads();
  const int nl = P.n_layers;
  const int batch = P.batch;

  // y starts as the residual (or zero); the main kernel adds its pieces
#pragma unroll
  for (int l = 0; l < POLYQ_MAX_GROUP; ++l) {
    if (l >= nl) break;
    float* y = P.L[l].y;
    const float* res = P.L[l].residual;
    if (y == res) continue;
    const int total = batch * P.L[l].N;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x)
      y[i] = res ? res[i] : 0.f;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) *P.status = 0;

  const int r = blockIdx.x;  // record index
  if (r >= P.recs) return;
  const int l = find_layer(S.rec0, nl, r);
  const int s = r - S.rec0[l];
  const int bi = find_block(S.blk[l], S.n_blocks[l], s);
  const GvBlock B = S.blk[l][bi];
  const int j = s - B.step0;
  uint32_t* rec = reinterpret_cast<uint32_t*>(P.rec + (size_t)r * rec_bytes(NB));
  const __nv_bfloat16* x = nullptr;
  const int32_t* gather = nullptr;
  int K = 0;
#pragma unroll
  for (int q = 0; q < POLYQ_MAX_GROUP; ++q)
    if (q == l) {
      x = P.L[q].x;
      gather = P.L[q].gather;
      K = P.L[q].K;
    }

  auto xval = [&](int b, int w) -> float {  // activation of block weight w
    if (b >= batch || w >= B.n_ch) return 0.f;
    const int p = B.pos0 + w;
    const int src = gather ? gather[p] : p;
    return __bfloat162float(x[(size_t)b * K + src]);
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
    const int su[2] = {lane_unit(B.bits, NB, t, ulo), lane_unit(B.bits, NB, t, uhi)};
    const int pp[2] = {plo, phi};
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      float v[2];
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
  if (UB == 3 && k == 2) return w[2] >> r;
  return __funnelshift_r(w[k], w[k + 1], r);
}

// Pair register for lane pair j from the lane's words of one row.  `magic` is
// 0x43004300 and lives in a register, so each pair costs one LOP3 with the
// mask as its immediate operand (plus the shift of its window, shared by the
// pairs that use the same window).
template <int UB>
__device__ __forceinline__ uint32_t make_pair(const uint32_t* words, int j, uint32_t magic) {
  constexpr int GP = group_pairs(UB);
  constexpr int GW = group_words(UB);
  const PairDef d = pair_def(UB, j % GP);
  const uint32_t* g = words + (j / GP) * GW;
  const uint32_t win = UB == 3 ? window<3>(g, d.win) : (d.win ? (g[0] >> d.win) : g[0]);
  const uint32_t m = (((1u << UB) - 1u) << d.plo) | ((((1u << UB) - 1u) << d.phi) << 16);
  return (win & m) | magic;
}

// Load the lane's words of tile row r from the stage's codes area (box h at
// h * 64 rows * pitch, row r at r * pitch, lane t at t * LB).
template <int BITS, int NB>
__device__ __forceinline__ void load_words(uint32_t* w, const uint8_t* codes, int r, int t) {
  constexpr int NBX = nbox_of(BITS, NB);
  constexpr int PITCH = box_pitch(BITS, NB);
  constexpr int LB = lane_box_bytes(BITS, NB);
  constexpr int WPB = LB / 4;
#pragma unroll
  for (int h = 0; h < NBX; ++h) {
    const uint8_t* p = codes + h * kRows * PITCH + r * PITCH + t * LB;
    uint32_t* o = w + h * WPB;
    if constexpr (LB % 16 == 0) {
#pragma unroll
      for (int k = 0; k < WPB / 4; ++k) {
        const uint4 a = reinterpret_cast<const uint4*>(p)[k];
        o[4 * k] = a.x; o[4 * k + 1] = a.y; o[4 * k + 2] = a.z; o[4 * k + 3] = a.w;
      }
    } else if constexpr (LB % 8 == 0) {
#pragma unroll
      for (int k = 0; k < WPB / 2; ++k) {
        const uint2 a = reinterpret_cast<const uint2*>(p)[k];
        o[2 * k] = a.x; o[2 * k + 1] = a.y;
      }
    } else {
#pragma unroll
      for (int k = 0; k < WPB; ++k) o[k] = reinterpret_cast<const uint32_t*>(p)[k];
    }
  }
}

// One MMA step of a b<16 block for this warp's 16 rows; adds the chunk
// results into acc[row][batch].
//
// The lane's codes come in groups (one word for 2/4-bit, three words for
// 3-bit); group q yields GP pairs = GP/2 MMAs.  Groups are visited in
// increasing unit order, so the first group that starts past the block's last
// code ends the step for the whole warp.
template <int NB, int BITS>
__device__ __forceinline__ void step_mma(const GvParams& P, const GvBlock& B, int j,
                                         const uint8_t* stage, const uint32_t* zero16,
                                         int warp, int lane, float (&acc)[2][NB]) {
  constexpr int UB = ubits(BITS);
  constexpr int NG = ng_of(NB);
  constexpr int NW = lane_words(BITS, NB);
  constexpr int LW = rec_lane_words(NB);
  constexpr int GP = group_pairs(UB), GU = group_units(UB), GW = group_words(UB);
  constexpr int NGRP = NW / GW;
  constexpr int NACC = 8;
  const int g = lane >> 2, t = lane & 3;
  const int rA = warp * 16 + g, rB = rA + 8;
  const uint32_t* meta_s = reinterpret_cast<const uint32_t*>(stage + kCodesBytes);
  const uint32_t* rec = reinterpret_cast<const uint32_t*>(stage + kCodesBytes + kMetaBytes);

  const uint32_t magic = P.magic;
  uint32_t wa[NW], wb[NW];
  load_words<BITS, NB>(wa, stage, rA, t);
  load_words<BITS, NB>(wb, stage, rB, t);

  // This lane holds column n = g of the B fragment for lane t's k-slots; the
  // column is non-zero only for the chunk (and batch) that the group of lane t
  // belongs to.  The chunk of group q is the lane's first chunk + a constant.
  const int my_b = g / NG, my_c = g % NG;
  const uint32_t* brow = rec + (my_b * 4 + t) * LW;
  const int dc = my_b < P.batch ? my_c - lane_unit(BITS, NB, t, 0) / 64 : -1000;

  const int per_step = units_of(NB);
  const int u_valid = min(per_step, (B.n_ch - j * (BITS == 8 ? per_step / 2 : per_step)) *
                                        (BITS == 8 ? 2 : 1));
  float d[NACC][4];
#pragma unroll
  for (int q = 0; q < NACC; ++q) d[q][0] = d[q][1] = d[q][2] = d[q][3] = 0.f;

#pragma unroll
  for (int q = 0; q < NGRP; ++q) {
    if (lane_unit(BITS, NB, 0, q * GU) >= u_valid) break;
    const int coff = lane_unit(BITS, NB, 0, q * GU) / 64 - lane_unit(BITS, NB, 0, 0) / 64;
    const uint32_t* bsrc = dc == coff ? brow + q * GP : zero16;
    const int bstep = dc == coff ? 4 : 0;
#pragma unroll
    for (int m2 = 0; m2 < GP / 4; ++m2) {  // two MMAs per 16-byte activation load
      const uint4 bv = *reinterpret_cast<const uint4*>(bsrc + m2 * bstep);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int jp = q * GP + 4 * m2 + 2 * h;  // lane pair index
        const uint32_t a0 = make_pair<UB>(wa, jp, magic);
        const uint32_t a1 = make_pair<UB>(wb, jp, magic);
        const uint32_t a2 = make_pair<UB>(wa, jp + 1, magic);
        const uint32_t a3 = make_pair<UB>(wb, jp + 1, magic);
        mma_bf16_16816(d[(jp / 2) % NACC], a0, a1, a2, a3, h ? bv.z : bv.x, h ? bv.w : bv.y);
      }
    }
  }
  float D[4];
#pragma unroll
  for (int v = 0; v < 4; ++v)
    D[v] = ((d[0][v] + d[1][v]) + (d[2][v] + d[3][v])) +
           ((d[4][v] + d[5][v]) + (d[6][v] + d[7][v]));

  // epilogue: columns 2t, 2t+1 -> batch be, chunks c0, c0+1
  const int be = (2 * t) / NG;
  if (be < P.batch) {
    const int c0 = (2 * t) % NG;
    constexpr bool nib = BITS == 8;
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
        const float v = sc * fmaf(-ze, X, D[2 * r + cc] - C1);
#pragma unroll
        for (int b = 0; b < NB; ++b)
          if (b == be) acc[r][b] += v;
      }
    }
  }
}

// One 16-bit step (fp16 weights, CUDA-core FMAs).  Lane t holds weights
// [16t, 16t+16) of each 64-weight half; the second half is skipped when the
// block ends in the first.
template <int NB>
__device__ __forceinline__ void step_16(const GvParams& P, const GvBlock& B, int j,
                                        const uint8_t* stage, int warp, int lane,
                                        float (&acc)[2][NB]) {
  constexpr int LW = rec_lane_words(NB);
  constexpr int PITCH = box_pitch(16, NB);
  const int g = lane >> 2, t = lane & 3;
  const int rA = warp * 16 + g, rB = rA + 8;
  const uint32_t* rec = reinterpret_cast<const uint32_t*>(stage + kCodesBytes + kMetaBytes);
  const int halves_used = (B.n_ch - j * kU16) > 64 ? 2 : 1;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    if (h >= halves_used) break;
    uint32_t wa[8], wb[8];
    {
      const uint4* pa = reinterpret_cast<const uint4*>(stage + h * kRows * PITCH + rA * PITCH + 32 * t);
      const uint4* pb = reinterpret_cast<const uint4*>(stage + h * kRows * PITCH + rB * PITCH + 32 * t);
      const uint4 a0 = pa[0], a1 = pa[1], b0 = pb[0], b1 = pb[1];
      wa[0] = a0.x; wa[1] = a0.y; wa[2] = a0.z; wa[3] = a0.w;
      wa[4] = a1.x; wa[5] = a1.y; wa[6] = a1.z; wa[7] = a1.w;
      wb[0] = b0.x; wb[1] = b0.y; wb[2] = b0.z; wb[3] = b0.w;
      wb[4] = b1.x; wb[5] = b1.y; wb[6] = b1.z; wb[7] = b1.w;
    }
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      if (b >= P.batch) break;
      const uint32_t* xr = rec + (b * 4 + t) * LW + 8 * h;
      float sa = 0.f, sb = 0.f;
#pragma unroll
      for (int k2 = 0; k2 < 2; ++k2) {
        const uint4 xv = reinterpret_cast<const uint4*>(xr)[k2];
        const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int k = 4 * k2 + q;
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
}

template <int NB>
__global__ void __launch_bounds__(160, 3) gemv_main(const __grid_constant__ GvParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* stages = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint32_t* zero16 = reinterpret_cast<uint32_t*>(bars + 2 * kStages);
  __shared__ GvShared S;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);

  load_shared(P, &S);
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
  const int nl = P.n_layers;

  // contiguous range of (layer, tile, step) items
  const long long I = P.items, C = gridDim.x;
  const int lo = (int)((long long)blockIdx.x * I / C);
  const int hi = (int)((long long)(blockIdx.x + 1) * I / C);
  const int n_mine = hi - lo;
  constexpr int RB = rec_bytes(NB);

  if (warp == kWarps) {
    // ---------------- producer ----------------
    if (lane != 0) return;
    for (int l = 0; l < nl; ++l) {
      for (int b = 0; b < S.n_blocks[l]; ++b) prefetch_tmap(&P.L[l].tm_codes[b]);
      prefetch_tmap(&P.L[l].tm_meta);
    }
    auto issue_weights = [&](int k, int slot) {
      const int item = lo + k;
      const int l = find_layer(S.item0, nl, item);
      const int li = item - S.item0[l];
      const int steps = S.steps[l];
      const int tile = li / steps, s = li - tile * steps;
      const int bi = find_block(S.blk[l], S.n_blocks[l], s);
      const GvBlock& B = S.blk[l][bi];
      const int j = s - B.step0;
      const uint32_t dst = smem_u32(stages + slot * kStageBytes);
      const uint32_t bar = full0 + 8 * slot;
      int sb, nbx, pitch;
      switch (B.bits) {
        case 2: sb = step_bytes(2, NB); nbx = nbox_of(2, NB); pitch = box_pitch(2, NB); break;
        case 3: sb = step_bytes(3, NB); nbx = nbox_of(3, NB); pitch = box_pitch(3, NB); break;
        case 4: sb = step_bytes(4, NB); nbx = nbox_of(4, NB); pitch = box_pitch(4, NB); break;
        case 8: sb = step_bytes(8, NB); nbx = nbox_of(8, NB); pitch = box_pitch(8, NB); break;
        default: sb = step_bytes(16, NB); nbx = nbox_of(16, NB); pitch = box_pitch(16, NB); break;
      }
      uint32_t bytes = nbx * pitch * kRows + RB;
      if (B.bits < 16) bytes += kMetaBytes;
      mbar_expect_tx(bar, bytes);
      const CUtensorMap* tm = &P.L[l].tm_codes[bi];
      for (int q = 0; q < nbx; ++q)
        tma_load_2d(dst + q * kRows * pitch, tm, B.seg_off + j * sb + q * (sb / nbx), tile * kRows,
                    bar);
      if (B.bits < 16) {
        const int ngs = B.bits == 8 ? ng_of(NB) / 2 : ng_of(NB);
        const int x0 = (B.grp_off + j * ngs) & ~3;
        tma_load_2d(dst + kCodesBytes, &P.L[l].tm_meta, x0, tile * kRows, bar);
      }
    };
    auto issue_rec = [&](int k, int slot) {
      const int item = lo + k;
      const int l = find_layer(S.item0, nl, item);
      const int s = (item - S.item0[l]) % S.steps[l];
      const uint32_t dst = smem_u32(stages + slot * kStageBytes + kCodesBytes + kMetaBytes);
      bulk_load(dst, P.rec + (size_t)(S.rec0[l] + s) * RB, RB, full0 + 8 * slot);
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
  const int g = lane >> 2, t = lane & 3;
  float acc[2][NB];
#pragma unroll
  for (int r = 0; r < 2; ++r)
#pragma unroll
    for (int b = 0; b < NB; ++b) acc[r][b] = 0.f;
  for (int k = 0; k < n_mine; ++k) {
    const int slot = k % kStages;
    const uint32_t par = (k / kStages) & 1;
    if (!mbar_wait(full0 + 8 * slot, par)) {
      if (lane == 0) atomicExch(P.status, kStatusTimeoutFull);
      return;
    }
    const int item = lo + k;
    const int l = find_layer(S.item0, nl, item);
    const int li = item - S.item0[l];
    const int steps = S.steps[l];
    const int tile = li / steps, s = li - tile * steps;
    const int bi = find_block(S.blk[l], S.n_blocks[l], s);
    const GvBlock B = S.blk[l][bi];
    const int j = s - B.step0;
    const uint8_t* stage = stages + slot * kStageBytes;
    switch (B.bits) {
      case 2: step_mma<NB, 2>(P, B, j, stage, zero16, warp, lane, acc); break;
      case 3: step_mma<NB, 3>(P, B, j, stage, zero16, warp, lane, acc); break;
      case 4: step_mma<NB, 4>(P, B, j, stage, zero16, warp, lane, acc); break;
      case 8: step_mma<NB, 8>(P, B, j, stage, zero16, warp, lane, acc); break;
      default: step_16<NB>(P, B, j, stage, warp, lane, acc); break;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty0 + 8 * slot);
    if (s != steps - 1 && k != n_mine - 1) continue;

    // ---- flush this warp's 16 rows of `tile` of layer l ----
    // Sum the four lanes of each row, then add the piece into y.  A tile whose
    // steps are split over CTAs receives one addition per piece.
#pragma unroll
    for (int r = 0; r < 2; ++r)
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        float v = acc[r][b];
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 2);
        acc[r][b] = v;
      }
    float* y = nullptr;
#pragma unroll
    for (int q = 0; q < POLYQ_MAX_GROUP; ++q)
      if (q == l) y = P.L[q].y;
    const int N = S.N[l];
#pragma unroll
    for (int r = 0; r < 2; ++r)
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        const int n = tile * kRows + warp * 16 + g + 8 * r;
        if (b == t && b < P.batch && n < N) atomicAdd(y + (size_t)b * N + n, acc[r][b]);
        acc[r][b] = 0.f;
      }
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int nb_of(int batch) { return batch == 1 ? 1 : batch == 2 ? 2 : 4; }

int steps_of(const polyq_dev_layer* L, int nb, GvBlock* blk) {
  int s = 0;
  for (int i = 0; i < L->n_blocks; ++i) {
    const polyq_block& b = L->blocks[i];
    GvBlock g;
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
    if (blk) blk[i] = g;
  }
  return s;
}

size_t workspace_for(const polyq_dev_layer* const* L, int n, int batch) {
  const int nb = nb_of(batch);
  size_t recs = 0;
  for (int i = 0; i < n; ++i) recs += (size_t)steps_of(L[i], nb, nullptr);
  return (recs * rec_bytes(nb) + 255) / 256 * 256 + 256;  // records + status word
}

int check_group(const char* who, const polyq_dev_layer* const* L, int n, int batch) {
  if (!L || n < 1 || n > POLYQ_MAX_GROUP)
    return polyq_set_error(POLYQ_EINVAL, "%s: need 1..%d layers", who, POLYQ_MAX_GROUP);
  if (batch < 1 || batch > 4)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "%s: batch %d not in 1..4", who, batch);
  for (int i = 0; i < n; ++i) {
    int rc = polyq_check_dev_layer(L[i], who);
    if (rc) return rc;
  }
  return POLYQ_OK;
}

template <int NB>
int launch(const GvParams& P, int recs, cudaStream_t st) {
  static bool attr_done[8] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  const size_t smem = (size_t)kStages * kStageBytes + 2 * kStages * 8 + 16;
  if (!attr_done[dev & 7]) {
    cudaError_t e = cudaFuncSetAttribute(gemv_main<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess)
      return polyq_set_error(POLYQ_ECUDA, "polyq gemv: smem attribute: %s", cudaGetErrorString(e));
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
  cfg.gridDim = dim3((unsigned)std::max(recs, 1));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, gemv_prep<NB>, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq gemv: prep launch: %s", cudaGetErrorString(e));

  cfg.gridDim = dim3((unsigned)std::min(std::min(P.items, kCtasPerSm * sms), kMaxGrid));
  cfg.blockDim = dim3(32 * (kWarps + 1));
  cfg.dynamicSmemBytes = smem;
  e = cudaLaunchKernelEx(&cfg, gemv_main<NB>, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq gemv: launch: %s", cudaGetErrorString(e));
  return POLYQ_OK;
}

int gemv_group(const char* who, const polyq_dev_layer* const* L, int n, const void* const* xs,
               int batch, float* const* ys, const float* const* res, void* workspace,
               size_t ws_bytes, cudaStream_t st) {
  int rc = check_group(who, L, n, batch);
  if (rc) return rc;
  if (!xs || !ys) return polyq_set_error(POLYQ_EINVAL, "%s: x or y is NULL", who);
  for (int i = 0; i < n; ++i)
    if (!xs[i] || !ys[i]) return polyq_set_error(POLYQ_EINVAL, "%s: x or y %d is NULL", who, i);
  const size_t need = workspace_for(L, n, batch);
  if (!workspace || ws_bytes < need)
    return polyq_set_error(POLYQ_ENOMEM, "%s: workspace needs %zu bytes, got %zu", who, need,
                           ws_bytes);
  if ((uintptr_t)workspace % 256)
    return polyq_set_error(POLYQ_EINVAL, "%s: workspace must be 256-byte aligned", who);
  const int nb = nb_of(batch);
  GvParams P;
  memset(&P, 0, sizeof P);
  int items = 0, recs = 0;
  for (int i = 0; i < n; ++i) {
    GvLayer& G = P.L[i];
    const polyq_dev_layer* D = L[i];
    const int steps = steps_of(D, nb, G.blk);
    for (int b = 0; b < D->n_blocks; ++b) {
      const int bw = box_pitch(D->blocks[b].bits, nb);
      rc = polyq_tensor_map_2d(&G.tm_codes[b], D->packed, 1, (uint64_t)D->row_stride,
                               (uint64_t)D->N, (uint64_t)D->row_stride, (uint32_t)bw, kRows);
      if (rc) return rc;
    }
    if (D->n_groups > 0) {
      rc = polyq_tensor_map_2d(&G.tm_meta, D->meta, 4, (uint64_t)D->meta_stride, (uint64_t)D->N,
                               (uint64_t)D->meta_stride * 4, kMetaBox, kRows);
      if (rc) return rc;
    }
    G.n_blocks = D->n_blocks;
    G.N = (int)D->N;
    G.K = (int)D->K;
    G.steps = steps;
    G.items = (int)((D->N + kRows - 1) / kRows) * steps;
    G.item0 = items;
    G.rec0 = recs;
    G.x = (const __nv_bfloat16*)xs[i];
    G.gather = D->gather;
    G.y = ys[i];
    G.residual = res ? res[i] : nullptr;
    items += G.items;
    recs += steps;
  }
  P.n_layers = n;
  P.items = items;
  P.recs = recs;
  P.batch = batch;
  P.magic = 0x43004300u;
  P.rec = (uint8_t*)workspace;
  P.status = (int*)((uint8_t*)workspace + need - 256);
  switch (nb) {
    case 1: return launch<1>(P, recs, st);
    case 2: return launch<2>(P, recs, st);
    default: return launch<4>(P, recs, st);
  }
}

}  // namespace

extern "C" int polyq_gemv_workspace_bytes(const polyq_dev_layer* L, int batch, size_t* bytes) {
  polyq_clear_error();
  const polyq_dev_layer* one[1] = {L};
  int rc = check_group("polyq_gemv_workspace_bytes", one, 1, batch);
  if (rc) return rc;
  if (!bytes) return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_workspace_bytes: bytes is NULL");
  *bytes = workspace_for(one, 1, batch);
  return POLYQ_OK;
}

extern "C" int polyq_gemv_group_workspace_bytes(const polyq_dev_layer* const* layers, int n,
                                                int batch, size_t* bytes) {
  polyq_clear_error();
  int rc = check_group("polyq_gemv_group_workspace_bytes", layers, n, batch);
  if (rc) return rc;
  if (!bytes)
    return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_group_workspace_bytes: bytes is NULL");
  *bytes = workspace_for(layers, n, batch);
  return POLYQ_OK;
}

extern "C" int polyq_linear_gemv(const polyq_dev_layer* L, const void* x, int batch, float* y,
                                 const float* residual, void* workspace, size_t ws_bytes,
                                 void* stream) {
  polyq_clear_error();
  const polyq_dev_layer* one[1] = {L};
  const void* xs[1] = {x};
  float* ys[1] = {y};
  const float* rs[1] = {residual};
  return gemv_group("polyq_linear_gemv", one, 1, xs, batch, ys, rs, workspace, ws_bytes,
                    (cudaStream_t)stream);
}

extern "C" int polyq_linear_gemv_group(const polyq_dev_layer* const* layers, int n,
                                       const void* const* xs, int batch, float* const* ys,
                                       const float* const* residuals, void* workspace,
                                       size_t ws_bytes, void* stream) {
  polyq_clear_error();
  return gemv_group("polyq_linear_gemv_group", layers, n, xs, batch, ys, residuals, workspace,
                    ws_bytes, (cudaStream_t)stream);
}

// ---------------------------------------------------------------------------
// the same GEMV with library-owned scratch instead of a caller workspace
// ---------------------------------------------------------------------------
// Some callers cannot allocate device memory: a plugin inside a host program
// whose own pool owns the device, or a latency-bound loop that cannot take the
// device-wide synchronisation cudaMalloc/cudaFree may cause.  For them the
// records and the status word live in this fixed array, one copy per device
// that loads the library, kept until the process exits.  In host code the name
// below stands for a host-side shadow, never the device address: the address
// is looked up with cudaGetSymbolAddress, once per device.
static __device__ __align__(256) uint8_t polyq_noalloc_scratch[POLYQ_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device; the first call
// per device does the lookup (so it must precede any stream capture there).
int noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemv_noalloc: cudaGetDevice: %s",
                           cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_linear_gemv_noalloc: device %d >= %d",
                           dev, kMaxDevices);
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, polyq_noalloc_scratch);
    if (e != cudaSuccess || !p)
      return polyq_set_error(POLYQ_ECUDA,
                             "polyq_linear_gemv_noalloc: scratch address on device %d: %s", dev,
                             cudaGetErrorString(e));
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return POLYQ_OK;
}

}  // namespace

extern "C" int polyq_linear_gemv_noalloc(const polyq_dev_layer* L, const void* x, int batch,
                                         float* y, const float* residual, void* stream) {
  polyq_clear_error();
  const char* who = "polyq_linear_gemv_noalloc";
  const polyq_dev_layer* one[1] = {L};
  int rc = check_group(who, one, 1, batch);
  if (rc) return rc;
  const size_t need = workspace_for(one, 1, batch);
  if (need > POLYQ_NOALLOC_SCRATCH_BYTES)
    return polyq_set_error(POLYQ_ENOMEM,
                           "%s: this layer at batch %d needs %zu bytes of scratch, above the "
                           "fixed maximum of %u; call polyq_linear_gemv with a workspace",
                           who, batch, need, (unsigned)POLYQ_NOALLOC_SCRATCH_BYTES);
  void* scratch = nullptr;
  rc = noalloc_scratch(&scratch);
  if (rc) return rc;
  // gemv_prep writes every record the main kernel reads and zeroes the status
  // word before anything reads it, so stale contents need no clearing here.
  const void* xs[1] = {x};
  float* ys[1] = {y};
  const float* rs[1] = {residual};
  return gemv_group(who, one, 1, xs, batch, ys, rs, scratch, POLYQ_NOALLOC_SCRATCH_BYTES,
                    (cudaStream_t)stream);
}
