// Decode GEMV of the PolyQ mixed-bit layer (Section 4.1 factorisation with
// the Section 4.2 bit blocks), one launch over all blocks of one or several
// independent layers:
//
//   y[b][n] = residual[b][n] + sum_p x[b][gather[p]] * t[p] * W'[n][p]
//
// (t = the Section 3.4 activation factors of a scaled layer, else 1.)
//
// Two kernels per call, chained with programmatic dependent launch:
//  * gemv_prep, one CTA per (layer, step): gathers x through `gather`, scales
//    each value by the power of two that the decoder leaves on its code,
//    rounds it to fp16 and stores the step's activation record together with
//    per-chunk sums for the magic-number and zero-point corrections.  The
//    gather indices are loaded before the wait for the previous kernel.
//  * gemv_main, persistent, 160 threads per CTA, 3 CTAs per SM.  The (layer,
//    64-row tile, step) work items of all layers of the call form one list;
//    each CTA takes a contiguous range of it.  Warp 4 (one thread) streams
//    each item's packed codes and scale/zero metadata with TMA through a
//    3-stage shared-memory ring, the first stages before the grid-dependency
//    wait (weights do not depend on earlier kernels), and adds the item's
//    record once the pre-pass is done.  Warps 0-3 each own 16 rows: a code
//    pair becomes two exact fp16 values 1024 + q*2^p with one LOP3 against the
//    register-held constant 0x64006400, and mma.sync m16n8k16 multiplies them
//    with the record.  Each MMA column holds one 64-code chunk (one
//    quantisation group), so a chunk's dot product D is exact up to fp32
//    accumulation and its scale/zero apply once:
//        y += s * (D - 1024*sum(x') - z*sum(x)).
//    16-bit blocks feed their fp16 weights to the same MMA directly.
//  * Row sums stay in registers across a tile's steps.  The pre-pass sets y
//    to the residual (or zero); each piece of a tile adds its rows into y
//    with one fp32 atomic addition per row, so a tile split over CTAs gets
//    its few additions in an order that may vary from run to run.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
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
constexpr int kThreads = 32 * (kWarps + 1);
constexpr int kConsumers = 32 * kWarps;

struct GvBlock {
  int bits, n_ch, pos0, seg_off, grp_off;
  int step0, n_steps;  // step range of this block inside its layer
  int units;           // units per step
};

// One layer of a call.  Tensor maps first (64-byte aligned).
struct GvLayer {
  CUtensorMap tm_codes[POLYQ_MAX_BLOCKS];
  CUtensorMap tm_meta;
  GvBlock blk[POLYQ_MAX_BLOCKS];
  int n_blocks;
  int N, K;
  int steps;  // steps per row
  int items;  // tiles * steps
  int item0;  // first item of this layer in the call's list
  int rec0;   // first activation record of this layer (one per step)
  const __nv_bfloat16* x;
  const int32_t* gather;
  const float* xscale;  // Section 3.4 activation factors or NULL
  float* y;
  const float* residual;
};

struct GvParams {
  GvLayer L[POLYQ_MAX_GROUP];
  int n_layers;
  int items;       // all layers
  int recs;        // activation records of all layers
  int batch;
  uint32_t magic;  // 0x64006400 (two fp16 1024.0), kept in a register
  // workspace
  int* status;     // sticky error word
  uint8_t* rec;    // [recs][rec_bytes(NB)] activation records
  // input transform shared by all layers (POLYQ_X_*); with POLYQ_X_BF16 each
  // layer reads its own L[l].x
  int xkind;
  float eps;
  const float* xa;  // fp32 input of the transforms
  const float* xb;  // second fp32 input of POLYQ_X_SILU_MUL
  uint16_t* xout;   // optional bf16 copy of the transformed input
};

// Per-CTA shared copy of the scalars and block tables (runtime-indexed reads
// of kernel parameters would become slow generic loads).
struct GvShared {
  GvBlock blk[POLYQ_MAX_GROUP][POLYQ_MAX_BLOCKS];
  int n_blocks[POLYQ_MAX_GROUP];
  int N[POLYQ_MAX_GROUP];
  int steps[POLYQ_MAX_GROUP];
  int item0[POLYQ_MAX_GROUP + 1];
  int rec0[POLYQ_MAX_GROUP + 1];
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
  if (threadIdx.x == 0) {
    S->item0[P.n_layers] = P.items;
    S->rec0[P.n_layers] = P.recs;
  }
}

// Position of a work item: layer, tile, step of the layer, block, step of the
// block.  Items of a CTA are consecutive, so the position advances in place.
struct ItemPos {
  int l, tile, s, bi, j;

  __device__ __forceinline__ void init(const GvShared& S, int nl, int item) {
    l = 0;
    while (l + 1 < nl && item >= S.item0[l + 1]) ++l;
    const int li = item - S.item0[l];
    tile = li / S.steps[l];
    s = li - tile * S.steps[l];
    bi = 0;
    while (bi + 1 < S.n_blocks[l] && s >= S.blk[l][bi + 1].step0) ++bi;
    j = s - S.blk[l][bi].step0;
  }
  __device__ __forceinline__ bool tile_end(const GvShared& S) const {
    return s == S.steps[l] - 1;
  }
  __device__ __forceinline__ void next(const GvShared& S, int nl) {
    ++s;
    ++j;
    if (s == S.steps[l]) {
      s = 0;
      j = 0;
      bi = 0;
      ++tile;
      if (l + 1 < nl && S.item0[l] + tile * S.steps[l] >= S.item0[l + 1]) {
        ++l;
        tile = 0;
      }
    } else if (j == S.blk[l][bi].n_steps) {
      ++bi;
      j = 0;
    }
  }
};

__device__ __forceinline__ const __nv_bfloat16* layer_x(const GvParams& P, int l) {
  const __nv_bfloat16* x = P.L[0].x;
#pragma unroll
  for (int q = 1; q < POLYQ_MAX_GROUP; ++q)
    if (q == l) x = P.L[q].x;
  return x;
}
__device__ __forceinline__ const int32_t* layer_gather(const GvParams& P, int l) {
  const int32_t* g = P.L[0].gather;
#pragma unroll
  for (int q = 1; q < POLYQ_MAX_GROUP; ++q)
    if (q == l) g = P.L[q].gather;
  return g;
}
__device__ __forceinline__ const float* layer_xscale(const GvParams& P, int l) {
  const float* f = P.L[0].xscale;
#pragma unroll
  for (int q = 1; q < POLYQ_MAX_GROUP; ++q)
    if (q == l) f = P.L[q].xscale;
  return f;
}
__device__ __forceinline__ int layer_K(const GvParams& P, int l) {
  int k = P.L[0].K;
#pragma unroll
  for (int q = 1; q < POLYQ_MAX_GROUP; ++q)
    if (q == l) k = P.L[q].K;
  return k;
}


__device__ __forceinline__ uint32_t pack_half2(__half lo, __half hi) {
  return (uint32_t)__half_as_ushort(lo) | ((uint32_t)__half_as_ushort(hi) << 16);
}

// ---------------------------------------------------------------------------
// activation records (consumer warps, shared memory)
// ---------------------------------------------------------------------------
// Which activation values one consumer thread contributes to a record.  A
// record has at most two slots per thread:
//  * b < 16: slot s is the (batch, chunk) pair bc = warp + 4s of the step;
//    lane q of the warp makes the q-th of the chunk's 32 lane pairs.
//  * 16-bit: slot s is entry e = tid + 128s of the [batch][lane][16] pairs.
struct SlotGeom {
  bool valid;
  int bb, c, t, jp;
  int ch[2];  // channels (inside the block) of the pair's low and high half
  int p[2];   // power-of-two scale exponents of the two halves
};

template <int NB, int BITS>
__device__ __forceinline__ SlotGeom slot_geom_t(int warp, int lane, int tid, int s, int j,
                                                const uint32_t* p3) {
  SlotGeom g;
  if constexpr (BITS == 16) {
    const int e = tid + kConsumers * s;
    g.valid = e < NB * 64;
    g.bb = e / 64;
    g.t = (e / 16) % 4;
    g.jp = e % 16;
    g.c = 0;
    g.ch[0] = j * 128 + lane_weight16(g.t, 2 * g.jp);
    g.ch[1] = j * 128 + lane_weight16(g.t, 2 * g.jp + 1);
    g.p[0] = g.p[1] = 0;
  } else {
    constexpr int U = step_units(BITS, NB), NGS = U / 64;
    constexpr int GP = group_pairs(BITS), GU = group_units(BITS);
    const int bc = warp + kWarps * s;
    g.valid = bc < NB * NGS;
    g.bb = bc / NGS;
    g.c = bc - g.bb * NGS;
    chunk_pair(BITS, NB, g.c, lane, &g.t, &g.jp);
    const int jj = g.jp % GP, base = (g.jp / GP) * GU;
    int lo, hi;
    if constexpr (BITS == 3) {
      const uint32_t e = p3[jj];  // lo | hi << 8 | (win + 16) << 16
      lo = (int)(e & 0xFF);
      hi = (int)((e >> 8) & 0xFF);
      const int win = (int)(e >> 16) - 16;
      g.p[0] = 3 * lo - win;
      g.p[1] = 3 * hi - win - 16;
    } else {
      const PairDef d = pair_def(BITS, jj);
      lo = d.lo;
      hi = d.hi;
      g.p[0] = d.plo;
      g.p[1] = d.phi;
    }
    g.ch[0] = j * U + lane_unit(BITS, NB, g.t, base + lo);
    g.ch[1] = j * U + lane_unit(BITS, NB, g.t, base + hi);
  }
  return g;
}

template <int NB>
__device__ __forceinline__ SlotGeom slot_geom(int bits, int warp, int lane, int tid, int s,
                                              int j, const uint32_t* p3) {
  switch (bits) {
    case 2: return slot_geom_t<NB, 2>(warp, lane, tid, s, j, p3);
    case 3: return slot_geom_t<NB, 3>(warp, lane, tid, s, j, p3);
    case 4: return slot_geom_t<NB, 4>(warp, lane, tid, s, j, p3);
    case 8: return slot_geom_t<NB, 8>(warp, lane, tid, s, j, p3);
    default: return slot_geom_t<NB, 16>(warp, lane, tid, s, j, p3);
  }
}

// Where a record's activations come from: the layer's input (bf16 x, or the
// fp32 inputs of a fused transform), its gather vector, its activation
// factors and its width K.
struct XIn {
  const __nv_bfloat16* x;
  const float* xa;
  const float* xb;
  uint16_t* xout;  // written when not NULL
  const int32_t* gather;
  const float* xscale;
  int kind, K, batch;
};

__device__ __forceinline__ XIn xin_of(const GvParams& P, int l) {
  XIn in;
  in.x = layer_x(P, l);
  in.xa = P.xa;
  in.xb = P.xb;
  in.xout = l == 0 ? P.xout : nullptr;  // layer 0's records cover every source element
  in.gather = layer_gather(P, l);
  in.xscale = layer_xscale(P, l);
  in.kind = P.xkind;
  in.K = layer_K(P, l);
  in.batch = P.batch;
  return in;
}

// Pass 1 of a record: the gather indices and activation factors (static
// layer data, so this may run before the grid-dependency wait).
template <int NB>
__device__ __forceinline__ void rec_sources(const XIn& in, const GvBlock& B, int j, int warp,
                                            int lane, const uint32_t* p3, int (&src)[2][2],
                                            float (&fac)[2][2]) {
  const int32_t* gather = in.gather;
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    src[s][0] = src[s][1] = -1;
    fac[s][0] = fac[s][1] = 1.f;
    const SlotGeom g = slot_geom<NB>(B.bits, warp, lane, threadIdx.x, s, j, p3);
    if (g.valid && g.bb < in.batch) {
#pragma unroll
      for (int h = 0; h < 2; ++h)
        if (g.ch[h] < B.n_ch) {
          const int p = B.pos0 + g.ch[h];
          src[s][h] = gather ? __ldg(gather + p) : p;
          if (in.xscale) fac[s][h] = __ldg(in.xscale + p);
        }
    }
  }
}

// Passes 2 and 3: load the activations, scale, round to fp16, store the
// pairs and (b < 16) the per-chunk sums C1 = 1024 * sum x' and X = sum x.
template <int NB>
__device__ __forceinline__ void rec_build(const XIn& in, const GvBlock& B, int j, int warp,
                                          int lane, const uint32_t* p3, const int (&src)[2][2],
                                          const float (&fac)[2][2], const float* rnorm,
                                          uint32_t* rec) {
  constexpr int LW = rec_lane_words(NB);
  constexpr int PW = rec_pair_words(NB);
  constexpr int NGM = 8 / NB;
  const __nv_bfloat16* x = in.x;
  const int K = in.K;
  float xv[2][2];
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const SlotGeom g = slot_geom<NB>(B.bits, warp, lane, threadIdx.x, s, j, p3);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (src[s][h] < 0) {
        xv[s][h] = 0.f;
        continue;
      }
      const size_t o = (size_t)g.bb * K + src[s][h];
      __nv_bfloat16 v;
      switch (in.kind) {
        case POLYQ_X_F32: v = __float2bfloat16_rn(in.xa[o]); break;
        case POLYQ_X_RMSNORM: v = __float2bfloat16_rn(in.xa[o] * rnorm[g.bb]); break;
        case POLYQ_X_SILU_MUL: {
          const float a = in.xa[o];
          v = __float2bfloat16_rn(a / (1.f + expf(-a)) * in.xb[o]);
          break;
        }
        default: v = x[o]; break;
      }
      if (in.xout) in.xout[o] = __bfloat16_as_ushort(v);
      xv[s][h] = __bfloat162float(v) * fac[s][h];  // Section 3.4 factor (1 if none)
    }
  }
  float* recf = reinterpret_cast<float*>(rec);
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const SlotGeom g = slot_geom<NB>(B.bits, warp, lane, threadIdx.x, s, j, p3);
    if (!g.valid) continue;  // uniform over the warp for b < 16
    const __half hlo = __float2half_rn(ldexpf(xv[s][0], -g.p[0]));
    const __half hhi = __float2half_rn(ldexpf(xv[s][1], -g.p[1]));
    rec[(g.bb * 4 + g.t) * LW + g.jp] = pack_half2(hlo, hhi);
    if (B.bits != 16) {
      // X sums the values the MMA multiplies (fp16 times 2^p), so that the
      // zero-point term removes exactly what the codes' z adds; with
      // activation factors these differ from the fp32 products x * t
      float s1 = __half2float(hlo) + __half2float(hhi);
      float s2 = ldexpf(__half2float(hlo), g.p[0]) + ldexpf(__half2float(hhi), g.p[1]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        s1 += __shfl_xor_sync(0xffffffffu, s1, o);
        s2 += __shfl_xor_sync(0xffffffffu, s2, o);
      }
      if (lane == 0) {
        recf[PW + g.bb * NGM + g.c] = kMagicF * s1;
        recf[PW + NB * NGM + g.bb * NGM + g.c] = s2;
      }
    }
  }
}

// Layer, block and block step of record r.
__device__ __forceinline__ void rec_pos(const GvShared& S, int nl, int r, int* l, int* bi,
                                        int* j) {
  int q = 0;
  while (q + 1 < nl && r >= S.rec0[q + 1]) ++q;
  const int s = r - S.rec0[q];
  int b = 0;
  while (b + 1 < S.n_blocks[q] && s >= S.blk[q][b + 1].step0) ++b;
  *l = q;
  *bi = b;
  *j = s - S.blk[q][b].step0;
}

// ---------------------------------------------------------------------------
// MMA steps
// ---------------------------------------------------------------------------
template <int BITS>
__device__ __forceinline__ uint32_t window(const uint32_t* w, int off) {
  // bits [off, off+32) of the little-endian stream held in w[]
  if (off < 0) return w[0] << (-off);
  const int k = off >> 5, r = off & 31;
  if (r == 0) return w[k];
  if (k + 1 >= group_words(BITS)) return w[k] >> r;
  return __funnelshift_r(w[k], w[k + 1], r);
}

// Pair register for lane pair j of one row's words: one LOP3 with the mask
// as its immediate and `magic` in a register, plus the window's shift, which
// the pairs sharing a window share.
template <int BITS>
__device__ __forceinline__ uint32_t make_pair(const uint32_t* words, int j, uint32_t magic) {
  constexpr int GP = group_pairs(BITS);
  constexpr int GW = group_words(BITS);
  constexpr uint32_t QM = (1u << BITS) - 1u;
  const PairDef d = pair_def(BITS, j % GP);
  const uint32_t* g = words + (j / GP) * GW;
  const uint32_t win = window<BITS>(g, d.win);
  const uint32_t m = (QM << d.plo) | ((QM << d.phi) << 16);
  return lop3_and_or(win, m, magic);
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

// One step of a b<16 block for this warp's 16 rows; adds the chunk results,
// scaled, into acc[row][batch].
template <int NB, int BITS>
__device__ __forceinline__ void step_mma(uint32_t magic, int batch, int uvalid, int g0,
                                         const uint8_t* stage, const uint32_t* rec,
                                         const uint32_t* zeros, int warp, int lane,
                                         float (&acc)[2][NB]) {
  constexpr int U = step_units(BITS, NB);
  constexpr int NGS = step_chunks(BITS, NB);
  constexpr int NGM = 8 / NB;
  constexpr int NW = lane_words(BITS, NB);
  constexpr int LW = rec_lane_words(NB);
  constexpr int PW = rec_pair_words(NB);
  constexpr int GP = group_pairs(BITS), GW = group_words(BITS);
  constexpr int NBX = nbox_of(BITS, NB);
  constexpr int GPB = NW / GW / NBX;      // groups per box
  constexpr int CPB = U / NBX / 64;       // chunks per box
  static_assert(GP % 4 == 0 && GPB * GW * NBX == NW, "step geometry");
  const int g = lane >> 2, t = lane & 3;
  const int rA = warp * 16 + g, rB = rA + 8;
  const uint32_t* meta_s = reinterpret_cast<const uint32_t*>(stage + kCodesBytes);

  uint32_t wa[NW], wb[NW];
  load_words<BITS, NB>(wa, stage, rA, t);
  load_words<BITS, NB>(wb, stage, rB, t);

  // Column g of the B fragment is (batch my_b, chunk my_c); lane t's codes in
  // box h belong to chunk c_t + h*CPB, so only a matching lane loads its
  // activations, the others read zeros.
  const int my_b = g / NGS, my_c = g % NGS;
  const int dc = my_b < batch ? my_c - lane_unit(BITS, NB, t, 0) / 64 : -1000;
  const uint32_t* brow = rec + (my_b * 4 + t) * LW;

  float d[4][4];
#pragma unroll
  for (int q = 0; q < 4; ++q) d[q][0] = d[q][1] = d[q][2] = d[q][3] = 0.f;
#pragma unroll
  for (int h = 0; h < NBX; ++h) {
    if (h == 1 && uvalid <= U / 2) break;  // the second half of the step is empty
    const uint32_t* bsrc = dc == h * CPB ? brow + h * GPB * GP : zeros;
#pragma unroll
    for (int qq = 0; qq < GPB; ++qq) {
      const int q = h * GPB + qq;
#pragma unroll
      for (int m2 = 0; m2 < GP / 4; ++m2) {  // two MMAs per 16-byte activation load
        const uint4 bv = *reinterpret_cast<const uint4*>(bsrc + qq * GP + 4 * m2);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int jp = q * GP + 4 * m2 + 2 * hh;  // lane pair index
          const uint32_t a0 = make_pair<BITS>(wa, jp, magic);
          const uint32_t a1 = make_pair<BITS>(wb, jp, magic);
          const uint32_t a2 = make_pair<BITS>(wa, jp + 1, magic);
          const uint32_t a3 = make_pair<BITS>(wb, jp + 1, magic);
          mma_f16_16816(d[(jp / 2) & 3], a0, a1, a2, a3, hh ? bv.z : bv.x, hh ? bv.w : bv.y);
        }
      }
    }
  }
  float D[4];
#pragma unroll
  for (int v = 0; v < 4; ++v) D[v] = (d[0][v] + d[1][v]) + (d[2][v] + d[3][v]);

  // epilogue: columns 2t, 2t+1 -> (batch, chunk) (col / NGS, col % NGS);
  // g0 is the step's first group in the meta box
  const float* recf = reinterpret_cast<const float*>(rec);
#pragma unroll
  for (int cc = 0; cc < 2; ++cc) {
    const int col = 2 * t + cc;
    const int be = col / NGS, c = col % NGS;
    if (be < batch) {
      const float C1 = recf[PW + be * NGM + c];
      const float X = recf[PW + NB * NGM + be * NGM + c];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const uint32_t m = meta_s[(r ? rB : rA) * kMetaBox + g0 + c];
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

// One 16-bit step: the fp16 weights are the MMA's A operand as stored; column
// n of B is batch row n.  Lane t holds weights [16t, 16t+16) of each of the
// two 64-weight boxes.
template <int NB>
__device__ __forceinline__ void step_16(int batch, int uvalid,
                                        const uint8_t* stage, const uint32_t* rec,
                                        const uint32_t* zeros, int warp, int lane,
                                        float (&acc)[2][NB]) {
  constexpr int LW = rec_lane_words(NB);
  constexpr int PITCH = kPitchSplit;
  static_assert(box_pitch(16, NB) == PITCH && nbox_of(16, NB) == 2, "16-bit geometry");
  const int g = lane >> 2, t = lane & 3;
  const int rA = warp * 16 + g, rB = rA + 8;
  const uint32_t* bsrc = g < batch ? rec + (g * 4 + t) * LW : zeros;
  float d[2][4];
#pragma unroll
  for (int q = 0; q < 2; ++q) d[q][0] = d[q][1] = d[q][2] = d[q][3] = 0.f;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    if (h == 1 && uvalid <= 64) break;
    const uint4* pa = reinterpret_cast<const uint4*>(stage + h * kRows * PITCH + rA * PITCH + 32 * t);
    const uint4* pb = reinterpret_cast<const uint4*>(stage + h * kRows * PITCH + rB * PITCH + 32 * t);
    const uint4 a0 = pa[0], a1 = pa[1], b0 = pb[0], b1 = pb[1];
    const uint32_t wa[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
    const uint32_t wb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
    for (int m2 = 0; m2 < 2; ++m2) {
      const uint4 bv = *reinterpret_cast<const uint4*>(bsrc + 8 * h + 4 * m2);
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int k = 4 * m2 + 2 * hh;
        mma_f16_16816(d[hh], wa[k], wb[k], wa[k + 1], wb[k + 1], hh ? bv.z : bv.x,
                      hh ? bv.w : bv.y);
      }
    }
  }
#pragma unroll
  for (int cc = 0; cc < 2; ++cc) {
    const int be = 2 * t + cc;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const float v = d[0][2 * r + cc] + d[1][2 * r + cc];
#pragma unroll
      for (int b = 0; b < NB; ++b)
        if (b == be) acc[r][b] += v;
    }
  }
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// ---------------------------------------------------------------------------
// pre-pass: one CTA of 128 threads per activation record (layer, step)
// ---------------------------------------------------------------------------
template <int NB>
__global__ void __launch_bounds__(kConsumers) gemv_prep(const __grid_constant__ GvParams P) {
  pdl_trigger();  // the main kernel may start streaming weights right away
  __shared__ GvShared S;
  __shared__ uint32_t s_p3[16];  // 3-bit pair schedule
  load_shared(P, &S);
  if (threadIdx.x < 16) {
    const PairDef d = pair3(threadIdx.x);
    s_p3[threadIdx.x] = (uint32_t)d.lo | ((uint32_t)d.hi << 8) | ((uint32_t)(d.win + 16) << 16);
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x;
  int l, bi, j;
  rec_pos(S, P.n_layers, r, &l, &bi, &j);
  int src[2][2];
  float fac[2][2];
  const XIn in = xin_of(P, l);
  rec_sources<NB>(in, S.blk[l][bi], j, warp, lane, s_p3, src, fac);  // static layer data
  pdl_wait();  // x comes from the previous kernel; the records and y may still be in use
  __shared__ float s_rnorm[4];
  if (P.xkind == POLYQ_X_RMSNORM) {
    // 1 / sqrt(mean(a^2) + eps) of each batch row
    __shared__ float s_part[4][kWarps];
    const int K = P.L[0].K;
    for (int bb = 0; bb < P.batch; ++bb) {
      float acc = 0.f;
      for (int i = threadIdx.x; i < K; i += kConsumers) {
        const float v = P.xa[(size_t)bb * K + i];
        acc = fmaf(v, v, acc);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (lane == 0) s_part[bb][warp] = acc;
    }
    __syncthreads();
    if (threadIdx.x < P.batch) {
      float t = 0.f;
      for (int w = 0; w < kWarps; ++w) t += s_part[threadIdx.x][w];
      s_rnorm[threadIdx.x] = rsqrtf(t / (float)K + P.eps);
    }
    __syncthreads();
  }
  rec_build<NB>(in, S.blk[l][bi], j, warp, lane, s_p3, src, fac, s_rnorm,
                reinterpret_cast<uint32_t*>(P.rec + (size_t)r * rec_bytes(NB)));
  // y starts as the residual (or zero); the main kernel adds its pieces
#pragma unroll
  for (int q = 0; q < POLYQ_MAX_GROUP; ++q) {
    if (q >= P.n_layers) break;
    float* y = P.L[q].y;
    const float* res = P.L[q].residual;
    if (y == res) continue;
    const int total = P.batch * P.L[q].N;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x)
      y[i] = res ? res[i] : 0.f;
  }
}

template <int NB>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) gemv_main(const __grid_constant__ GvParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int RB = rec_bytes(NB);
  uint8_t* stages = smem;
  uint32_t* zeros = reinterpret_cast<uint32_t*>(smem + kStages * kStageBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(zeros + 64);
  __shared__ GvShared S;
  // Set once any wait of this CTA gives up: later waits are skipped so that
  // every warp still reaches the consumer barriers and the kernel ends.
  __shared__ volatile int s_abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);

  load_shared(P, &S);
  if (threadIdx.x == 0) s_abort = 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kWarps);
    }
    mbar_fence_init();
  }
  if (threadIdx.x < 64) zeros[threadIdx.x] = 0u;
  __syncthreads();
  pdl_trigger();
  const int nl = P.n_layers;

  // contiguous range of (layer, tile, step) items
  const long long I = P.items, C = gridDim.x;
  const int lo = (int)((long long)blockIdx.x * I / C);
  const int hi = (int)((long long)(blockIdx.x + 1) * I / C);
  const int n_mine = hi - lo;

  if (warp == kWarps) {
    // ---------------- producer ----------------
    // The packed weights do not depend on earlier kernels: request the first
    // stages before the grid-dependency wait.  The activation records come
    // from this call's builders and are loaded once they are flagged ready.
    ItemPos it;
    it.init(S, nl, lo);
    auto issue_weights = [&](int k, const ItemPos& q) {
      const int slot = k % kStages;
      const GvBlock& B = S.blk[q.l][q.bi];
      int sb, nbx, pitch;
      switch (B.bits) {
        case 2: sb = step_bytes(2, NB); nbx = nbox_of(2, NB); pitch = box_pitch(2, NB); break;
        case 3: sb = step_bytes(3, NB); nbx = nbox_of(3, NB); pitch = box_pitch(3, NB); break;
        case 4: sb = step_bytes(4, NB); nbx = nbox_of(4, NB); pitch = box_pitch(4, NB); break;
        case 8: sb = step_bytes(8, NB); nbx = nbox_of(8, NB); pitch = box_pitch(8, NB); break;
        default: sb = step_bytes(16, NB); nbx = nbox_of(16, NB); pitch = box_pitch(16, NB); break;
      }
      const uint32_t dst = smem_u32(stages + slot * kStageBytes);
      const uint32_t bar = full0 + 8 * slot;
      {
        // what the consumers need of this item: width, whether the item ends
        // a tile piece, layer, valid units, first meta entry, tile
        const int uvalid = min(B.units, B.n_ch - q.j * B.units);
        const int g0 = (B.grp_off + q.j * (B.units / 64)) & 3;
        const bool flush = q.tile_end(S) || k == n_mine - 1;
        uint4 d;
        d.x = (uint32_t)B.bits | ((uint32_t)flush << 8) | ((uint32_t)q.l << 16);
        d.y = (uint32_t)uvalid | ((uint32_t)g0 << 16);
        d.z = (uint32_t)q.tile;
        d.w = 0u;
        *reinterpret_cast<uint4*>(stages + slot * kStageBytes + kDescOff) = d;
      }
      uint32_t bytes = nbx * pitch * kRows + RB;
      if (B.bits < 16) bytes += kMetaBytes;
      mbar_expect_tx(bar, bytes);
      const CUtensorMap* tm = &P.L[q.l].tm_codes[q.bi];
      for (int h = 0; h < nbx; ++h)
        tma_load_2d(dst + h * kRows * pitch, tm, B.seg_off + q.j * sb + h * (sb / nbx),
                    q.tile * kRows, bar);
      if (B.bits < 16) {
        const int x0 = (B.grp_off + q.j * (B.units / 64)) & ~3;
        tma_load_2d(dst + kCodesBytes, &P.L[q.l].tm_meta, x0, q.tile * kRows, bar);
      }
    };
    const int pre = min(n_mine, kStages);
    if (lane == 0) {
      for (int l = 0; l < nl; ++l) {
        for (int b = 0; b < S.n_blocks[l]; ++b) prefetch_tmap(&P.L[l].tm_codes[b]);
        prefetch_tmap(&P.L[l].tm_meta);
      }
      ItemPos q = it;
      for (int k = 0; k < pre; ++k) {
        issue_weights(k, q);
        q.next(S, nl);
      }
    }
    pdl_wait();  // the records come from the pre-pass of this call
    fence_proxy_async_global();  // it wrote them through the generic proxy
    if (lane != 0) return;
    for (int k = 0; k < n_mine; ++k) {
      const int slot = k % kStages;
      if (s_abort) break;
      if (k >= kStages) {
        if (!mbar_wait(empty0 + 8 * slot, ((k / kStages) - 1) & 1)) {
          atomicExch(P.status, kStatusTimeoutEmpty);
          s_abort = 1;
          break;
        }
        issue_weights(k, it);
      }
      const int r = S.rec0[it.l] + it.s;
      bulk_load(smem_u32(stages + slot * kStageBytes + kRecOff),
                P.rec + (size_t)r * RB, RB, full0 + 8 * slot);
      it.next(S, nl);
    }
    return;
  }

  // ---------------- consumers ----------------
  const int g = lane >> 2, t = lane & 3;
  pdl_wait();  // y, the workspace and the records are this call's from here on
  float acc[2][NB];
#pragma unroll
  for (int r = 0; r < 2; ++r)
#pragma unroll
    for (int b = 0; b < NB; ++b) acc[r][b] = 0.f;
  int slot = 0;
  uint32_t phase = 0;
  for (int k = 0; k < n_mine; ++k) {
    if (s_abort || !mbar_wait(full0 + 8 * slot, phase)) {
      if (lane == 0 && !s_abort) atomicExch(P.status, kStatusTimeoutFull);
      s_abort = 1;
      break;
    }
    const uint8_t* stage = stages + slot * kStageBytes;
    const uint32_t* rec = reinterpret_cast<const uint32_t*>(stage + kRecOff);
    const uint4 desc = *reinterpret_cast<const uint4*>(stage + kDescOff);
    const int bits = (int)(desc.x & 0xFFu);
    const int uvalid = (int)(desc.y & 0xFFFFu), g0 = (int)(desc.y >> 16);
    switch (bits) {
      case 2: step_mma<NB, 2>(P.magic, P.batch, uvalid, g0, stage, rec, zeros, warp, lane, acc); break;
      case 3: step_mma<NB, 3>(P.magic, P.batch, uvalid, g0, stage, rec, zeros, warp, lane, acc); break;
      case 4: step_mma<NB, 4>(P.magic, P.batch, uvalid, g0, stage, rec, zeros, warp, lane, acc); break;
      case 8: step_mma<NB, 8>(P.magic, P.batch, uvalid, g0, stage, rec, zeros, warp, lane, acc); break;
      default: step_16<NB>(P.batch, uvalid, stage, rec, zeros, warp, lane, acc); break;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty0 + 8 * slot);
    if (++slot == kStages) {
      slot = 0;
      phase ^= 1u;
    }

    if (desc.x & 0x100u) {
      // ---- add this warp's 16 rows of the tile piece into y ----
      // Sum the four lanes of each row; lane t adds batch row t.  A tile
      // whose steps are split over CTAs gets one addition per piece.
#pragma unroll
      for (int r = 0; r < 2; ++r)
#pragma unroll
        for (int b = 0; b < NB; ++b) {
          float v = acc[r][b];
          v += __shfl_xor_sync(0xffffffffu, v, 1);
          v += __shfl_xor_sync(0xffffffffu, v, 2);
          acc[r][b] = v;
        }
      const int l = (int)(desc.x >> 16);
      float* y = P.L[0].y;
      int N = P.L[0].N;
#pragma unroll
      for (int q = 1; q < POLYQ_MAX_GROUP; ++q)
        if (q == l) {
          y = P.L[q].y;
          N = P.L[q].N;
        }
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int n = (int)desc.z * kRows + warp * 16 + g + 8 * r;
#pragma unroll
        for (int b = 0; b < NB; ++b)
          if (b == t && b < P.batch && n < N) atomicAdd(y + (size_t)b * N + n, acc[r][b]);
#pragma unroll
        for (int b = 0; b < NB; ++b) acc[r][b] = 0.f;
      }
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
    g.units = step_units(b.bits, nb);
    g.step0 = s;
    g.n_steps = (b.n_ch + g.units - 1) / g.units;
    s += g.n_steps;
    if (blk) blk[i] = g;
  }
  return s;
}

// CTAs of one launch: all of them must be resident at once (an owner waits
// for pieces of later CTAs), so never more than the device holds.
int grid_for(int items, int* grid) {
  int sms = 0;
  int rc = polyq_sm_count(&sms);
  if (rc) return rc;
  *grid = std::max(1, std::min(std::min(items, kCtasPerSm * sms), kMaxGrid));
  return POLYQ_OK;
}

// Workspace: [0, 256) status word, then one activation record per step of
// every layer of the call.
struct WsLayout {
  size_t rec_off, bytes;
  int grid, items, recs;
};

int workspace_layout(const polyq_dev_layer* const* L, int n, int batch, WsLayout* w) {
  const int nb = nb_of(batch);
  long long items = 0, recs = 0;
  for (int i = 0; i < n; ++i) {
    const long long t = (L[i]->N + kRows - 1) / kRows;
    const long long st = steps_of(L[i], nb, nullptr);
    items += t * st;
    recs += st;
  }
  if (items > (1ll << 30) || recs > (1ll << 20))
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq gemv: too many work items (%lld)", items);
  w->items = (int)items;
  w->recs = (int)recs;
  int rc = grid_for(w->items, &w->grid);
  if (rc) return rc;
  w->rec_off = 256;
  w->bytes = w->rec_off + (size_t)recs * rec_bytes(nb);
  return POLYQ_OK;
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

constexpr size_t kSmemBytes = (size_t)kStages * kStageBytes + 64 * 4 + 2 * kStages * 8;

template <int NB>
int launch(const GvParams& P, int grid, cudaStream_t st) {
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (!attr_done[dev & 63]) {
    cudaError_t e = cudaFuncSetAttribute(gemv_main<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBytes);
    if (e != cudaSuccess)
      return polyq_set_error(POLYQ_ECUDA, "polyq gemv: smem attribute: %s", cudaGetErrorString(e));
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gemv_main<NB>, kThreads, kSmemBytes);
    if (e != cudaSuccess || per_sm < kCtasPerSm)
      return polyq_set_error(POLYQ_ECUDA, "polyq gemv: %d CTAs per SM fit, %d needed (%s)", per_sm,
                             kCtasPerSm, cudaGetErrorString(e));
    attr_done[dev & 63] = true;
  }
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3((unsigned)P.recs);
  cfg.blockDim = dim3(kConsumers);
  cfg.dynamicSmemBytes = 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, gemv_prep<NB>, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq gemv: pre-pass launch: %s", cudaGetErrorString(e));
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  e = cudaLaunchKernelEx(&cfg, gemv_main<NB>, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq gemv: launch: %s", cudaGetErrorString(e));
  return POLYQ_OK;
}

int gemv_group(const char* who, const polyq_dev_layer* const* L, int n, const void* const* xs,
               int batch, float* const* ys, const float* const* res, void* workspace,
               size_t ws_bytes, cudaStream_t st, const polyq_gemv_input* in = nullptr) {
  int rc = check_group(who, L, n, batch);
  if (rc) return rc;
  const void* shared_x[POLYQ_MAX_GROUP];
  if (in) {
    if (in->kind < POLYQ_X_BF16 || in->kind > POLYQ_X_SILU_MUL)
      return polyq_set_error(POLYQ_EINVAL, "%s: unknown input kind %d", who, in->kind);
    if (!in->a || (in->kind == POLYQ_X_SILU_MUL) != (in->b != nullptr))
      return polyq_set_error(POLYQ_EINVAL, "%s: input pointers do not match kind %d", who,
                             in->kind);
    if (in->kind == POLYQ_X_RMSNORM && !(in->eps >= 0.f))
      return polyq_set_error(POLYQ_EINVAL, "%s: eps must be >= 0", who);
    for (int i = 0; i < n; ++i) {
      if (L[i]->K != L[0]->K)
        return polyq_set_error(POLYQ_EINVAL, "%s: layers sharing one input need the same K", who);
      shared_x[i] = in->a;
    }
    xs = shared_x;
  }
  if (!xs || !ys) return polyq_set_error(POLYQ_EINVAL, "%s: x or y is NULL", who);
  for (int i = 0; i < n; ++i)
    if (!xs[i] || !ys[i]) return polyq_set_error(POLYQ_EINVAL, "%s: x or y %d is NULL", who, i);
  WsLayout w;
  rc = workspace_layout(L, n, batch, &w);
  if (rc) return rc;
  if (!workspace || ws_bytes < w.bytes)
    return polyq_set_error(POLYQ_ENOMEM, "%s: workspace needs %zu bytes, got %zu", who, w.bytes,
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
    const int t = (int)((D->N + kRows - 1) / kRows);
    G.items = t * steps;
    G.item0 = items;
    G.rec0 = recs;
    G.x = (const __nv_bfloat16*)xs[i];
    G.gather = D->gather;
    G.xscale = D->xscale;
    G.y = ys[i];
    G.residual = res ? res[i] : nullptr;
    items += G.items;
    recs += steps;
  }
  P.n_layers = n;
  P.items = items;
  P.recs = recs;
  P.batch = batch;
  P.magic = kMagic;
  uint8_t* ws = (uint8_t*)workspace;
  P.status = (int*)ws;
  P.rec = ws + w.rec_off;
  P.xkind = in ? in->kind : POLYQ_X_BF16;
  P.eps = in ? in->eps : 0.f;
  P.xa = in ? (const float*)in->a : nullptr;
  P.xb = in ? in->b : nullptr;
  P.xout = in ? in->x_out : nullptr;
  switch (nb) {
    case 1: return launch<1>(P, w.grid, st);
    case 2: return launch<2>(P, w.grid, st);
    default: return launch<4>(P, w.grid, st);
  }
}

}  // namespace

extern "C" int polyq_gemv_workspace_bytes(const polyq_dev_layer* L, int batch, size_t* bytes) {
  polyq_clear_error();
  const polyq_dev_layer* one[1] = {L};
  int rc = check_group("polyq_gemv_workspace_bytes", one, 1, batch);
  if (rc) return rc;
  if (!bytes) return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_workspace_bytes: bytes is NULL");
  WsLayout w;
  rc = workspace_layout(one, 1, batch, &w);
  if (rc) return rc;
  *bytes = w.bytes;
  return POLYQ_OK;
}

extern "C" int polyq_gemv_group_workspace_bytes(const polyq_dev_layer* const* layers, int n,
                                                int batch, size_t* bytes) {
  polyq_clear_error();
  int rc = check_group("polyq_gemv_group_workspace_bytes", layers, n, batch);
  if (rc) return rc;
  if (!bytes)
    return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_group_workspace_bytes: bytes is NULL");
  WsLayout w;
  rc = workspace_layout(layers, n, batch, &w);
  if (rc) return rc;
  *bytes = w.bytes;
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

extern "C" int polyq_linear_gemv_input(const polyq_dev_layer* const* layers, int n,
                                       const polyq_gemv_input* in, int batch, float* const* ys,
                                       const float* const* residuals, void* workspace,
                                       size_t ws_bytes, void* stream) {
  polyq_clear_error();
  if (!in) return polyq_set_error(POLYQ_EINVAL, "polyq_linear_gemv_input: input is NULL");
  return gemv_group("polyq_linear_gemv_input", layers, n, nullptr, batch, ys, residuals,
                    workspace, ws_bytes, (cudaStream_t)stream, in);
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
// status word, tile counters and piece sums live in this fixed array, one copy
// per device that loads the library, kept until the process exits.  In host
// code the name below stands for a host-side shadow, never the device address:
// the address is looked up with cudaGetSymbolAddress, once per device.
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
  WsLayout w;
  rc = workspace_layout(one, 1, batch, &w);
  if (rc) return rc;
  if (w.bytes > POLYQ_NOALLOC_SCRATCH_BYTES)
    return polyq_set_error(POLYQ_ENOMEM,
                           "%s: this layer at batch %d needs %zu bytes of scratch, above the "
                           "fixed maximum of %u; call polyq_linear_gemv with a workspace",
                           who, batch, w.bytes, (unsigned)POLYQ_NOALLOC_SCRATCH_BYTES);
  void* scratch = nullptr;
  rc = noalloc_scratch(&scratch);
  if (rc) return rc;
  // The status word must start at zero.  A call that gave up on a wait
  // leaves it set, and this caller cannot reset the library's array itself:
  // clear it on every call.
  cudaError_t e = cudaMemsetAsync(scratch, 0, 256, (cudaStream_t)stream);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "%s: clearing the scratch counters: %s", who,
                           cudaGetErrorString(e));
  const void* xs[1] = {x};
  float* ys[1] = {y};
  const float* rs[1] = {residual};
  return gemv_group(who, one, 1, xs, batch, ys, rs, scratch, POLYQ_NOALLOC_SCRATCH_BYTES,
                    (cudaStream_t)stream);
}
