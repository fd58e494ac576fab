// Device building blocks of the decode GEMV shared by the per-call kernels
// and the chained persistent kernel: the bit-block table entry, the
// activation-record builder (which activation each consumer thread gathers,
// scales and rounds for a step) and the tensor-core steps that decode a
// step's codes and multiply them with its record.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "polyq.h"
#include "polyq_dev.cuh"
#include "polyq_gemv_layout.cuh"

namespace polyq {
namespace gv {

constexpr int kThreads = 32 * (kWarps + 1);  // consumer warps + one producer warp
constexpr int kConsumers = 32 * kWarps;

struct GvBlock {
  int bits, n_ch, pos0, seg_off, grp_off;
  int step0, n_steps;  // step range of this block inside its layer
  int units;           // units per step
};

// 2^k as a float, for -126 <= k <= 127 (a normal number: exponent field k + 127).
__device__ __forceinline__ float pow2i(int k) { return __int_as_float((k + 127) << 23); }

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

// NW warps build a record: a thread has slots s < rec_slots(NW).
__host__ __device__ constexpr int rec_slots(int nw) { return nw >= 8 ? 1 : 2; }

template <int NB, int BITS, int NW>
__device__ __forceinline__ SlotGeom slot_geom_t(int warp, int lane, int tid, int s, int j,
                                                const uint32_t* p3) {
  SlotGeom g;
  if constexpr (BITS == 16) {
    const int e = tid + 32 * NW * s;
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
    const int bc = warp + NW * s;
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

template <int NB, int NW>
__device__ __forceinline__ SlotGeom slot_geom(int bits, int warp, int lane, int tid, int s,
                                              int j, const uint32_t* p3) {
  switch (bits) {
    case 2: return slot_geom_t<NB, 2, NW>(warp, lane, tid, s, j, p3);
    case 3: return slot_geom_t<NB, 3, NW>(warp, lane, tid, s, j, p3);
    case 4: return slot_geom_t<NB, 4, NW>(warp, lane, tid, s, j, p3);
    case 8: return slot_geom_t<NB, 8, NW>(warp, lane, tid, s, j, p3);
    default: return slot_geom_t<NB, 16, NW>(warp, lane, tid, s, j, p3);
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

__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// Pass 1 of a record: the gather indices and activation factors (static
// layer data, so this may run before the grid-dependency wait), and an L2
// prefetch of the activations the record will read.  L2 is where writes of
// earlier kernels land, so prefetching before their completion is safe: the
// loads after the wait still see the final values.
template <int NB, int NW = kWarps>
__device__ __forceinline__ void rec_sources(const XIn& in, const GvBlock& B, int j, int warp,
                                            int lane, const uint32_t* p3, int (&src)[2][2],
                                            float (&fac)[2][2]) {
  const int32_t* gather = in.gather;
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    src[s][0] = src[s][1] = -1;
    fac[s][0] = fac[s][1] = 1.f;
    if (s >= rec_slots(NW)) continue;
    const SlotGeom g = slot_geom<NB, NW>(B.bits, warp, lane, threadIdx.x, s, j, p3);
    if (g.valid && g.bb < in.batch) {
#pragma unroll
      for (int h = 0; h < 2; ++h)
        if (g.ch[h] < B.n_ch) {
          const int p = B.pos0 + g.ch[h];
          src[s][h] = gather ? __ldg(gather + p) : p;
          if (in.xscale) fac[s][h] = __ldg(in.xscale + p);
          const size_t o = (size_t)g.bb * in.K + src[s][h];
          if (in.kind == POLYQ_X_BF16) {
            prefetch_l2(in.x + o);
          } else {
            prefetch_l2(in.xa + o);
            if (in.kind == POLYQ_X_SILU_MUL) prefetch_l2(in.xb + o);
          }
        }
    }
  }
}

// Barrier of the 32 * NW threads that build records (named barrier 1; the
// producer warp of a streaming kernel does not take part).
template <int NW = kWarps>
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(32 * NW) : "memory");
}

// L2 prefetch of the batch rows the RMSNorm factor reads (before a wait).
__device__ __forceinline__ void rms_prefetch(const float* xa, int K, int batch) {
  for (int bb = 0; bb < batch; ++bb)
    for (int i = 32 * threadIdx.x; i < K; i += 32 * kConsumers)  // one 128-byte line each
      prefetch_l2(xa + (size_t)bb * K + i);
}

// s_rnorm[b] = 1 / sqrt(mean_k a[b][k]^2 + eps) for each batch row, computed
// by the 128 consumer threads with loads through L2.  s_part holds
// batch x kWarps partial sums.  A thread's loads of up to kRmsBatch float4
// are issued together (one L2 round trip for rows up to 8192 wide).
constexpr int kRmsBatch = 16;
template <int NW = kWarps>
__device__ __forceinline__ void rms_rnorm(const float* xa, int K, int batch, float eps,
                                          float (*s_part)[NW], float* s_rnorm) {
  constexpr int NT = 32 * NW;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool vec = (K % 4 == 0) && (reinterpret_cast<uintptr_t>(xa) % 16 == 0);
  for (int bb = 0; bb < batch; ++bb) {
    const float* row = xa + (size_t)bb * K;
    float acc = 0.f;
    if (vec) {
      const int n4 = K / 4;
      for (int i0 = threadIdx.x; i0 < n4; i0 += kRmsBatch * NT) {
        float4 v[kRmsBatch];
#pragma unroll
        for (int u = 0; u < kRmsBatch; ++u) {
          const int i = i0 + u * NT;
          v[u] = i < n4 ? __ldcg(reinterpret_cast<const float4*>(row) + i)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < kRmsBatch; ++u) {
          acc = fmaf(v[u].x, v[u].x, acc);
          acc = fmaf(v[u].y, v[u].y, acc);
          acc = fmaf(v[u].z, v[u].z, acc);
          acc = fmaf(v[u].w, v[u].w, acc);
        }
      }
    } else {
      for (int i = threadIdx.x; i < K; i += NT) {
        const float v = __ldcg(row + i);
        acc = fmaf(v, v, acc);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) s_part[bb][warp] = acc;
  }
  consumer_sync<NW>();
  if (threadIdx.x < batch) {
    float t = 0.f;
    for (int w = 0; w < NW; ++w) t += s_part[threadIdx.x][w];
    s_rnorm[threadIdx.x] = rsqrtf(t / (float)K + eps);
  }
  consumer_sync<NW>();
}

// Pass 2 of a record: load the thread's raw inputs (bf16 x, or the fp32
// inputs of the transform).  Loads go through L2 (ld.global.cg) because in
// the chained kernel the inputs are written during the same launch.
template <int NB, int NW = kWarps>
__device__ __forceinline__ void rec_load(const XIn& in, const GvBlock& B, int j, int warp,
                                         int lane, const uint32_t* p3, const int (&src)[2][2],
                                         float (&ra)[2][2], float (&rb)[2][2]) {
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    ra[s][0] = ra[s][1] = rb[s][0] = rb[s][1] = 0.f;
    if (s >= rec_slots(NW)) continue;
    const SlotGeom g = slot_geom<NB, NW>(B.bits, warp, lane, threadIdx.x, s, j, p3);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (src[s][h] < 0) continue;
      const size_t o = (size_t)g.bb * in.K + src[s][h];
      if (in.kind == POLYQ_X_BF16) {
        ra[s][h] = __bfloat162float(__ushort_as_bfloat16(
            __ldcg(reinterpret_cast<const unsigned short*>(in.x) + o)));
      } else {
        ra[s][h] = __ldcg(in.xa + o);
        if (in.kind == POLYQ_X_SILU_MUL) rb[s][h] = __ldcg(in.xb + o);
      }
    }
  }
}

// Pass 3: apply the transform (the bf16 activation x), write the optional
// bf16 copy, multiply by the activation factor, scale each value by the power
// of two its code carries, round to fp16 and store the pairs and (b < 16)
// the per-chunk sums C1 = 1024 * sum x' and X = sum x' * 2^p.
template <int NB, int NW = kWarps>
__device__ __forceinline__ void rec_store(const XIn& in, const GvBlock& B, int j, int warp,
                                          int lane, const uint32_t* p3, const int (&src)[2][2],
                                          const float (&fac)[2][2], const float (&ra)[2][2],
                                          const float (&rb)[2][2], const float* rnorm,
                                          uint32_t* rec) {
  constexpr int LW = rec_lane_words(NB);
  constexpr int PW = rec_pair_words(NB);
  constexpr int NGM = 8 / NB;
  constexpr int SL = rec_slots(NW);
  float xv[2][2];
#pragma unroll
  for (int s = 0; s < SL; ++s) {
    const SlotGeom g = slot_geom<NB, NW>(B.bits, warp, lane, threadIdx.x, s, j, p3);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (src[s][h] < 0) {
        xv[s][h] = 0.f;
        continue;
      }
      const float a = ra[s][h];
      float v;  // the bf16 activation, as a float
      switch (in.kind) {
        case POLYQ_X_F32: v = __bfloat162float(__float2bfloat16_rn(a)); break;
        case POLYQ_X_RMSNORM: v = __bfloat162float(__float2bfloat16_rn(a * rnorm[g.bb])); break;
        case POLYQ_X_SILU_MUL:
          v = __bfloat162float(__float2bfloat16_rn(a / (1.f + expf(-a)) * rb[s][h]));
          break;
        default: v = a; break;
      }
      if (in.xout) {
        const size_t o = (size_t)g.bb * in.K + src[s][h];
        in.xout[o] = __bfloat16_as_ushort(__float2bfloat16_rn(v));  // exact: v is bf16
      }
      xv[s][h] = v * fac[s][h];  // Section 3.4 factor (1 if none)
    }
  }
  // Largest magnitude of each slot's values over the warp (the bit patterns of
  // non-negative floats order as integers).  For b < 16 a slot's warp holds
  // exactly one chunk; a 16-bit batch row spans warps w and w ^ 1, which
  // exchange their maxima through shared memory (the width is uniform over
  // the record, so every consumer thread takes the same branch).
  uint32_t mx[2] = {0u, 0u};
#pragma unroll
  for (int s = 0; s < SL; ++s)
    mx[s] = __reduce_max_sync(0xffffffffu, max(__float_as_uint(fabsf(xv[s][0])),
                                               __float_as_uint(fabsf(xv[s][1]))));
  if (B.bits == 16) {
    __shared__ uint32_t s_wmax[NW][2];
    consumer_sync<NW>();  // an earlier record's readers are done with s_wmax
    if (lane == 0) {
      s_wmax[warp][0] = mx[0];
      s_wmax[warp][1] = mx[1];
    }
    consumer_sync<NW>();
    mx[0] = max(mx[0], s_wmax[warp ^ 1][0]);
    mx[1] = max(mx[1], s_wmax[warp ^ 1][1]);
  }
  float* recf = reinterpret_cast<float*>(rec);
#pragma unroll
  for (int s = 0; s < SL; ++s) {
    const SlotGeom g = slot_geom<NB, NW>(B.bits, warp, lane, threadIdx.x, s, j, p3);
    if (!g.valid) continue;  // uniform over the warp
    // e: floor(log2(max)) - kRecExp (an fp32 subnormal maximum counts as 2^-127)
    const int e = mx[s] ? max((int)(mx[s] >> 23) - 127 - kRecExp, kRecExpMin) : 0;
    // 2^(-p-e) lies in [2^-121, 2^126] (p <= 8, -126 <= e <= 113): a
    // normal float, so the products are exact scalings (rounded like any
    // product where they fall below the normal range)
    const __half hlo = __float2half_rn(xv[s][0] * pow2i(-g.p[0] - e));
    const __half hhi = __float2half_rn(xv[s][1] * pow2i(-g.p[1] - e));
    rec[(g.bb * 4 + g.t) * LW + g.jp] = pack_half2(hlo, hhi);
    if (B.bits != 16) {
      // X sums the values the MMA multiplies (fp16 times 2^p), so that the
      // zero-point term removes exactly what the codes' z adds; with
      // activation factors these differ from the fp32 products x * t
      float s1 = __half2float(hlo) + __half2float(hhi);
      float s2 = __half2float(hlo) * pow2i(g.p[0]) + __half2float(hhi) * pow2i(g.p[1]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        s1 += __shfl_xor_sync(0xffffffffu, s1, o);
        s2 += __shfl_xor_sync(0xffffffffu, s2, o);
      }
      if (lane == 0) {
        recf[PW + g.bb * NGM + g.c] = kMagicF * s1;
        recf[PW + NB * NGM + g.bb * NGM + g.c] = s2;
        recf[PW + 2 * NB * NGM + g.bb * NGM + g.c] = pow2i(e);
      }
    } else if (g.jp == 0 && g.t == 0) {
      recf[PW + 2 * NB * NGM + g.bb * NGM] = pow2i(e);
    }
  }
}

// ---------------------------------------------------------------------------
// row sums of a tile piece
// ---------------------------------------------------------------------------
// Lane t of a quad keeps one partial sum per row for batch row t*NB/4: at
// batch 1 every lane row 0, at batch 2 lanes 0-1 row 0 and lanes 2-3 row 1,
// at batch 4 lane t row t.  For 2/3/4/8-bit steps that is the batch row of
// both MMA columns the lane holds (columns of other rows are past the
// batch); 16-bit steps hand their values to the first lane of the group.
template <int NB>
__device__ __forceinline__ int lane_batch(int t) {
  return t * NB / 4;
}
template <int NB>
__device__ __forceinline__ bool lane_first(int t) {
  return t % (4 / NB) == 0;
}

// Add the warp's 16 rows (row0 + g, row0 + g + 8) of a finished tile piece
// into y, summing first the lanes of a quad that hold the same batch row, and
// clear the sums.
template <int NB>
__device__ __forceinline__ void flush_rows(float (&acc)[2], float* y, int N, int batch, int row0,
                                           int lane) {
  const int g = lane >> 2, t = lane & 3;
  const int bl = lane_batch<NB>(t);
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    float v = acc[r];
    if (NB <= 2) v += __shfl_xor_sync(0xffffffffu, v, 1);
    if (NB == 1) v += __shfl_xor_sync(0xffffffffu, v, 2);
    const int n = row0 + g + 8 * r;
    if (lane_first<NB>(t) && bl < batch && n < N) atomicAdd(y + (size_t)bl * N + n, v);
    acc[r] = 0.f;
  }
}

#ifdef POLYQ_DEBUG
// Debug build only: every code an MMA step decodes is written to
// g_dbg_codes[row][position] (uint16, the layer's clustered order; for
// 16-bit weights the fp16 bit pattern), so that tests can compare the hot
// decoder with the packed bytes bit for bit.  The producer writes the step's
// first position, first tile row, the layer's N and (paired stages) the
// second step's first position into the 16 bytes after the descriptor.
__device__ uint16_t* g_dbg_codes;
__device__ long long g_dbg_K;

// The two codes of pair register v: (fp16 half - 1024) >> p for each half.
template <int NB, int BITS>
__device__ __forceinline__ void dbg_pair(uint32_t v, int jp, int t, int row, int uvalid,
                                         const uint4& d) {
  uint16_t* out = g_dbg_codes;
  if (!out) return;
  const int r = (int)d.y + row;
  if (r >= (int)d.z) return;
  int ulo, plo, uhi, phi;
  pair_units(BITS, jp, &ulo, &plo, &uhi, &phi);
  const int u0 = lane_unit(BITS, NB, t, ulo), u1 = lane_unit(BITS, NB, t, uhi);
  if (u0 < uvalid)
    out[(long long)r * g_dbg_K + d.x + u0] = (uint16_t)(((v & 0x3FFu) >> plo));
  if (u1 < uvalid)
    out[(long long)r * g_dbg_K + d.x + u1] = (uint16_t)((((v >> 16) & 0x3FFu) >> phi));
}
#endif

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
                                         const uint8_t* codes, const uint8_t* stage,
                                         const uint32_t* rec,
                                         const uint32_t* zeros, int warp, int lane,
                                         float (&acc)[2]) {
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
  load_words<BITS, NB>(wa, codes, rA, t);
  load_words<BITS, NB>(wb, codes, rB, t);

  // Column g of the B fragment is (batch my_b, chunk my_c); lane t's codes in
  // box h belong to chunk c_t + h*CPB, so only a matching lane loads its
  // activations, the others read zeros.
  const int my_b = g / NGS, my_c = g % NGS;
  const int dc = my_b < batch ? my_c - lane_unit(BITS, NB, t, 0) / 64 : -1000;
  const uint32_t* brow = rec + (my_b * 4 + t) * LW;
#ifdef POLYQ_DEBUG
  const uint4 dbg = *reinterpret_cast<const uint4*>(stage + kDescOff + 16);
#endif

  // independent accumulator sets for the step's MMA chain: four for the 32
  // MMAs of a batch-1 step, two for the 8-16 of a batch 2-4 step
  constexpr int NACC = NB == 1 ? 4 : 2;
  float d[NACC][4];
#pragma unroll
  for (int q = 0; q < NACC; ++q) d[q][0] = d[q][1] = d[q][2] = d[q][3] = 0.f;
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
#ifdef POLYQ_DEBUG
          dbg_pair<NB, BITS>(a0, jp, t, rA, uvalid, dbg);
          dbg_pair<NB, BITS>(a1, jp, t, rB, uvalid, dbg);
          dbg_pair<NB, BITS>(a2, jp + 1, t, rA, uvalid, dbg);
          dbg_pair<NB, BITS>(a3, jp + 1, t, rB, uvalid, dbg);
#endif
          mma_f16_16816(d[(jp / 2) % NACC], a0, a1, a2, a3, hh ? bv.z : bv.x, hh ? bv.w : bv.y);
        }
      }
    }
  }
  float D[4];
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    D[v] = d[0][v] + d[1][v];
    if constexpr (NACC == 4) D[v] += d[2][v] + d[3][v];
  }

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
      const float E = recf[PW + 2 * NB * NGM + be * NGM + c];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const uint32_t m = meta_s[(r ? rB : rA) * kMetaBox + g0 + c];
        const float sc = __half2float(__ushort_as_half((uint16_t)(m & 0xFFFFu)));
        const float ze = __half2float(__ushort_as_half((uint16_t)(m >> 16)));
        acc[r] += (sc * E) * fmaf(-ze, X, D[2 * r + cc] - C1);  // be is this lane's row
      }
    }
  }
}

// Two consecutive one-box steps of a block and tile that share a stage (batch
// 2-4): the same arithmetic as two step_mma calls, with both steps' loads and
// MMAs interleaved so that each warp has two independent MMA chains in
// flight.  The second step's box, record and meta chunks follow the first's.
template <int NB, int BITS>
__device__ __forceinline__ void step_mma_pair(uint32_t magic, int batch, int g0,
                                              const uint8_t* codes0, const uint8_t* codes1,
                                              const uint8_t* stage, const uint32_t* rec0,
                                              const uint32_t* rec1, const uint32_t* zeros,
                                              int warp, int lane, float (&acc)[2]) {
  constexpr int NGS = step_chunks(BITS, NB);
  constexpr int NGM = 8 / NB;
  constexpr int NW = lane_words(BITS, NB);
  constexpr int LW = rec_lane_words(NB);
  constexpr int PW = rec_pair_words(NB);
  constexpr int GP = group_pairs(BITS), GW = group_words(BITS);
  static_assert(nbox_of(BITS, NB) == 1 && GP % 4 == 0 && NW % GW == 0, "pair geometry");
  constexpr int GPB = NW / GW;  // groups per step
  const int g = lane >> 2, t = lane & 3;
  const int rA = warp * 16 + g, rB = rA + 8;
  const uint32_t* meta_s = reinterpret_cast<const uint32_t*>(stage + kCodesBytes);

  uint32_t wa[2][NW], wb[2][NW];
  load_words<BITS, NB>(wa[0], codes0, rA, t);
  load_words<BITS, NB>(wb[0], codes0, rB, t);
  load_words<BITS, NB>(wa[1], codes1, rA, t);
  load_words<BITS, NB>(wb[1], codes1, rB, t);

  const int my_b = g / NGS, my_c = g % NGS;
  const int dc = my_b < batch ? my_c - lane_unit(BITS, NB, t, 0) / 64 : -1000;
  const uint32_t* bs[2] = {dc == 0 ? rec0 + (my_b * 4 + t) * LW : zeros,
                           dc == 0 ? rec1 + (my_b * 4 + t) * LW : zeros};
#ifdef POLYQ_DEBUG
  const uint4 dbg0 = *reinterpret_cast<const uint4*>(stage + kDescOff + 16);
  const uint4 dbg1 = make_uint4(dbg0.w, dbg0.y, dbg0.z, 0u);
  const uint4 dsc = *reinterpret_cast<const uint4*>(stage + kDescOff);
  const int uv[2] = {(int)(dsc.y & 0xFFFFu), (int)dsc.w};
#endif

  float d[2][2][4];  // per step two accumulator sets: four independent chains
#pragma unroll
  for (int k = 0; k < 2; ++k)
#pragma unroll
    for (int q = 0; q < 2; ++q) d[k][q][0] = d[k][q][1] = d[k][q][2] = d[k][q][3] = 0.f;
#pragma unroll
  for (int qq = 0; qq < GPB; ++qq) {
#pragma unroll
    for (int m2 = 0; m2 < GP / 4; ++m2) {
      const uint4 bv0 = *reinterpret_cast<const uint4*>(bs[0] + qq * GP + 4 * m2);
      const uint4 bv1 = *reinterpret_cast<const uint4*>(bs[1] + qq * GP + 4 * m2);
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int jp = qq * GP + 4 * m2 + 2 * hh;
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const uint32_t a0 = make_pair<BITS>(wa[k], jp, magic);
          const uint32_t a1 = make_pair<BITS>(wb[k], jp, magic);
          const uint32_t a2 = make_pair<BITS>(wa[k], jp + 1, magic);
          const uint32_t a3 = make_pair<BITS>(wb[k], jp + 1, magic);
#ifdef POLYQ_DEBUG
          {
            const uint4& dg = k ? dbg1 : dbg0;
            dbg_pair<NB, BITS>(a0, jp, t, rA, uv[k], dg);
            dbg_pair<NB, BITS>(a1, jp, t, rB, uv[k], dg);
            dbg_pair<NB, BITS>(a2, jp + 1, t, rA, uv[k], dg);
            dbg_pair<NB, BITS>(a3, jp + 1, t, rB, uv[k], dg);
          }
#endif
          const uint4& bv = k ? bv1 : bv0;
          mma_f16_16816(d[k][(jp / 2) & 1], a0, a1, a2, a3, hh ? bv.z : bv.x, hh ? bv.w : bv.y);
        }
      }
    }
  }
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    float D[4];
#pragma unroll
    for (int v = 0; v < 4; ++v) D[v] = d[k][0][v] + d[k][1][v];
    const float* recf = reinterpret_cast<const float*>(k ? rec1 : rec0);
#pragma unroll
    for (int cc = 0; cc < 2; ++cc) {
      const int col = 2 * t + cc;
      const int be = col / NGS, c = col % NGS;
      if (be < batch) {
        const float C1 = recf[PW + be * NGM + c];
        const float X = recf[PW + NB * NGM + be * NGM + c];
        const float E = recf[PW + 2 * NB * NGM + be * NGM + c];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const uint32_t m = meta_s[(r ? rB : rA) * kMetaBox + g0 + k * NGS + c];
          const float sc = __half2float(__ushort_as_half((uint16_t)(m & 0xFFFFu)));
          const float ze = __half2float(__ushort_as_half((uint16_t)(m >> 16)));
          acc[r] += (sc * E) * fmaf(-ze, X, D[2 * r + cc] - C1);  // be is this lane's row
        }
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
                                        float (&acc)[2]) {
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
#ifdef POLYQ_DEBUG
    if (g_dbg_codes) {
      const uint4 dg = *reinterpret_cast<const uint4*>(stage + kDescOff + 16);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int u = 64 * h + 16 * t + i;
        const uint16_t va = (uint16_t)(wa[i / 2] >> (16 * (i & 1)));
        const uint16_t vb = (uint16_t)(wb[i / 2] >> (16 * (i & 1)));
        if (u < uvalid && (int)dg.y + rA < (int)dg.z)
          g_dbg_codes[((long long)dg.y + rA) * g_dbg_K + dg.x + u] = va;
        if (u < uvalid && (int)dg.y + rB < (int)dg.z)
          g_dbg_codes[((long long)dg.y + rB) * g_dbg_K + dg.x + u] = vb;
      }
    }
#endif
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
  // column c of D is batch row c: lane t holds rows 2t and 2t+1, and the
  // first lane of each group takes its row's value from there, times the
  // row's 2^e
  constexpr int PW = rec_pair_words(NB);
  constexpr int NGM = 8 / NB;
  const float* Erow = reinterpret_cast<const float*>(rec) + PW + 2 * NB * NGM;
  if constexpr (NB == 1) {
    // row 0 is column 0, which lane 0 of the quad holds already
    const float E = Erow[0];
#pragma unroll
    for (int r = 0; r < 2; ++r)
      if (t == 0) acc[r] += E * (d[0][2 * r] + d[1][2 * r]);
  } else {
    const int bl = lane_batch<NB>(t);
    const int src = (lane & ~3) | (bl >> 1);
    const float E = bl < batch ? Erow[bl * NGM] : 0.f;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const float v0 = __shfl_sync(0xffffffffu, d[0][2 * r] + d[1][2 * r], src);
      const float v1 = __shfl_sync(0xffffffffu, d[0][2 * r + 1] + d[1][2 * r + 1], src);
      if (lane_first<NB>(t)) acc[r] += E * ((bl & 1) ? v1 : v0);
    }
  }
}


}  // namespace gv
}  // namespace polyq
