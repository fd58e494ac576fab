// Geometry of the decode GEMV: which codes each lane reads, how it turns them
// into bf16 pairs for the m16n8k16 tensor-core MMA, and where the matching
// activation values sit in the per-step activation record.  Used by both the
// activation pre-pass and the main kernel so the two always agree.
//
// Terms
//   unit   one code of a 2/3/4-bit block, or one 4-bit nibble of an 8-bit
//          block (an 8-bit code q = lo + 16*hi is two units).
//   step   the units of one block that one work item covers per row:
//          U = 64*NG units, NG = 8/NB column groups ("chunks" of 64 units).
//   chunk  64 consecutive units; one quantisation group (b<8) or half a group
//          (b=8).  MMA column n = b*NG + chunk keeps chunks apart, so each
//          chunk gets its own fp32 dot product and its own scale/zero later.
//   lane   lane = 4*g + t of the warp: g selects the rows (g, g+8) of the
//          16-row MMA tile, t selects which units of the step it decodes.
#pragma once
#include <stdint.h>

namespace polyq {
namespace gv {

constexpr int kRows = 64;          // rows per work tile (4 consumer warps x 16)
constexpr int kWarps = 4;          // consumer warps per CTA
constexpr int kStages = 3;         // TMA pipeline depth per CTA (3 CTAs per SM)
constexpr int kPitchSplit = 144;   // row pitch of 128-byte half boxes (16 extra bytes)
constexpr int kMetaBox = 16;       // meta entries per row loaded per step
constexpr int kCodesBytes = 2 * kRows * kPitchSplit;  // largest codes area per stage (2 boxes)
constexpr int kMetaBytes = kRows * kMetaBox * 4;
constexpr int kRecMax = 1344;
constexpr int kStageBytes = ((kCodesBytes + kMetaBytes + kRecMax) + 127) / 128 * 128;
constexpr int kU16 = 128;          // 16-bit weights per row per step

__host__ __device__ constexpr int ng_of(int nb) { return 8 / nb; }
__host__ __device__ constexpr int cpl_of(int nb) { return 16 * ng_of(nb); }   // units per lane
__host__ __device__ constexpr int units_of(int nb) { return 64 * ng_of(nb); }
// bits per unit: 2, 3, 4 (8-bit blocks are read as 4-bit nibbles)
__host__ __device__ constexpr int ubits(int bits) { return bits == 8 ? 4 : bits; }
__host__ __device__ constexpr int step_bytes(int bits, int nb) {
  return bits == 16 ? 2 * kU16 : units_of(nb) * ubits(bits) / 8;
}
// A step is loaded as nbox boxes of equal byte width, box h covering bytes
// [h*SB/nbox, (h+1)*SB/nbox) of every row.  Lane t reads bytes
// [t*LB, (t+1)*LB) of each box.  A box that is 128 bytes wide gets a 144-byte
// row pitch (16 bytes of the next box ride along) so that rows g and g+1 land
// in different shared-memory banks; all other widths are conflict-free as is.
__host__ __device__ constexpr int nbox_of(int bits, int nb) { return (bits == 16 || nb == 1) ? 2 : 1; }
__host__ __device__ constexpr int box_bytes(int bits, int nb) {
  return step_bytes(bits, nb) / nbox_of(bits, nb);
}
__host__ __device__ constexpr int box_pitch(int bits, int nb) {
  return box_bytes(bits, nb) == 128 ? kPitchSplit : box_bytes(bits, nb);
}
__host__ __device__ constexpr int lane_box_bytes(int bits, int nb) { return box_bytes(bits, nb) / 4; }
__host__ __device__ constexpr int lane_words(int bits, int nb) {
  return nbox_of(bits, nb) * lane_box_bytes(bits, nb) / 4;
}
// Words per record row (one lane, one batch): pairs plus 16 bytes of padding.
__host__ __device__ constexpr int rec_lane_words(int nb) { return cpl_of(nb) / 2 + 4; }
__host__ __device__ constexpr int rec_pair_words(int nb) { return nb * 4 * rec_lane_words(nb); }
__host__ __device__ constexpr int rec_bytes(int nb) {
  return (rec_pair_words(nb) + 2 * nb * ng_of(nb)) * 4;
}
static_assert(rec_bytes(1) <= kRecMax && rec_bytes(2) <= kRecMax && rec_bytes(4) <= kRecMax, "");
static_assert(rec_bytes(1) % 16 == 0 && rec_bytes(2) % 16 == 0 && rec_bytes(4) % 16 == 0, "");

// Step-relative unit index of the i-th unit that lane t decodes.  With two
// boxes (batch 1) lane t owns chunks t and t+4, so MMA i of the lane loop
// covers the same chunk position in every lane and a partly filled step can
// stop early.
__host__ __device__ inline int lane_unit(int bits, int nb, int t, int i) {
  const int nbx = nbox_of(bits, nb);
  const int per = cpl_of(nb) / nbx;  // units per lane per box
  const int h = i / per;
  return h * (units_of(nb) / nbx) + t * per + (i % per);
}

// 16-bit steps: step-relative weight index of the lane's i-th weight (i < 32).
__host__ __device__ inline int lane_weight16(int t, int i) {
  return 64 * (i / 16) + 16 * t + (i % 16);
}

// ---------------------------------------------------------------------------
// Pair tables.  A pair register holds two bf16 values 128 + q*2^p (exact):
// (window >> 0 & mask) | 0x43004300 where the mask selects code `lo` at bit p_lo
// of the low half and code `hi` at bit 16 + p_hi.  The activation matching the
// pair is (x_lo * 2^-p_lo, x_hi * 2^-p_hi).
// ---------------------------------------------------------------------------
struct PairDef {
  int8_t win;  // window offset in bits (negative: shift left)
  int8_t lo, plo, hi, phi;  // units relative to the group, bit positions
};

// 2-bit: one word = 16 units, 8 pairs, windows at 0, 6, 12.
__host__ __device__ inline PairDef pair2(int j) {
  const int8_t sh[8] = {0, 0, 0, 6, 6, 6, 12, 12};
  const int8_t p[8] = {0, 2, 4, 0, 2, 4, 0, 2};
  return PairDef{sh[j], (int8_t)j, p[j], (int8_t)(j + 8), p[j]};
}
// 4-bit (and 8-bit nibbles): one word = 8 units, 4 pairs (c, c+4).
__host__ __device__ inline PairDef pair4(int j) {
  return PairDef{(int8_t)(4 * j), (int8_t)j, 0, (int8_t)(j + 4), 0};
}
// 3-bit: three words = 32 units, 16 pairs.  Window offsets -1, 5, 11, 29, 35,
// 41, 59, 64, 69, 72, 77 (eleven windows, one of them a plain word).
__host__ __device__ inline PairDef pair3(int j) {
  const int8_t t[16][5] = {{-1, 0, 1, 5, 0},   {-1, 1, 4, 6, 3},   {5, 2, 1, 7, 0},
                           {5, 3, 4, 8, 3},    {11, 4, 1, 9, 0},   {29, 10, 1, 15, 0},
                           {29, 11, 4, 16, 3}, {35, 12, 1, 17, 0}, {35, 13, 4, 18, 3},
                           {41, 14, 1, 19, 0}, {59, 20, 1, 25, 0}, {59, 21, 4, 26, 3},
                           {64, 22, 2, 28, 4}, {69, 23, 0, 29, 2}, {72, 24, 0, 30, 2},
                           {77, 27, 4, 31, 0}};
  return PairDef{t[j][0], t[j][1], t[j][2], t[j][3], t[j][4]};
}
__host__ __device__ constexpr int group_units(int ub) { return ub == 3 ? 32 : 32 / ub; }
__host__ __device__ constexpr int group_pairs(int ub) { return group_units(ub) / 2; }
__host__ __device__ constexpr int group_words(int ub) { return ub == 3 ? 3 : 1; }
__host__ __device__ inline PairDef pair_def(int ub, int j) {
  return ub == 2 ? pair2(j) : ub == 3 ? pair3(j) : pair4(j);
}

// Lane-unit indices (0..CPL-1) of the two halves of lane pair j.
__host__ __device__ inline void pair_units(int ub, int j, int* ulo, int* plo, int* uhi,
                                           int* phi) {
  const int gp = group_pairs(ub);
  const PairDef d = pair_def(ub, j % gp);
  const int base = (j / gp) * group_units(ub);
  *ulo = base + d.lo;
  *plo = d.plo;
  *uhi = base + d.hi;
  *phi = d.phi;
}

// Step-relative chunk (0..NG-1) that lane t's pair j belongs to.
__host__ __device__ inline int pair_chunk(int bits, int nb, int t, int j) {
  const int ub = ubits(bits);
  const int base = (j / group_pairs(ub)) * group_units(ub);
  return lane_unit(bits, nb, t, base) / 64;
}

}  // namespace gv
}  // namespace polyq
