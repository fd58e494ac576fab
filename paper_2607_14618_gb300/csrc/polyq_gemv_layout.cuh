// Geometry of the decode GEMV: which codes each lane reads, how it turns them
// into fp16 pairs for the m16n8k16 tensor-core MMA, and where the matching
// activation values sit in the per-step activation record.  The record
// builder and the MMA loop both use these tables, so the two always agree.
//
// Terms
//   unit   one code of a 2/3/4/8-bit block (or one fp16 weight of a 16-bit
//          block).
//   step   the units of one block that one work item covers per row: U units,
//          U = 64 * NGS chunks (NGS <= 8 / NB, see step_units()).
//   chunk  64 consecutive units = one quantisation group.  MMA column
//          n = b * NGS + chunk keeps chunks (and batch rows b) apart, so each
//          chunk gets its own fp32 dot product and its own scale/zero.
//   box    a step is loaded as nbx TMA boxes of 64 rows; box h holds units
//          [h*U/nbx, (h+1)*U/nbx) of every row.
//   lane   lane = 4*g + t of the warp: g selects the rows (g, g+8) of the
//          16-row MMA tile, t selects which units of each box it decodes:
//          units [t*per, (t+1)*per) of the box, per = U / (4*nbx).
#pragma once
#include <stdint.h>

namespace polyq {
namespace gv {

constexpr int kRows = 64;          // rows per work tile (4 consumer warps x 16)
constexpr int kWarps = 4;          // consumer warps per CTA
constexpr int kStages = 3;         // TMA pipeline depth per CTA (3 CTAs per SM)
constexpr int kPitchSplit = 144;   // row pitch of 128-byte boxes (16 extra bytes)
constexpr int kMetaBox = 12;       // meta entries per row loaded per step
constexpr int kCodesBytes = 2 * kRows * kPitchSplit;  // largest codes area (2 boxes)
constexpr int kMetaBytes = kRows * kMetaBox * 4;
constexpr int kRecOne = 1376;      // largest activation record (NB = 4)
constexpr int kRecMax = 2 * kRecOne;  // a stage may hold two steps' records
// A stage holds an item's code boxes, its scale/zero box, its record(s) and
// a 16-byte descriptor written by the producer.  At batch 2-4 a step whose
// codes take one box can share its stage with the next step of the same
// block and tile (the second step's box follows the first, both records
// follow each other).
constexpr int kRecOff = kCodesBytes + kMetaBytes;
constexpr int kDescOff = kRecOff + kRecMax;
// the descriptor, and 16 bytes that only the debug build writes
constexpr int kStageBytes = ((kDescOff + 32) + 127) / 128 * 128;
constexpr uint32_t kMagic = 0x64006400u;  // two fp16 1024.0
constexpr float kMagicF = 1024.0f;

// Units per step: 64 * 8/NB for 2/3/4-bit; at most 256 for 8-bit (so a step
// row stays within 256 bytes); 128 fp16 weights for 16-bit.
__host__ __device__ constexpr int step_units(int bits, int nb) {
  return bits == 16 ? 128 : (bits == 8 ? (nb == 4 ? 128 : 256) : 64 * (8 / nb));
}
__host__ __device__ constexpr int step_chunks(int bits, int nb) {  // NGS
  return bits == 16 ? 1 : step_units(bits, nb) / 64;
}
__host__ __device__ constexpr int step_bytes(int bits, int nb) {
  return step_units(bits, nb) * bits / 8;
}
// Two boxes at batch 1 (so a half-filled step can skip its second half) and
// whenever a step row is wider than 128 bytes; otherwise one.
__host__ __device__ constexpr int nbox_of(int bits, int nb) {
  return (nb == 1 || step_bytes(bits, nb) > 128) ? 2 : 1;
}
__host__ __device__ constexpr int box_bytes(int bits, int nb) {
  return step_bytes(bits, nb) / nbox_of(bits, nb);
}
// A box that is 128 bytes wide gets a 144-byte row pitch so that rows g and
// g+1 land in different shared-memory banks; other widths are conflict-free.
__host__ __device__ constexpr int box_pitch(int bits, int nb) {
  return box_bytes(bits, nb) == 128 ? kPitchSplit : box_bytes(bits, nb);
}
__host__ __device__ constexpr int lane_box_bytes(int bits, int nb) { return box_bytes(bits, nb) / 4; }
__host__ __device__ constexpr int lane_words(int bits, int nb) {
  return nbox_of(bits, nb) * lane_box_bytes(bits, nb) / 4;
}
// units per lane per box
__host__ __device__ constexpr int lane_per(int bits, int nb) {
  return step_units(bits, nb) / (4 * nbox_of(bits, nb));
}
// Pairs per lane per step.
__host__ __device__ constexpr int lane_pairs(int bits, int nb) {
  return step_units(bits, nb) / 8;
}

// Record: for each batch row b and lane t, LW words of fp16 pairs (the lane's
// pairs in order, then 16 bytes of padding); then C1[b][8/NB], X[b][8/NB] and
// E[b][8/NB] (fp32).  The record holds each activation as x * 2^-(e+p): e is
// the chunk's exponent (kRecExp below), p the one its code carries.
// C1 = 1024 * sum x' and X = sum x' * 2^p over the chunk, in those scaled
// units, and E = 2^e multiplies the chunk's result back.  A 16-bit step has
// one exponent per batch row, in E[b][0].
__host__ __device__ constexpr int rec_lane_words(int nb) { return 64 / nb + 4; }
__host__ __device__ constexpr int rec_pair_words(int nb) { return nb * 4 * rec_lane_words(nb); }
__host__ __device__ constexpr int rec_bytes(int nb) {
  return (rec_pair_words(nb) + 3 * nb * (8 / nb)) * 4;
}
// Each chunk is scaled by the power of two 2^-e that brings its largest
// magnitude into [2^kRecExp, 2^(kRecExp+1)): every value then rounds to fp16
// without overflow, and values down to 2^-(kRecExp+14-8) of the chunk's
// largest stay fp16 normals even after the decoder's 2^-p (p <= 8).
constexpr int kRecExp = 14;
constexpr int kRecExpMin = -126;  // 2^e stays a normal float
static_assert(rec_bytes(1) <= kRecOne && rec_bytes(2) <= kRecOne && rec_bytes(4) <= kRecOne, "");
static_assert(rec_bytes(1) % 16 == 0 && rec_bytes(2) % 16 == 0 && rec_bytes(4) % 16 == 0, "");
static_assert(lane_pairs(2, 1) + 4 <= rec_lane_words(1) && lane_pairs(2, 4) + 4 <= rec_lane_words(4), "");

// Step-relative unit index of the i-th unit that lane t decodes.
__host__ __device__ inline int lane_unit(int bits, int nb, int t, int i) {
  const int per = lane_per(bits, nb);
  const int h = i / per;
  return h * (step_units(bits, nb) / nbox_of(bits, nb)) + t * per + (i % per);
}

// ---------------------------------------------------------------------------
// Pair tables.  A pair register holds two fp16 values 1024 + q*2^p (exact):
// (window & mask) | 0x64006400, the mask selecting code `lo` at bit p_lo of
// the low half and code `hi` at bit 16 + p_hi (both within the 10 mantissa
// bits).  The window is bits [win, win+32) of the group's little-endian code
// stream.  The activation matching the pair is (x_lo * 2^-p_lo, x_hi * 2^-p_hi).
// ---------------------------------------------------------------------------
struct PairDef {
  int8_t win;  // window offset in bits (negative: shift left)
  int8_t lo, plo, hi, phi;  // codes relative to the group, bit positions
};

// 2-bit: one word = 16 codes, 8 pairs, windows at 0 and 10.
__host__ __device__ inline PairDef pair2(int j) {
  return j < 5 ? PairDef{0, (int8_t)j, (int8_t)(2 * j), (int8_t)(j + 8), (int8_t)(2 * j)}
               : PairDef{10, (int8_t)j, (int8_t)(2 * (j - 5)), (int8_t)(j + 8),
                         (int8_t)(2 * (j - 5))};
}
// 4-bit: one word = 8 codes, 4 pairs (c, c+4), windows at 0 and 8.
__host__ __device__ inline PairDef pair4(int j) {
  const int w = (j >> 1) * 8;
  const int c = (j >> 1) * 2 + (j & 1);
  return PairDef{(int8_t)w, (int8_t)c, (int8_t)(4 * (j & 1)), (int8_t)(c + 4),
                 (int8_t)(4 * (j & 1))};
}
// 8-bit: two words = 8 codes, 4 pairs (c, c+2) of each word, windows 0, 8,
// 32, 40.
__host__ __device__ inline PairDef pair8(int j) {
  const int word = j >> 1, c = (j >> 1) * 4 + (j & 1);
  return PairDef{(int8_t)(32 * word + 8 * (j & 1)), (int8_t)c, 0, (int8_t)(c + 2), 0};
}
// 3-bit: three words = 32 codes, 16 pairs, seven windows: -7, 1, 11, 32, 41,
// 62, 71 (found by exhaustive search for the fewest windows).
__host__ __device__ inline PairDef pair3(int j) {
  const int8_t t[16][5] = {{-7, 0, 7, 3, 0},   {1, 1, 2, 7, 4},    {1, 2, 5, 8, 7},
                           {11, 4, 1, 9, 0},   {11, 5, 4, 10, 3},  {11, 6, 7, 11, 6},
                           {32, 12, 4, 17, 3}, {32, 13, 7, 18, 6}, {41, 14, 1, 19, 0},
                           {41, 15, 4, 20, 3}, {41, 16, 7, 21, 6}, {62, 22, 4, 27, 3},
                           {62, 23, 7, 28, 6}, {71, 24, 1, 29, 0}, {71, 25, 4, 30, 3},
                           {71, 26, 7, 31, 6}};
  return PairDef{t[j][0], t[j][1], t[j][2], t[j][3], t[j][4]};
}
__host__ __device__ constexpr int group_units(int bits) { return bits == 3 ? 32 : bits == 2 ? 16 : 8; }
__host__ __device__ constexpr int group_pairs(int bits) { return group_units(bits) / 2; }
__host__ __device__ constexpr int group_words(int bits) { return bits == 3 ? 3 : bits == 8 ? 2 : 1; }
__host__ __device__ inline PairDef pair_def(int bits, int j) {
  return bits == 2 ? pair2(j) : bits == 3 ? pair3(j) : bits == 4 ? pair4(j) : pair8(j);
}

// Lane-unit indices (0..per*nbx-1) of the two halves of lane pair j.
__host__ __device__ inline void pair_units(int bits, int j, int* ulo, int* plo, int* uhi,
                                           int* phi) {
  const int gp = group_pairs(bits);
  const PairDef d = pair_def(bits, j % gp);
  const int base = (j / gp) * group_units(bits);
  *ulo = base + d.lo;
  *plo = d.plo;
  *uhi = base + d.hi;
  *phi = d.phi;
}

// The 32 lane pairs that cover chunk c of a step: the q-th of them is pair jp
// of lane t.
__host__ __device__ inline void chunk_pair(int bits, int nb, int c, int q, int* t, int* jp) {
  const int per = lane_per(bits, nb);
  const int cpb = step_units(bits, nb) / nbox_of(bits, nb) / 64;  // chunks per box
  const int h = c / cpb, cb = c % cpb;
  const int lpc = 64 / per;  // lanes per chunk (1 or 2)
  *t = cb * lpc + q / (per / 2);
  *jp = h * (per / 2) + q % (per / 2);
}

// 16-bit steps: step-relative weight index of the lane's i-th weight (i < 32):
// lane t holds weights [16t, 16t+16) of each 64-weight box.
__host__ __device__ inline int lane_weight16(int t, int i) {
  return 64 * (i / 16) + 16 * t + (i % 16);
}

}  // namespace gv
}  // namespace polyq
