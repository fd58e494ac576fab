// Decode GEMV of the PolyQ mixed-bit layer (Section 4.1 factorisation with
// the Section 4.2 bit blocks), one launch over all blocks of one or several
// independent layers:
//
//   y[b][n] = residual[b][n] + sum_p x[b][gather[p]] * t[p] * W'[n][p]
//
// (t = the Section 3.4 activation factors of a scaled layer, else 1.)
//
// Two kernels per call, chained with programmatic dependent launch:
//  * gemv_prep, one 256-thread CTA per (layer, step) and a few more CTAs
//    that set y to the residual (or zero): gathers x through `gather`,
//    scales each value by the power of two that the decoder leaves on its
//    code (and by its chunk's exponent), rounds it to fp16 and stores the
//    step's activation record together with per-chunk sums for the
//    magic-number and zero-point corrections.  The gather indices are loaded
//    before the wait for the previous kernel.
//  * gemv_main, persistent, 160 threads per CTA, 3 CTAs per SM.  The (layer,
//    64-row tile, step) work items of all layers of the call form one list;
//    each CTA takes a contiguous range of it.  Warp 4 (one thread) streams
//    each item's packed codes and scale/zero metadata with TMA through a
//    3-stage shared-memory ring, the first stage before the grid-dependency
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
#ifdef POLYQ_DEBUG
#include "polyq_debug.h"
#endif
#include "polyq_dev.cuh"
#include "polyq_gemv_dev.cuh"
#include "polyq_gemv_layout.cuh"
#include "polyq_internal.h"

namespace {

using namespace polyq;
using namespace polyq::gv;

constexpr int kCtasPerSm = 3;

// Bounded wait that also gives up once another warp of the CTA has failed
// (`abort` set): true when the phase completed.  The flag is read only after
// a poll has failed, so a stage whose barrier has already completed costs one
// poll and no shared load.
__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity,
                                              const volatile int* abort) {
  for (uint32_t it = 0; it < kWaitLimit; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
  }
  return false;
}
constexpr int kMaxGrid = 1024;  // persistent CTAs at most
constexpr uint32_t kDescEnd = 0x200u;   // descriptor flag: no more items
constexpr uint32_t kDescPair = 0x400u;  // descriptor flag: the stage holds two steps


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
  int clear_status;  // 1: the pre-pass zeroes the status word first
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

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// y starts as the residual (or zero); the main kernel adds its pieces.  Done
// by CTAs of the pre-pass that build no record (CTA `cta` of `n_cta`), in
// parallel with those that do.
__device__ __forceinline__ void init_outputs(const GvParams& P, int cta, int n_cta) {
  // 16-byte stores (and residual loads) where y and the residual allow them;
  // a thread's loads of one round are in flight together.
#pragma unroll
  for (int q = 0; q < POLYQ_MAX_GROUP; ++q) {
    if (q >= P.n_layers) break;
    float* y = P.L[q].y;
    const float* res = P.L[q].residual;
    if (y == res) continue;
    const int total = P.batch * P.L[q].N;
    const int st = n_cta * blockDim.x;
    const int t0 = cta * blockDim.x + threadIdx.x;
    const bool vec = total % 4 == 0 && reinterpret_cast<uintptr_t>(y) % 16 == 0 &&
                     reinterpret_cast<uintptr_t>(res) % 16 == 0;
    if (vec) {
      float4* y4 = reinterpret_cast<float4*>(y);
      const float4* r4 = reinterpret_cast<const float4*>(res);
      const int n4 = total / 4;
      for (int i0 = t0; i0 < n4; i0 += 2 * st) {
        float4 v[2];
#pragma unroll
        for (int u = 0; u < 2; ++u)
          v[u] = (res && i0 + u * st < n4) ? r4[i0 + u * st] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 2; ++u)
          if (i0 + u * st < n4) y4[i0 + u * st] = v[u];
      }
    } else {
      for (int i0 = t0; i0 < total; i0 += 4 * st) {
        float v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = (res && i0 + u * st < total) ? res[i0 + u * st] : 0.f;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (i0 + u * st < total) y[i0 + u * st] = v[u];
      }
    }
  }
}

// ---------------------------------------------------------------------------
// pre-pass: one CTA of 256 threads per activation record (layer, step); each
// thread builds at most one (batch, chunk) slot of it, which keeps the chain
// of dependent instructions between the activation loads and the record
// stores short.  A few more CTAs initialise the outputs.
// ---------------------------------------------------------------------------
constexpr int kPrepWarps = 8;
constexpr int kPrepThreads = 32 * kPrepWarps;

template <int NB>
__global__ void __launch_bounds__(kPrepThreads) gemv_prep(const __grid_constant__ GvParams P) {
  pdl_trigger();  // the main kernel may start streaming weights right away
  if ((int)blockIdx.x >= P.recs) {
    pdl_wait();  // y may still be in use by earlier kernels
    init_outputs(P, (int)blockIdx.x - P.recs, (int)gridDim.x - P.recs);
    return;
  }
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
  rec_sources<NB, kPrepWarps>(in, S.blk[l][bi], j, warp, lane, s_p3, src, fac);  // static layer data
  if (P.xkind == POLYQ_X_RMSNORM) rms_prefetch(P.xa, P.L[0].K, P.batch);
  pdl_wait();  // x comes from the previous kernel; the records and y may still be in use
  // The streaming kernel writes the status only after its own wait for this
  // grid, so clearing it here cannot lose one of its reports.
  if (P.clear_status && blockIdx.x == 0 && threadIdx.x == 0) *P.status = 0;
  float ra[2][2], rb[2][2];
  rec_load<NB, kPrepWarps>(in, S.blk[l][bi], j, warp, lane, s_p3, src, ra, rb);
  __shared__ float s_rnorm[4];
  __shared__ float s_part[4][kPrepWarps];
  if (P.xkind == POLYQ_X_RMSNORM)
    rms_rnorm<kPrepWarps>(P.xa, P.L[0].K, P.batch, P.eps, s_part, s_rnorm);
  rec_store<NB, kPrepWarps>(in, S.blk[l][bi], j, warp, lane, s_p3, src, fac, ra, rb, s_rnorm,
                            reinterpret_cast<uint32_t*>(P.rec + (size_t)r * rec_bytes(NB)));
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

  if (warp == kWarps) {
    // ---------------- producer ----------------
    // The packed weights do not depend on earlier kernels: request the first
    // stage before the grid-dependency wait (more would compete for DRAM with
    // the pre-pass's activation loads, which are on the critical path).  The
    // activation records come from this call's pre-pass and are loaded after
    // it.
    ItemPos it;
    int item = lo;
    if (lo < hi) it.init(S, nl, lo);
    int rec_a[kStages], rec_b[kStages];  // records of each stage's steps (-1: none)
    // Weights of a stage: one item, or at batch 2-4 two consecutive steps of
    // one block and tile whose codes take one box each.  A stage is planned
    // (its descriptor and copy coordinates, from the shared layer tables)
    // before the wait for its slot, and issued after it.
    struct Plan {
      uint4 d;
#ifdef POLYQ_DEBUG
      uint4 dbg;
#endif
      const CUtensorMap* tm;
      const CUtensorMap* tm_meta;
      int nbx, pitch, x0, xstep, x2, xmeta, y, pair, rec_a;
      uint32_t bytes;
    };
    auto plan_stage = [&](Plan& p) {
      const GvBlock& B = S.blk[it.l][it.bi];
      int sb, nbx, pitch;
      switch (B.bits) {
        case 2: sb = step_bytes(2, NB); nbx = nbox_of(2, NB); pitch = box_pitch(2, NB); break;
        case 3: sb = step_bytes(3, NB); nbx = nbox_of(3, NB); pitch = box_pitch(3, NB); break;
        case 4: sb = step_bytes(4, NB); nbx = nbox_of(4, NB); pitch = box_pitch(4, NB); break;
        case 8: sb = step_bytes(8, NB); nbx = nbox_of(8, NB); pitch = box_pitch(8, NB); break;
        default: sb = step_bytes(16, NB); nbx = nbox_of(16, NB); pitch = box_pitch(16, NB); break;
      }
      const bool pair = NB > 1 && nbx == 1 && item + 1 < hi && it.j + 1 < B.n_steps;
      const int j2 = it.j + 1;
      // what the consumers need: width, whether the stage ends a tile
      // piece, pairing, layer, valid units of each step, first meta entry,
      // tile
      const int uvalid = min(B.units, B.n_ch - it.j * B.units);
      const int uvalid2 = pair ? min(B.units, B.n_ch - j2 * B.units) : 0;
      const int g0 = (B.grp_off + it.j * (B.units / 64)) & 3;
      const int last_s = it.s + (pair ? 1 : 0);
      const bool flush = last_s == S.steps[it.l] - 1 || item + (pair ? 2 : 1) == hi;
      p.d.x = (uint32_t)B.bits | ((uint32_t)flush << 8) | ((uint32_t)pair << 10) |
              ((uint32_t)it.l << 16);
      p.d.y = (uint32_t)uvalid | ((uint32_t)g0 << 16);
      p.d.z = (uint32_t)it.tile;
      p.d.w = (uint32_t)uvalid2;
#ifdef POLYQ_DEBUG
      p.dbg = make_uint4((uint32_t)(B.pos0 + it.j * B.units), (uint32_t)(it.tile * kRows),
                         (uint32_t)S.N[it.l], (uint32_t)(B.pos0 + j2 * B.units));
#endif
      p.bytes = (pair ? 2 : 1) * (nbx * pitch * kRows + RB);
      if (B.bits < 16) p.bytes += kMetaBytes;
      p.tm = &P.L[it.l].tm_codes[it.bi];
      p.tm_meta = B.bits < 16 ? &P.L[it.l].tm_meta : nullptr;
      p.nbx = nbx;
      p.pitch = pitch;
      p.x0 = B.seg_off + it.j * sb;
      p.xstep = sb / nbx;
      p.x2 = B.seg_off + j2 * sb;
      // one box of kMetaBox groups covers both steps of a pair
      p.xmeta = (B.grp_off + it.j * (B.units / 64)) & ~3;
      p.y = it.tile * kRows;
      p.pair = pair;
      p.rec_a = S.rec0[it.l] + it.s;
      it.next(S, nl);
      ++item;
      if (pair) {
        it.next(S, nl);
        ++item;
      }
    };
    auto issue_stage = [&](int k, const Plan& p) {
      const int slot = k % kStages;
      const uint32_t dst = smem_u32(stages + slot * kStageBytes);
      const uint32_t bar = full0 + 8 * slot;
      *reinterpret_cast<uint4*>(stages + slot * kStageBytes + kDescOff) = p.d;
#ifdef POLYQ_DEBUG
      *reinterpret_cast<uint4*>(stages + slot * kStageBytes + kDescOff + 16) = p.dbg;
#endif
      mbar_expect_tx(bar, p.bytes);
      for (int h = 0; h < p.nbx; ++h)
        tma_load_2d(dst + h * kRows * p.pitch, p.tm, p.x0 + h * p.xstep, p.y, bar);
      if (p.pair) tma_load_2d(dst + kRows * p.pitch, p.tm, p.x2, p.y, bar);
      if (p.tm_meta) tma_load_2d(dst + kCodesBytes, p.tm_meta, p.xmeta, p.y, bar);
      rec_a[slot] = p.rec_a;
      rec_b[slot] = p.pair ? p.rec_a + 1 : -1;
    };
    auto issue_records = [&](int k) {
      const int slot = k % kStages;
      const uint32_t dst = smem_u32(stages + slot * kStageBytes + kRecOff);
      // a paired stage's two records are consecutive: one copy
      bulk_load(dst, P.rec + (size_t)rec_a[slot] * RB, (rec_b[slot] >= 0 ? 2 : 1) * RB,
                full0 + 8 * slot);
    };
    int ks = 0;  // stages issued
    if (lane == 0) {
      for (int l = 0; l < nl; ++l) {
        for (int b = 0; b < S.n_blocks[l]; ++b) prefetch_tmap(&P.L[l].tm_codes[b]);
        prefetch_tmap(&P.L[l].tm_meta);
      }
      if (item < hi) {
        Plan p0;
        plan_stage(p0);
        issue_stage(ks++, p0);
      }
    }
    pdl_wait();  // the records come from the pre-pass of this call
    fence_proxy_async_global();  // it wrote them through the generic proxy
    if (lane != 0) return;
    if (ks > 0) issue_records(0);
    // At batch 2-4, where the producer's per-stage work is on the ring's
    // critical path, the next stage is planned while its slot is still in
    // use; at batch 1 after the wait (measured 0.7% faster there).
    constexpr bool kPlanAhead = NB > 1;
    bool ok = true;
    Plan pn;
    bool have = item < hi;
    if (kPlanAhead && have) plan_stage(pn);
    while (have) {
      const int slot = ks % kStages;
      if (ks >= kStages && !wait_or_abort(empty0 + 8 * slot, ((ks / kStages) - 1) & 1, &s_abort)) {
        if (!s_abort) atomicExch(P.status, kStatusTimeoutEmpty);
        s_abort = 1;
        ok = false;
        break;
      }
      if (!kPlanAhead) plan_stage(pn);
      issue_stage(ks, pn);
      issue_records(ks);
      ++ks;
      have = item < hi;
      if (kPlanAhead && have) plan_stage(pn);
    }
    // wait (bounded) for the copies still in flight, then mark the end of
    // the items in the next stage
    for (int k = max(0, ks - kStages); k < ks; ++k)
      mbar_wait(full0 + 8 * (k % kStages), (k / kStages) & 1);
    if (ok) {
      const int slot = ks % kStages;
      if (ks < kStages || mbar_wait(empty0 + 8 * slot, ((ks / kStages) - 1) & 1)) {
        *reinterpret_cast<uint4*>(stages + slot * kStageBytes + kDescOff) =
            make_uint4(kDescEnd, 0u, 0u, 0u);
        mbar_arrive(full0 + 8 * slot);
      } else {
        atomicExch(P.status, kStatusTimeoutEmpty);
        s_abort = 1;
      }
    }
    return;
  }

  // ---------------- consumers ----------------
  pdl_wait();  // y, the workspace and the records are this call's from here on
  float acc[2] = {0.f, 0.f};  // this lane's row sums (see lane_batch)
  int slot = 0;
  uint32_t phase = 0;
  for (;;) {
    if (!wait_or_abort(full0 + 8 * slot, phase, &s_abort)) {
      if (lane == 0 && !s_abort) atomicExch(P.status, kStatusTimeoutFull);
      s_abort = 1;
      break;
    }
    const uint8_t* stage = stages + slot * kStageBytes;
    const uint32_t* rec = reinterpret_cast<const uint32_t*>(stage + kRecOff);
    const uint4 desc = *reinterpret_cast<const uint4*>(stage + kDescOff);
    if (desc.x & kDescEnd) break;
    const int bits = (int)(desc.x & 0xFFu);
    const int uvalid = (int)(desc.y & 0xFFFFu), g0 = (int)(desc.y >> 16);
    if (NB > 1 && (desc.x & kDescPair)) {
      // two steps of one block and tile: the second one's box follows the
      // first, its record follows the first record, its chunks follow in the
      // meta box (the valid-unit counts are not needed: units past a block's
      // end carry zero activations)
      if constexpr (NB > 1) {
        const uint32_t* rec2 = rec + RB / 4;
        switch (bits) {
          case 2: step_mma_pair<NB, 2>(P.magic, P.batch, g0, stage, stage + kRows * box_pitch(2, NB), stage, rec, rec2, zeros, warp, lane, acc); break;
          case 3: step_mma_pair<NB, 3>(P.magic, P.batch, g0, stage, stage + kRows * box_pitch(3, NB), stage, rec, rec2, zeros, warp, lane, acc); break;
          case 4: step_mma_pair<NB, 4>(P.magic, P.batch, g0, stage, stage + kRows * box_pitch(4, NB), stage, rec, rec2, zeros, warp, lane, acc); break;
          default:  // 8-bit steps take one box, so pair, only at batch 4
            if constexpr (nbox_of(8, NB) == 1)
              step_mma_pair<NB, 8>(P.magic, P.batch, g0, stage, stage + kRows * box_pitch(8, NB), stage, rec, rec2, zeros, warp, lane, acc);
            break;
        }
      }
    } else {
      switch (bits) {
        case 2: step_mma<NB, 2>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
        case 3: step_mma<NB, 3>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
        case 4: step_mma<NB, 4>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
        case 8: step_mma<NB, 8>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
        default: step_16<NB>(P.batch, uvalid, stage, rec, zeros, warp, lane, acc); break;
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty0 + 8 * slot);
    if (++slot == kStages) {
      slot = 0;
      phase ^= 1u;
    }

    if (desc.x & 0x100u) {
      // ---- add this warp's 16 rows of the tile piece into y ----
      // A tile whose steps are split over CTAs gets one addition per piece.
      const int l = (int)(desc.x >> 16);
      float* y = P.L[0].y;
      int N = P.L[0].N;
#pragma unroll
      for (int q = 1; q < POLYQ_MAX_GROUP; ++q)
        if (q == l) {
          y = P.L[q].y;
          N = P.L[q].N;
        }
      flush_rows<NB>(acc, y, N, P.batch, (int)desc.z * kRows + warp * 16, lane);
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

// CTAs of one launch: persistent, one wave of them (never more than the
// device holds at once) and no more than there are work items.
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
  // record CTAs, then output-initialising CTAs (eight floats per thread)
  long long init = 0;
  for (int q = 0; q < P.n_layers; ++q)
    if (P.L[q].y != P.L[q].residual) init += (long long)P.batch * P.L[q].N;
  const int n_init = (int)std::min<long long>(64, (init + 8 * kPrepThreads - 1) / (8 * kPrepThreads));
  cfg.gridDim = dim3((unsigned)(P.recs + n_init));
  cfg.blockDim = dim3(kPrepThreads);
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
               size_t ws_bytes, cudaStream_t st, const polyq_gemv_input* in = nullptr,
               bool clear_status = false) {
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
  P.clear_status = clear_status ? 1 : 0;
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

#ifdef POLYQ_DEBUG
// Debug build only: polyq_linear_gemv with every code the streaming kernel
// decodes written to codes_out [N][K] (uint16, clustered order).
extern "C" int polyq_debug_gemv_codes(const polyq_dev_layer* L, const void* x, int batch, float* y,
                                      void* workspace, size_t ws_bytes, uint16_t* codes_out,
                                      void* stream) {
  polyq_clear_error();
  cudaStream_t st = (cudaStream_t)stream;
  const long long K = L ? L->K : 0;
  cudaError_t e = cudaMemcpyToSymbolAsync(g_dbg_codes, &codes_out, sizeof codes_out, 0,
                                          cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyToSymbolAsync(g_dbg_K, &K, sizeof K, 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return polyq_set_error(POLYQ_ECUDA, "debug: %s", cudaGetErrorString(e));
  const int rc = polyq_linear_gemv(L, x, batch, y, nullptr, workspace, ws_bytes, stream);
  uint16_t* none = nullptr;
  cudaMemcpyToSymbolAsync(g_dbg_codes, &none, sizeof none, 0, cudaMemcpyHostToDevice, st);
  cudaStreamSynchronize(st);
  return rc;
}
#endif

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
// status word and the activation records live in this fixed array, one copy
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
  const void* xs[1] = {x};
  float* ys[1] = {y};
  const float* rs[1] = {residual};
  // The status word must start at zero, and this caller cannot reset the
  // library's array: the call's pre-pass clears it (after its wait for the
  // previous kernel, so the previous call's status is readable until then).
  return gemv_group(who, one, 1, xs, batch, ys, rs, scratch, POLYQ_NOALLOC_SCRATCH_BYTES,
                    (cudaStream_t)stream, nullptr, /*clear_status=*/true);
}

extern "C" int polyq_noalloc_status(int* status, void* stream) {
  polyq_clear_error();
  if (!status) return polyq_set_error(POLYQ_EINVAL, "polyq_noalloc_status: status is NULL");
  void* scratch = nullptr;
  int rc = noalloc_scratch(&scratch);
  if (rc) return rc;
  return polyq_workspace_status(scratch, status, stream);
}
