// Chained decode GEMVs: every phase of a decoder's decode step (each phase
// the Section 4.1 product of one to eight layers that read one input) in one
// persistent launch.
//
// One CTA per resident slot (3 per SM, all co-resident: cooperative launch).
//  * Warp 4, one thread, streams the packed codes and scale/zero boxes of
//    the CTA's items of phase 0, 1, 2, ... through a 3-stage TMA ring without
//    stopping at phase boundaries (the weights are static), and adds each
//    item's activation record once every record of its phase has been built
//    (a per-phase counter in the workspace).
//  * Warps 0-3 (16 rows each) run the phases in order.  A grid-wide barrier
//    (an arrival counter) separates phases, because phase p+1 reads what
//    phase p wrote.  After it, CTA b builds record b (b+G, ...) of the phase
//    into the workspace: gather, transform (RMSNorm, SiLU * up, rounding to
//    bf16), activation factor, fp16 rounding, per-chunk sums.  The warps then
//    set the next phase's outputs to its residual (or zero) and decode and
//    multiply their items exactly as the per-call kernel does, adding each
//    tile piece's rows into y with fp32 atomics.
// Items of a phase are (layer, tile, step) in tile-major order, split into
// contiguous ranges of equal modelled cost, so each CTA streams the rows of
// a few tiles from start to end.  Every wait is bounded; a wait that gives
// up records a status, makes the CTA skip the rest, waits (bounded) for its
// own copies in flight and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <new>
#include <vector>

#include "polyq.h"
#include "polyq_dev.cuh"
#include "polyq_gemv_dev.cuh"
#include "polyq_gemv_layout.cuh"
#include "polyq_internal.h"

namespace {

using namespace polyq;
using namespace polyq::gv;

constexpr int kChCtasPerSm = 3;
constexpr int kChMaxGrid = 1024;
// Polls of a grid barrier or a record counter before giving up (each poll
// sleeps at least 128-256 ns and reads L2): about a second, against waits of
// microseconds in a working launch.
constexpr uint32_t kGridWaitLimit = 1u << 21;
constexpr int kItemFixedCost = 2048;  // per-item overhead in the cost model, bytes
// workspace: status word at 0; barrier arrivals, CTAs done and the launch
// count at 64; per-phase record-ready counters from 256; then the records
constexpr size_t kWsCounters = 64;
constexpr size_t kWsReady = 256;

struct ChLayer {
  CUtensorMap tm_codes[POLYQ_MAX_BLOCKS];
  CUtensorMap tm_meta;
  GvBlock blk[POLYQ_MAX_BLOCKS];
  int n_blocks, N, K, steps, tiles, item0, rec0, pad;
  const __nv_bfloat16* x;  // POLYQ_X_BF16 input of this layer
  const int32_t* gather;
  const float* xscale;
  float* y;
  const float* residual;
};

struct ChPhase {
  ChLayer L[POLYQ_MAX_GROUP];
  int n_layers, items, recs, kind;
  float eps;
  int pad0;
  const float* xa;
  const float* xb;
  uint16_t* xout;
};

struct ChParams {
  const ChPhase* ph;
  const int* ranges;  // [n_phases][gridDim.x + 1] item boundaries
  int n_phases, batch;
  uint32_t magic;
  int* status;
  unsigned int* bar;    // [0] barrier arrivals, [1] CTAs done, [2] launches completed
  unsigned int* ready;  // [n_phases] records built, summed over launches
  uint8_t* rec;         // records of the current phase
};

// Consumer-side copy of one phase's tables.
struct ChShared {
  GvBlock blk[POLYQ_MAX_GROUP][POLYQ_MAX_BLOCKS];
  int n_blocks[POLYQ_MAX_GROUP], N[POLYQ_MAX_GROUP], K[POLYQ_MAX_GROUP];
  int item0[POLYQ_MAX_GROUP + 1], rec0[POLYQ_MAX_GROUP + 1];
  const __nv_bfloat16* x[POLYQ_MAX_GROUP];
  const int32_t* gather[POLYQ_MAX_GROUP];
  const float* xscale[POLYQ_MAX_GROUP];
  float* y[POLYQ_MAX_GROUP];
  int n_layers, kind, recs;
  float eps;
  const float* xa;
  const float* xb;
  uint16_t* xout;
};

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// The tensor maps live in global memory, written by a host copy: make the
// tensor-map proxy see the current contents (the same memory may have held
// another plan's maps in an earlier launch).
__device__ __forceinline__ void tmap_acquire(const CUtensorMap* m) {
  asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(m) : "memory");
}

__device__ void load_phase(const ChPhase* ph, ChShared* S) {
  const int t = threadIdx.x;
  const int nl = ph->n_layers;
  if (t < POLYQ_MAX_GROUP * POLYQ_MAX_BLOCKS) {
    const int l = t / POLYQ_MAX_BLOCKS, b = t % POLYQ_MAX_BLOCKS;
    if (l < nl) S->blk[l][b] = ph->L[l].blk[b];
  }
  if (t < POLYQ_MAX_GROUP && t < nl) {
    const ChLayer& L = ph->L[t];
    S->n_blocks[t] = L.n_blocks;
    S->N[t] = L.N;
    S->K[t] = L.K;
    S->item0[t] = L.item0;
    S->rec0[t] = L.rec0;
    S->x[t] = L.x;
    S->gather[t] = L.gather;
    S->xscale[t] = L.xscale;
    S->y[t] = L.y;
  }
  if (t == 32) {
    S->n_layers = nl;
    S->item0[nl] = ph->items;
    S->rec0[nl] = ph->recs;
    S->recs = ph->recs;
    S->kind = ph->kind;
    S->eps = ph->eps;
    S->xa = ph->xa;
    S->xb = ph->xb;
    S->xout = ph->xout;
  }
}

// Layer, block and block step of flat record f.
__device__ __forceinline__ void rec_where(const ChShared& S, int f, int* l, int* bi, int* j) {
  int q = 0;
  while (q + 1 < S.n_layers && f >= S.rec0[q + 1]) ++q;
  const int s = f - S.rec0[q];
  int b = 0;
  while (b + 1 < S.n_blocks[q] && s >= S.blk[q][b + 1].step0) ++b;
  *l = q;
  *bi = b;
  *j = s - S.blk[q][b].step0;
}

__device__ __forceinline__ XIn chain_xin(const ChShared& S, int l, int batch) {
  XIn in;
  in.x = S.x[l];
  in.xa = S.xa;
  in.xb = S.xb;
  in.xout = l == 0 ? S.xout : nullptr;  // layer 0's records cover every source element
  in.gather = S.gather[l];
  in.xscale = S.xscale[l];
  in.kind = S.kind;
  in.K = S.K[l];
  in.batch = batch;
  return in;
}

// One activation record of the phase (flat index f) into global memory.
template <int NB>
__device__ __noinline__ void build_record(const ChShared& S, int f, int batch, const uint32_t* p3,
                                          const float* s_rnorm, uint8_t* dst) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int l, bi, j;
  rec_where(S, f, &l, &bi, &j);
  const XIn in = chain_xin(S, l, batch);
  int src[2][2];
  float fac[2][2], ra[2][2], rb[2][2];
  rec_sources<NB>(in, S.blk[l][bi], j, warp, lane, p3, src, fac);
  rec_load<NB>(in, S.blk[l][bi], j, warp, lane, p3, src, ra, rb);
  rec_store<NB>(in, S.blk[l][bi], j, warp, lane, p3, src, fac, ra, rb, s_rnorm,
                reinterpret_cast<uint32_t*>(dst));
}

// Outputs of a phase start as the residual (or zero); grid-stride over all
// consumer threads of the launch.
__device__ void init_outputs(const ChPhase* ph, int batch) {
  const int nl = ph->n_layers;
  const int stride = gridDim.x * kConsumers;
  for (int l = 0; l < nl; ++l) {
    float* y = ph->L[l].y;
    const float* res = ph->L[l].residual;
    if (y == res) continue;
    const int total = batch * ph->L[l].N;
    for (int i = blockIdx.x * kConsumers + threadIdx.x; i < total; i += stride)
      y[i] = res ? __ldcg(res + i) : 0.f;
  }
}

template <int NB>
__global__ void __launch_bounds__(kThreads, kChCtasPerSm) gemv_chain(const __grid_constant__ ChParams P) {
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int RB = rec_bytes(NB);
  uint8_t* stages = smem;
  uint32_t* zeros = reinterpret_cast<uint32_t*>(smem + kStages * kStageBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(zeros + 64);
  __shared__ ChShared S;
  __shared__ uint32_t s_p3[16];
  __shared__ float s_rnorm[4];
  __shared__ float s_part[4][kWarps];
  __shared__ volatile int s_abort;
  __shared__ int s_ok;
  __shared__ unsigned s_epoch;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kStages);
  const int G = gridDim.x;

  if (threadIdx.x == 0) {
    s_abort = 0;
    s_epoch = ld_acquire_gpu(P.bar + 2);  // launches completed on this workspace
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kWarps);
    }
    mbar_fence_init();
  }
  if (threadIdx.x < 64) zeros[threadIdx.x] = 0u;
  if (threadIdx.x < 16) {
    const PairDef d = pair3(threadIdx.x);
    s_p3[threadIdx.x] = (uint32_t)d.lo | ((uint32_t)d.hi << 8) | ((uint32_t)(d.win + 16) << 16);
  }
  __syncthreads();

  if (warp == kWarps) {
    // ---------------- producer ----------------
    // Weights are issued as soon as a stage is free, across phase
    // boundaries; an item's activation record is issued once its phase's
    // records are all built (a counter per phase, summed over launches).
    if (lane != 0) return;
    const unsigned epoch = s_epoch;
    int kg = 0, kr = 0;           // items whose weights / records were issued
    int ready_phase = -1;         // phases whose records are known to be built
    const uint8_t* rsrc[kStages]; // record source of each pending item, by slot
    int rphase[kStages];
    auto wait_ready = [&](int p) -> bool {
      // the counter grows by recs per launch and wraps after 2^32 / recs
      // launches: compare by signed difference
      const unsigned target = (epoch + 1u) * (unsigned)P.ph[p].recs;
      uint32_t it = 0;
      while ((int)(target - ld_acquire_gpu(P.ready + p)) > 0) {
        if (++it > kGridWaitLimit || s_abort) return false;
        __nanosleep(32);
      }
      fence_proxy_async_global();  // the builders wrote through the generic proxy
      return true;
    };
    // issue the records of items kr..upto (blocking until their phases are built)
    auto issue_records = [&](int upto) -> bool {
      while (kr <= upto) {
        const int sl = kr % kStages;
        if (rphase[sl] > ready_phase) {
          if (!wait_ready(rphase[sl])) {
            if (!s_abort) atomicExch(P.status, kStatusTimeoutRecords);
            s_abort = 1;
            return false;
          }
          ready_phase = rphase[sl];
        }
        bulk_load(smem_u32(stages + sl * kStageBytes + kRecOff), rsrc[sl], RB, full0 + 8 * sl);
        ++kr;
      }
      return true;
    };
    bool go = true;
    for (int p = 0; p < P.n_phases && go; ++p) {
      const ChPhase* ph = P.ph + p;
      const int lo = __ldg(P.ranges + p * (G + 1) + blockIdx.x);
      const int hi = __ldg(P.ranges + p * (G + 1) + blockIdx.x + 1);
      if (lo >= hi) continue;
      const int nl = ph->n_layers;
      for (int q = 0; q < nl; ++q) {
        for (int b = 0; b < ph->L[q].n_blocks; ++b) tmap_acquire(&ph->L[q].tm_codes[b]);
        tmap_acquire(&ph->L[q].tm_meta);
      }
      // position of item lo: layer, tile, step (tile-major)
      int l = 0;
      while (l + 1 < nl && lo >= ph->L[l + 1].item0) ++l;
      int steps = ph->L[l].steps;
      int tile = (lo - ph->L[l].item0) / steps;
      int s = lo - ph->L[l].item0 - tile * steps;
      for (int it = lo; it < hi && go; ++it) {
        const int slot = kg % kStages;
        if (kg >= kStages) {
          // the consumers free this stage only after the item it holds, so
          // that item's record goes first
          if (!issue_records(kg - kStages)) {
            go = false;
            break;
          }
          const uint32_t bar = empty0 + 8 * slot, par = ((kg / kStages) - 1) & 1;
          bool ok = false;
          for (uint32_t w = 0; w < kWaitLimit && !s_abort; ++w)
            if (mbar_try_wait(bar, par)) {
              ok = true;
              break;
            }
          if (!ok) {
            if (!s_abort) atomicExch(P.status, kStatusTimeoutEmpty);
            s_abort = 1;
            go = false;
            break;
          }
        }
        const ChLayer& L = ph->L[l];
        int bi = 0;
        while (bi + 1 < L.n_blocks && s >= L.blk[bi + 1].step0) ++bi;
        const GvBlock B = L.blk[bi];
        const int j = s - B.step0;
        const bool flush = s == steps - 1 || it == hi - 1;
        int sb, nbx, pitch;
        switch (B.bits) {
          case 2: sb = step_bytes(2, NB); nbx = nbox_of(2, NB); pitch = box_pitch(2, NB); break;
          case 3: sb = step_bytes(3, NB); nbx = nbox_of(3, NB); pitch = box_pitch(3, NB); break;
          case 4: sb = step_bytes(4, NB); nbx = nbox_of(4, NB); pitch = box_pitch(4, NB); break;
          case 8: sb = step_bytes(8, NB); nbx = nbox_of(8, NB); pitch = box_pitch(8, NB); break;
          default: sb = step_bytes(16, NB); nbx = nbox_of(16, NB); pitch = box_pitch(16, NB); break;
        }
        uint8_t* st = stages + slot * kStageBytes;
        const uint32_t dst = smem_u32(st);
        const uint32_t bar = full0 + 8 * slot;
        {
          const int uvalid = min(B.units, B.n_ch - j * B.units);
          const int g0 = (B.grp_off + j * (B.units / 64)) & 3;
          uint4 d;
          d.x = (uint32_t)B.bits | ((uint32_t)flush << 8) | ((uint32_t)l << 16);
          d.y = (uint32_t)uvalid | ((uint32_t)g0 << 16);
          d.z = (uint32_t)tile;
          d.w = 0u;
          *reinterpret_cast<uint4*>(st + kDescOff) = d;
        }
        uint32_t bytes = nbx * pitch * kRows + RB;
        if (B.bits < 16) bytes += kMetaBytes;
        mbar_expect_tx(bar, bytes);
        for (int h = 0; h < nbx; ++h)
          tma_load_2d(dst + h * kRows * pitch, &L.tm_codes[bi], B.seg_off + j * sb + h * (sb / nbx),
                      tile * kRows, bar);
        if (B.bits < 16) {
          const int x0 = (B.grp_off + j * (B.units / 64)) & ~3;
          tma_load_2d(dst + kCodesBytes, &L.tm_meta, x0, tile * kRows, bar);
        }
        rsrc[slot] = P.rec + (size_t)(L.rec0 + s) * RB;
        rphase[slot] = p;
        ++kg;
        if (p <= ready_phase && !issue_records(kg - 1)) {
          go = false;
          break;
        }
        // next item
        if (++s == steps) {
          s = 0;
          if (++tile == L.tiles) {
            tile = 0;
            if (++l < nl) steps = ph->L[l].steps;
          }
        }
      }
    }
    if (go) issue_records(kg - 1);
    // After a give-up, records still missing are issued anyway (their
    // contents no longer matter) so that every issued stage completes; then
    // wait (bounded) for the copies in flight before leaving.
    for (; kr < kg; ++kr) {
      const int sl = kr % kStages;
      bulk_load(smem_u32(stages + sl * kStageBytes + kRecOff), rsrc[sl], RB, full0 + 8 * sl);
    }
    for (int k = max(0, kg - kStages); k < kg; ++k)
      mbar_wait(full0 + 8 * (k % kStages), (k / kStages) & 1);
    return;
  }

  // ---------------- consumers ----------------
  float acc[2] = {0.f, 0.f};  // this lane's row sums (see lane_batch)
  int slot = 0;
  uint32_t phase = 0;
  unsigned gen = 0;

  // Named-barrier discipline: every consumer warp passes the same sequence
  // of consumer_sync() calls whatever happens, so a wait that gives up never
  // strands a warp at a barrier; decisions that steer control flow are taken
  // by thread 0 and read by all after a consumer_sync().
  auto grid_sync = [&]() -> bool {
    consumer_sync();  // this CTA's atomic additions are issued
    if (threadIdx.x == 0) {
      bool ok = !s_abort;
      if (ok) {
        __threadfence();
        atomicAdd(P.bar, 1u);
        const unsigned target = (gen + 1) * (unsigned)G;
        uint32_t it = 0;
        while (ld_acquire_gpu(P.bar) < target) {
          if (++it > kGridWaitLimit) {
            ok = false;
            atomicExch(P.status, kStatusTimeoutGrid);
            s_abort = 1;
            break;
          }
          __nanosleep(32);
        }
        __threadfence();
      }
      s_ok = ok;
    }
    ++gen;
    consumer_sync();
    return s_ok;
  };

  init_outputs(P.ph, P.batch);
  bool alive = grid_sync();
  for (int p = 0; p < P.n_phases && alive; ++p) {
    const ChPhase* ph = P.ph + p;
    load_phase(ph, &S);
    consumer_sync();
    // this CTA's share of the phase's records (the inputs are complete)
    if (blockIdx.x < S.recs) {
      if (S.kind == POLYQ_X_RMSNORM) rms_rnorm(S.xa, S.K[0], P.batch, S.eps, s_part, s_rnorm);
      int built = 0;
      for (int f = blockIdx.x; f < S.recs; f += G, ++built)
        build_record<NB>(S, f, P.batch, s_p3, s_rnorm, P.rec + (size_t)f * RB);
      consumer_sync();
      if (threadIdx.x == 0) {
        __threadfence();
        atomicAdd(P.ready + p, (unsigned)built);
      }
    }
    if (p + 1 < P.n_phases) init_outputs(P.ph + p + 1, P.batch);
    const int lo = __ldg(P.ranges + p * (G + 1) + blockIdx.x);
    const int hi = __ldg(P.ranges + p * (G + 1) + blockIdx.x + 1);
    for (int it = lo; it < hi; ++it) {
      bool ok = false;
      for (uint32_t w = 0; w < kWaitLimit && !s_abort; ++w)
        if (mbar_try_wait(full0 + 8 * slot, phase)) {
          ok = true;
          break;
        }
      if (!ok && !s_abort) {
        if (lane == 0) atomicExch(P.status, kStatusTimeoutFull);
        s_abort = 1;
      }
      if (ok) {
        const uint8_t* stage = stages + slot * kStageBytes;
        const uint32_t* rec = reinterpret_cast<const uint32_t*>(stage + kRecOff);
        const uint4 desc = *reinterpret_cast<const uint4*>(stage + kDescOff);
        const int bits = (int)(desc.x & 0xFFu);
        const int uvalid = (int)(desc.y & 0xFFFFu), g0 = (int)(desc.y >> 16);
        switch (bits) {
          case 2: step_mma<NB, 2>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
          case 3: step_mma<NB, 3>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
          case 4: step_mma<NB, 4>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
          case 8: step_mma<NB, 8>(P.magic, P.batch, uvalid, g0, stage, stage, rec, zeros, warp, lane, acc); break;
          default: step_16<NB>(P.batch, uvalid, stage, rec, zeros, warp, lane, acc); break;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty0 + 8 * slot);
        if (desc.x & 0x100u) {
          // add this warp's 16 rows of the tile piece into y
          const int l = (int)(desc.x >> 16);
          flush_rows<NB>(acc, S.y[l], S.N[l], P.batch, (int)desc.z * kRows + warp * 16, lane);
        }
      }
      if (++slot == kStages) {
        slot = 0;
        phase ^= 1u;
      }
    }
    if (p + 1 < P.n_phases) alive = grid_sync();
  }
  // the last CTA to finish clears the barrier counters and counts the launch
  consumer_sync();
  if (threadIdx.x == 0 && !s_abort) {
    __threadfence();
    if (atomicAdd(P.bar + 1, 1u) == (unsigned)G - 1) {
      atomicExch(P.bar, 0u);
      atomicExch(P.bar + 1, 0u);
      atomicAdd(P.bar + 2, 1u);
    }
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
constexpr size_t kChSmemBytes = (size_t)kStages * kStageBytes + 64 * 4 + 2 * kStages * 8;

int nb_of_batch(int batch) { return batch == 1 ? 1 : batch == 2 ? 2 : 4; }

// Byte range [lo, hi) of a buffer, for the overlap rules.
struct Span {
  const char* lo;
  const char* hi;
};
bool overlap(const Span& a, const Span& b) {
  return a.lo && b.lo && a.lo < b.hi && b.lo < a.hi;
}
Span span(const void* p, size_t bytes) {
  const char* c = static_cast<const char*>(p);
  return Span{c, c ? c + bytes : nullptr};
}

}  // namespace

struct polyq_gemv_chain {
  int n_phases = 0, batch = 0, nb = 1, grid = 0;
  std::vector<ChPhase> ph;
  std::vector<int> ranges;
  size_t ranges_off = 0, plan_bytes = 0;
  size_t rec_off = 0, ws_bytes = 0;  // workspace: records region, total
  void* plan_dev = nullptr;
};

namespace {

int check_phase(const polyq_gemv_phase& P, int batch, int idx) {
  const char* who = "polyq_gemv_chain_create";
  if (P.n_layers < 1 || P.n_layers > POLYQ_MAX_GROUP)
    return polyq_set_error(POLYQ_EINVAL, "%s: phase %d has %d layers", who, idx, P.n_layers);
  const polyq_gemv_input& in = P.in;
  if (in.kind < POLYQ_X_BF16 || in.kind > POLYQ_X_SILU_MUL)
    return polyq_set_error(POLYQ_EINVAL, "%s: phase %d: unknown input kind %d", who, idx, in.kind);
  if ((in.kind == POLYQ_X_SILU_MUL) != (in.b != nullptr))
    return polyq_set_error(POLYQ_EINVAL, "%s: phase %d: b is the second input of "
                           "POLYQ_X_SILU_MUL only", who, idx);
  if (in.kind == POLYQ_X_RMSNORM && !(in.eps >= 0.f))
    return polyq_set_error(POLYQ_EINVAL, "%s: phase %d: eps must be >= 0", who, idx);
  for (int i = 0; i < P.n_layers; ++i) {
    int rc = polyq_check_dev_layer(P.layers[i], who);
    if (rc) return rc;
    if (P.layers[i]->K != P.layers[0]->K)
      return polyq_set_error(POLYQ_EINVAL, "%s: phase %d: layers sharing one input need the "
                             "same K", who, idx);
    const void* x = (in.kind == POLYQ_X_BF16 && P.xs[i]) ? P.xs[i] : in.a;
    if (!x || !P.ys[i])
      return polyq_set_error(POLYQ_EINVAL, "%s: phase %d: input or output %d is NULL", who, idx, i);
    if (P.residuals[i] && P.residuals[i] != P.ys[i]) {
      // a residual is read while y is written: distinct buffers only
      const size_t ob = (size_t)batch * P.layers[i]->N * 4;
      if (overlap(span(P.ys[i], ob), span(P.residuals[i], ob)))
        return polyq_set_error(POLYQ_EINVAL, "%s: phase %d: residual %d overlaps its output",
                               who, idx, i);
    }
  }
  (void)batch;
  return POLYQ_OK;
}

// What a phase reads (inputs and residuals) and writes (outputs, x_out).
void phase_spans(const polyq_gemv_phase& P, int batch, std::vector<Span>* reads,
                 std::vector<Span>* writes, std::vector<Span>* fresh_writes) {
  const int64_t K = P.layers[0]->K;
  const size_t in_elem = P.in.kind == POLYQ_X_BF16 ? 2 : 4;
  reads->push_back(span(P.in.a, (size_t)batch * K * in_elem));
  reads->push_back(span(P.in.b, (size_t)batch * K * 4));
  for (int i = 0; i < P.n_layers; ++i) {
    if (P.in.kind == POLYQ_X_BF16 && P.xs[i]) reads->push_back(span(P.xs[i], (size_t)batch * K * 2));
    const size_t ob = (size_t)batch * P.layers[i]->N * 4;
    writes->push_back(span(P.ys[i], ob));
    if (P.residuals[i] && P.residuals[i] != P.ys[i]) reads->push_back(span(P.residuals[i], ob));
    if (P.residuals[i] != P.ys[i]) fresh_writes->push_back(span(P.ys[i], ob));
  }
  if (P.in.x_out) writes->push_back(span(P.in.x_out, (size_t)batch * K * 2));
}

int fill_phase(const polyq_gemv_phase& P, int nb, ChPhase* C) {
  std::memset(static_cast<void*>(C), 0, sizeof *C);
  int items = 0, recs = 0;
  for (int i = 0; i < P.n_layers; ++i) {
    const polyq_dev_layer* D = P.layers[i];
    ChLayer& G = C->L[i];
    int s = 0;
    for (int b = 0; b < D->n_blocks; ++b) {
      const polyq_block& pb = D->blocks[b];
      GvBlock gb;
      gb.bits = pb.bits;
      gb.n_ch = pb.n_ch;
      gb.pos0 = pb.pos0;
      gb.seg_off = pb.seg_off;
      gb.grp_off = pb.grp_off;
      gb.units = step_units(pb.bits, nb);
      gb.step0 = s;
      gb.n_steps = (pb.n_ch + gb.units - 1) / gb.units;
      s += gb.n_steps;
      G.blk[b] = gb;
      const int bw = box_pitch(pb.bits, nb);
      int rc = polyq_tensor_map_2d(&G.tm_codes[b], D->packed, 1, (uint64_t)D->row_stride,
                                   (uint64_t)D->N, (uint64_t)D->row_stride, (uint32_t)bw, kRows);
      if (rc) return rc;
    }
    if (D->n_groups > 0) {
      int rc = polyq_tensor_map_2d(&G.tm_meta, D->meta, 4, (uint64_t)D->meta_stride,
                                   (uint64_t)D->N, (uint64_t)D->meta_stride * 4, kMetaBox, kRows);
      if (rc) return rc;
    }
    G.n_blocks = D->n_blocks;
    G.N = (int)D->N;
    G.K = (int)D->K;
    G.steps = s;
    G.tiles = (int)((D->N + kRows - 1) / kRows);
    G.item0 = items;
    G.rec0 = recs;
    G.x = (const __nv_bfloat16*)((P.in.kind == POLYQ_X_BF16 && P.xs[i]) ? P.xs[i] : P.in.a);
    G.gather = D->gather;
    G.xscale = D->xscale;
    G.y = P.ys[i];
    G.residual = P.residuals[i];
    items += G.tiles * s;
    recs += s;
  }
  C->n_layers = P.n_layers;
  C->items = items;
  C->recs = recs;
  C->kind = P.in.kind;
  C->eps = P.in.eps;
  C->xa = P.in.kind == POLYQ_X_BF16 ? nullptr : (const float*)P.in.a;
  C->xb = P.in.b;
  C->xout = P.in.x_out;
  return POLYQ_OK;
}

// Contiguous item ranges of equal modelled cost (bytes streamed plus a fixed
// per-item cost) for `grid` CTAs; items are (layer, tile, step) tile-major.
void split_phase(const ChPhase& C, int nb, int grid, int* out) {
  std::vector<long long> prefix(1, 0);  // cost of items [0, i)
  prefix.reserve((size_t)C.items + 1);
  for (int l = 0; l < C.n_layers; ++l) {
    const ChLayer& L = C.L[l];
    std::vector<long long> per;
    for (int b = 0; b < L.n_blocks; ++b) {
      const GvBlock& B = L.blk[b];
      const long long c = (long long)kRows * step_bytes(B.bits, nb) +
                          (B.bits < 16 ? kRows * 4LL * (B.units / 64) : 0) + kItemFixedCost;
      for (int j = 0; j < B.n_steps; ++j) per.push_back(c);
    }
    for (int t = 0; t < L.tiles; ++t)
      for (long long c : per) prefix.push_back(prefix.back() + c);
  }
  const long long total = prefix.back();
  int item = 0;
  for (int b = 0; b <= grid; ++b) {
    const long long goal = (long long)((__int128)total * b / grid);
    while (item < C.items && prefix[item + 1] <= goal) ++item;
    out[b] = item;
  }
  out[grid] = C.items;
}

template <int NB>
int launch_chain(const polyq_gemv_chain* ch, void* ws, cudaStream_t st) {
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (!attr_done[dev & 63]) {
    cudaError_t e = cudaFuncSetAttribute(gemv_chain<NB>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kChSmemBytes);
    if (e != cudaSuccess)
      return polyq_set_error(POLYQ_ECUDA, "polyq chain: smem attribute: %s", cudaGetErrorString(e));
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gemv_chain<NB>, kThreads,
                                                      kChSmemBytes);
    if (e != cudaSuccess || per_sm < kChCtasPerSm)
      return polyq_set_error(POLYQ_ECUDA, "polyq chain: %d CTAs per SM fit, %d needed (%s)",
                             per_sm, kChCtasPerSm, cudaGetErrorString(e));
    attr_done[dev & 63] = true;
  }
  ChParams P;
  P.ph = static_cast<const ChPhase*>(ch->plan_dev);
  P.ranges = reinterpret_cast<const int*>(static_cast<const char*>(ch->plan_dev) + ch->ranges_off);
  P.n_phases = ch->n_phases;
  P.batch = ch->batch;
  P.magic = kMagic;
  P.status = static_cast<int*>(ws);
  P.bar = reinterpret_cast<unsigned int*>(static_cast<char*>(ws) + kWsCounters);
  P.ready = reinterpret_cast<unsigned int*>(static_cast<char*>(ws) + kWsReady);
  P.rec = static_cast<uint8_t*>(ws) + ch->rec_off;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;
  at[0].val.cooperative = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3((unsigned)ch->grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kChSmemBytes;
  cudaError_t e = cudaLaunchKernelEx(&cfg, gemv_chain<NB>, P);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "polyq_linear_gemv_chain: launch: %s",
                           cudaGetErrorString(e));
  return POLYQ_OK;
}

}  // namespace

extern "C" int polyq_gemv_chain_create(const polyq_gemv_phase* phases, int n_phases, int batch,
                                       polyq_gemv_chain** out) {
  polyq_clear_error();
  const char* who = "polyq_gemv_chain_create";
  if (!out) return polyq_set_error(POLYQ_EINVAL, "%s: out is NULL", who);
  *out = nullptr;
  if (!phases || n_phases < 1 || n_phases > 65536)
    return polyq_set_error(POLYQ_EINVAL, "%s: need 1..65536 phases", who);
  if (batch < 1 || batch > 4)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "%s: batch %d not in 1..4", who, batch);
  for (int p = 0; p < n_phases; ++p) {
    int rc = check_phase(phases[p], batch, p);
    if (rc) return rc;
  }
  // overlap rules: inside a phase, and between consecutive phases
  for (int p = 0; p < n_phases; ++p) {
    std::vector<Span> rd, wr, fresh;
    phase_spans(phases[p], batch, &rd, &wr, &fresh);
    for (size_t i = 0; i < wr.size(); ++i) {
      for (const Span& r : rd)
        if (overlap(wr[i], r))
          return polyq_set_error(POLYQ_EINVAL, "%s: phase %d writes what it reads", who, p);
      for (size_t k = i + 1; k < wr.size(); ++k)
        if (overlap(wr[i], wr[k]))
          return polyq_set_error(POLYQ_EINVAL, "%s: phase %d has overlapping outputs", who, p);
    }
    if (p + 1 < n_phases) {
      std::vector<Span> rd2, wr2, fresh2;
      phase_spans(phases[p + 1], batch, &rd2, &wr2, &fresh2);
      for (const Span& f : fresh2) {
        for (const Span& r : rd)
          if (overlap(f, r))
            return polyq_set_error(POLYQ_EINVAL, "%s: phase %d output overlaps an input of "
                                   "phase %d", who, p + 1, p);
        for (const Span& w : wr)
          if (overlap(f, w))
            return polyq_set_error(POLYQ_EINVAL, "%s: phase %d output overlaps an output of "
                                   "phase %d", who, p + 1, p);
      }
    }
  }
  int sms = 0;
  int rc = polyq_sm_count(&sms);
  if (rc) return rc;
  polyq_gemv_chain* ch = new (std::nothrow) polyq_gemv_chain;
  if (!ch) return polyq_set_error(POLYQ_ENOMEM, "%s: out of host memory", who);
  try {
    ch->n_phases = n_phases;
    ch->batch = batch;
    ch->nb = nb_of_batch(batch);
    ch->grid = std::max(1, std::min(kChCtasPerSm * sms, kChMaxGrid));
    ch->ph.resize(n_phases);
    ch->ranges.assign((size_t)n_phases * (ch->grid + 1), 0);
    for (int p = 0; p < n_phases; ++p) {
      rc = fill_phase(phases[p], ch->nb, &ch->ph[p]);
      if (rc) {
        delete ch;
        return rc;
      }
      if (ch->ph[p].items > (1 << 30)) {
        delete ch;
        return polyq_set_error(POLYQ_EUNSUPPORTED, "%s: phase %d has too many items", who, p);
      }
      split_phase(ch->ph[p], ch->nb, ch->grid, ch->ranges.data() + (size_t)p * (ch->grid + 1));
    }
  } catch (const std::bad_alloc&) {
    delete ch;
    return polyq_set_error(POLYQ_ENOMEM, "%s: out of host memory", who);
  }
  ch->ranges_off = (size_t)n_phases * sizeof(ChPhase);
  ch->plan_bytes = ch->ranges_off + ch->ranges.size() * sizeof(int);
  int max_recs = 0;
  for (const ChPhase& c : ch->ph) max_recs = std::max(max_recs, c.recs);
  ch->rec_off = (kWsReady + 4 * (size_t)n_phases + 255) / 256 * 256;
  ch->ws_bytes = ch->rec_off + (size_t)max_recs * rec_bytes(ch->nb);
  *out = ch;
  return POLYQ_OK;
}

extern "C" int polyq_gemv_chain_workspace_bytes(const polyq_gemv_chain* ch, size_t* bytes) {
  polyq_clear_error();
  if (!ch || !bytes)
    return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_chain_workspace_bytes: NULL argument");
  *bytes = ch->ws_bytes;
  return POLYQ_OK;
}

extern "C" int polyq_gemv_chain_plan_bytes(const polyq_gemv_chain* ch, size_t* bytes) {
  polyq_clear_error();
  if (!ch || !bytes) return polyq_set_error(POLYQ_EINVAL, "polyq_gemv_chain_plan_bytes: NULL");
  *bytes = ch->plan_bytes;
  return POLYQ_OK;
}

extern "C" int polyq_gemv_chain_upload(polyq_gemv_chain* ch, void* plan_dev, size_t bytes,
                                       void* stream) {
  polyq_clear_error();
  const char* who = "polyq_gemv_chain_upload";
  if (!ch || !plan_dev) return polyq_set_error(POLYQ_EINVAL, "%s: NULL argument", who);
  if (bytes < ch->plan_bytes)
    return polyq_set_error(POLYQ_ENOMEM, "%s: plan needs %zu bytes, got %zu", who,
                           ch->plan_bytes, bytes);
  if ((uintptr_t)plan_dev % alignof(ChPhase))
    return polyq_set_error(POLYQ_EINVAL, "%s: plan memory must be %zu-byte aligned", who,
                           alignof(ChPhase));
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = cudaMemcpyAsync(plan_dev, ch->ph.data(), ch->ranges_off,
                                  cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(static_cast<char*>(plan_dev) + ch->ranges_off, ch->ranges.data(),
                        ch->ranges.size() * sizeof(int), cudaMemcpyHostToDevice, st);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "%s: copy: %s", who, cudaGetErrorString(e));
  // the host plan must outlive the asynchronous copies from pageable memory
  e = cudaStreamSynchronize(st);
  if (e != cudaSuccess)
    return polyq_set_error(POLYQ_ECUDA, "%s: %s", who, cudaGetErrorString(e));
  ch->plan_dev = plan_dev;
  return POLYQ_OK;
}

extern "C" int polyq_linear_gemv_chain(const polyq_gemv_chain* ch, void* workspace,
                                       size_t ws_bytes, void* stream) {
  polyq_clear_error();
  const char* who = "polyq_linear_gemv_chain";
  if (!ch) return polyq_set_error(POLYQ_EINVAL, "%s: chain is NULL", who);
  if (!ch->plan_dev) return polyq_set_error(POLYQ_EINVAL, "%s: plan not uploaded", who);
  if (!workspace || ws_bytes < ch->ws_bytes)
    return polyq_set_error(POLYQ_ENOMEM, "%s: workspace needs %zu bytes, got %zu", who,
                           ch->ws_bytes, ws_bytes);
  if ((uintptr_t)workspace % 256)
    return polyq_set_error(POLYQ_EINVAL, "%s: workspace must be 256-byte aligned", who);
  int dev_sms = 0;
  int rc = polyq_sm_count(&dev_sms);
  if (rc) return rc;
  if (std::max(1, std::min(kChCtasPerSm * dev_sms, kChMaxGrid)) != ch->grid)
    return polyq_set_error(POLYQ_EINVAL, "%s: chain was built for another device", who);
  switch (ch->nb) {
    case 1: return launch_chain<1>(ch, workspace, (cudaStream_t)stream);
    case 2: return launch_chain<2>(ch, workspace, (cudaStream_t)stream);
    default: return launch_chain<4>(ch, workspace, (cudaStream_t)stream);
  }
}

extern "C" void polyq_gemv_chain_free(polyq_gemv_chain* ch) { delete ch; }
