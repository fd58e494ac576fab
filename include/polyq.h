/*
 * polyq.h - C ABI of the PolyQ mixed-bit linear layer for GB300 (sm_103a).
 *
 * PolyQ (arXiv 2607.14618) gives every input channel of a linear layer
 * y = x W^T a width from {2,3,4,8,16} under a fractional average budget B
 * (Section 3), permutes the channels into bit-homogeneous blocks (Section 4.1
 * and 4.2) and folds consumer permutations into producer output rows
 * (Section 4.3).  This library packs a layer on the host and runs the layer
 * on the GPU.
 *
 * Conventions for every call:
 *   - Return value: 0 (POLYQ_OK) on success, a negative POLYQ_E* code
 *     otherwise; polyq_last_error() then returns a message (thread-local,
 *     valid until the next call on the same thread).
 *   - The caller owns every buffer passed in.  Host buffers are read during
 *     the call only.  Device buffers must stay valid until the work queued on
 *     `stream` has finished.
 *   - GPU entry points never allocate device memory and never synchronise:
 *     they validate arguments on the host, then enqueue kernels on `stream`
 *     (a cudaStream_t passed as void*; NULL = legacy default stream) and
 *     return.  Launch errors are reported as POLYQ_ECUDA.
 *   - Device pointers must be 16-byte aligned unless stated otherwise.
 *
 * Packed format of one layer (host and device identical):
 *   widths   bits[K]        (original channel order)
 *   perm     int32 perm[K]: clustered position p holds original channel
 *            perm[p]; blocks in ascending width, channels ascending in a
 *            block (Section 4.1: only P_W W is materialised).
 *   blocks   at most 5, one per width present, ascending.
 *   packed   uint8 [N][row_stride]: per row the concatenation of one segment
 *            per block.  A b<16 segment is an LSB-first bitstream (code p of
 *            the block at bits [p*b, p*b+b), little-endian bytes); a 16-bit
 *            segment holds little-endian fp16 weights.  Segments are padded
 *            with zeros to a multiple of 16 bytes.
 *   meta     uint32 [N][n_groups]: per row and per 64-position group of a
 *            b<16 block (groups ordered by block, then position; the last
 *            group of a block may be shorter) the fp16 scale in bits 0..15
 *            and the fp16 zero point (an integer) in bits 16..31.
 *   Dequantised weight: w' = (q - zero) * scale for b<16; the fp16 value for
 *   b=16.  Quantiser: lo/hi = min/max of the group, scale =
 *   fp16_rn((hi-lo)/(2^b-1)) (if 0: fp16_rn(max(|lo|,|hi|,2^-14))),
 *   zero = clamp(rint(-lo/scale), 0, 2^b-1), q = clamp(rint(w/scale)+zero).
 */
#ifndef POLYQ_H
#define POLYQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define POLYQ_OK 0
#define POLYQ_EINVAL (-1)       /* bad argument, shape, alignment, permutation */
#define POLYQ_ENOMEM (-2)       /* host allocation failed / workspace too small */
#define POLYQ_ECUDA (-3)        /* a CUDA runtime call or launch failed */
#define POLYQ_EUNSUPPORTED (-4) /* option or size this build does not handle */
#define POLYQ_ETIMEOUT (-5)     /* a bounded device-side wait gave up */

#define POLYQ_MAX_BLOCKS 5
#define POLYQ_GROUP 64
#define POLYQ_MAX_GROUP 8 /* layers per GEMV group call or chain phase */

#define POLYQ_ALLOC_WATERFILL 0 /* Section 3.2 max-heap waterfilling (default) */
#define POLYQ_ALLOC_LADDER 1    /* descending saliency, each channel climbs */

/* Section 3.1 error proxy E_b[k] that drives the allocation. */
#define POLYQ_PROXY_SALIENCY 0 /* (a_k * ||W[:,k]||_2 / (2^b - 1))^2, E_16 = 0 */
#define POLYQ_PROXY_QUANT 1    /* ||Q_b(W)[:,k] - W[:,k]||^2 * E[x_k^2], E_16 = 0:
                                  the whole layer quantised at width b with groups
                                  of 64 consecutive original channels; the sum
                                  over rows in row order, fp64 */

/* Default channel quanta of the Section 3.3 quanta matching, widths
 * 2,3,4,8,16: one quantum of each width fills a whole number of 16-byte
 * chunks, so blocks of these sizes need no segment padding. */
#define POLYQ_GPU_QUANTA {64, 128, 32, 16, 8}

/* Options of polyq_pack.  Zero-initialise, then set what you need;
 * polyq_pack_opts_default() gives the defaults. */
typedef struct {
  int32_t group_size;        /* must be 64 */
  uint32_t palette_mask;     /* bit b set: width b allowed (b in 2,3,4,8,16);
                                0 means all five */
  int32_t alloc_rule;        /* POLYQ_ALLOC_WATERFILL or POLYQ_ALLOC_LADDER */
  int32_t snap_quanta;       /* 1: Section 3.3 quanta matching (below) */
  int32_t n_threads;         /* host threads, 0 = hardware concurrency */
  const uint8_t* forced_bits;/* optional [K] width map; skips allocation
                                (and then snap_quanta must be 0) */
  int32_t proxy;             /* POLYQ_PROXY_SALIENCY (default) or
                                POLYQ_PROXY_QUANT; POLYQ_ALLOC_LADDER needs
                                the saliency proxy */
  int32_t act_scaling;       /* 1: Section 3.4 bit-specific activation-aware
                                scaling (below) */
  int32_t quanta[5];         /* channels per quantum for widths 2,3,4,8,16
                                (each > 0), or all 0 for POLYQ_GPU_QUANTA */
  const float* act_sqmean;   /* [K] E[x_k^2] for POLYQ_PROXY_QUANT and the
                                scaling search; NULL = act_absmean[k]^2 */
} polyq_pack_opts;
/* Quanta matching (snap_quanta = 1), Section 3.3, after the allocation:
 *  1. target counts: for each palette width b the candidates are the
 *     multiples q_b*(floor(c_b/q_b)+d), d in {-1,0,1,2}, inside [0,K]; of the
 *     combinations summing to K the one with the smallest
 *     |sum b*count - round(B*K)| is taken, then the one closest to the
 *     allocation's counts (sum of |differences|), then the lexicographically
 *     smallest count vector (widths ascending).  If no combination sums to K,
 *     the narrowest width takes K minus the others' counts.
 *  2. reassignment between neighbouring widths: with f_i the net number of
 *     channels that must cross from widths <= w_i to widths > w_i, upward
 *     crossings are made from the lowest boundary up, each promoting the
 *     channels of width w_i with the largest gain per bit
 *     (E_{w_i} - E_{w_i+1}) / (w_{i+1} - w_i) (ties: lower channel first),
 *     then downward crossings from the top boundary down, each demoting the
 *     channels of width w_{i+1} with the smallest gain (ties: higher channel
 *     first).
 * Activation-aware scaling (act_scaling = 1), Section 3.4, on the final map:
 * m_k = a_k / mean(a) (a = act_absmean, mean summed in channel order); for
 * each width b present the exponent alpha_b in {0, 0.1, ..., 1} (j/10) that
 * minimises the mean over the block's channels of
 * ||Q_b(W/t)[:,k]*t_k - W[:,k]||^2 * E[x_k^2] with t_k = fp32_rn(m_k^-alpha_b),
 * evaluated with the block's own groups (ties: the smaller alpha; an alpha
 * giving a non-finite or non-positive t_k or |W/t| > 65504 is skipped; for
 * b = 16 alpha is 0).  The block is then packed from W/t (one fp64 division
 * per weight) and the layer carries the activation factor t at each
 * clustered position (polyq_layer_xscale): the GEMV and GEMM multiply the
 * gathered activation by it, so the layer still computes y = x W'^T with
 * W' = Q(W/t) * t. */

/* One bit-homogeneous block (Section 4.2). */
typedef struct {
  int32_t bits;      /* 2, 3, 4, 8 or 16 */
  int32_t n_ch;      /* channels in the block (K_b) */
  int32_t pos0;      /* first clustered position */
  int32_t seg_off;   /* byte offset of the block's segment inside a row */
  int32_t seg_bytes; /* segment bytes per row (multiple of 16) */
  int32_t grp_off;   /* first meta group of the block */
  int32_t n_grp;     /* ceil(n_ch/64) for b<16, 0 for b=16 */
} polyq_block;

typedef struct {
  int64_t N, K;          /* out x in */
  int64_t row_stride;    /* bytes per packed row */
  int64_t n_groups;      /* meta entries per row */
  int32_t n_blocks;
  polyq_block blocks[POLYQ_MAX_BLOCKS];
  double budget;         /* requested B */
  double b_real;         /* realised mean width (Section 3.3, B_real) */
  int64_t packed_bytes;  /* N * row_stride */
  int64_t meta_bytes;    /* N * n_groups * 4 */
  int64_t meta_stride;   /* device meta row stride in entries: n_groups
                            rounded up to a multiple of 4 (16-byte rows) */
  int64_t pad_bytes;     /* segment padding bytes in one packed row */
  double alpha[5];       /* Section 3.4 exponent of widths 2,3,4,8,16; -1 where
                            the width is absent or the layer is not scaled */
  int32_t has_xscale;    /* 1 when the layer carries activation factors */
} polyq_info;

/* A packed layer resident on the device.  Filled by polyq_dev_layer_fill()
 * (or by hand).  The library only reads it. */
typedef struct {
  const uint8_t* packed;  /* device [N][row_stride], 16-byte aligned */
  const uint32_t* meta;   /* device [N][meta_stride], 16-byte aligned; entries
                             past n_groups in a row are ignored */
  const int32_t* gather;  /* device [K]: xs[p] = x[gather[p]]; NULL = identity
                             (a merged edge, Section 4.3) */
  int64_t N, K, row_stride, n_groups;
  int64_t meta_stride;    /* entries per meta row, multiple of 4, >= n_groups */
  int32_t n_blocks;
  polyq_block blocks[POLYQ_MAX_BLOCKS];
  const float* xscale;    /* device fp32 [K], 16-byte aligned: Section 3.4
                             activation factor at each clustered position,
                             xs[p] = x[gather[p]] * xscale[p]; NULL = none
                             (polyq_dev_layer_fill leaves it NULL) */
} polyq_dev_layer;

typedef struct polyq_layer polyq_layer; /* opaque host-side packed layer */

const char* polyq_last_error(void);
void polyq_pack_opts_default(polyq_pack_opts* opts);

/* Allocate widths, cluster and pack one layer (Sections 3.1 to 3.4, 4.1,
 * 4.2).
 * W: host fp32 [N][K] row-major (out x in), finite, |W| <= 65504.
 * act_absmean: host fp32 [K], per-input-channel activation magnitude: the
 * saliency a_k * ||W[:,k]||_2 of the saliency proxy, the default E[x_k^2]
 * (its square) and the metric m of the Section 3.4 scaling.  Needed unless
 * forced_bits is given without act_scaling.
 * budget_bits: average width B in [2, 16] (Section 3.2).
 * Greedy waterfilling: all channels start at the narrowest palette width,
 * Delta = round(B*K) - b_min*K, upgrades popped from a max-heap by gain per
 * extra bit (E_b - E_b')/(b' - b) of the chosen proxy (ties: lower channel
 * first); a step that does not fit is dropped.  Then, as the options ask,
 * quanta matching and activation-aware scaling (see polyq_pack_opts).
 * On success *out owns a new layer (free with polyq_free). */
int polyq_pack(const float* W, int64_t N, int64_t K, const float* act_absmean,
               double budget_bits, const polyq_pack_opts* opts,
               polyq_layer** out);

void polyq_free(polyq_layer* layer);

/* Shape, blocks and byte counts of a packed layer. */
int polyq_layer_info(const polyq_layer* layer, polyq_info* out);

/* Copy the packed layer into caller buffers (each may be NULL to skip):
 * packed [N*row_stride] bytes, meta [N*meta_stride] uint32 (rows padded
 * with zero entries; meta_stride >= n_groups, use n_groups for the compact
 * host format or polyq_info.meta_stride for the device layout), perm [K]
 * int32, bits [K] uint8 (original channel order), out_perm [N] int32 (the
 * layer emits output i = y_original[out_perm[i]]). */
int polyq_layer_export(const polyq_layer* layer, uint8_t* packed,
                       uint32_t* meta, int64_t meta_stride, int32_t* perm,
                       uint8_t* bits, int32_t* out_perm);

/* Section 3.4 activation factors of a scaled layer (act_scaling = 1):
 * xscale [K] floats, xscale[p] = t at clustered position p (all 1.0 for a
 * layer packed without scaling).  Upload them and set
 * polyq_dev_layer.xscale; a scaled layer gives wrong results without them. */
int polyq_layer_xscale(const polyq_layer* layer, float* xscale);

/* Section 4.3 merge, producer side: permute whole output rows (packed bytes
 * and meta) so that afterwards the layer emits
 * new_output[i] = old_output[row_perm[i]].  row_perm: host int32 [N], a
 * permutation.  Passing a consumer's perm makes the producer emit in the
 * consumer's clustered basis, so the consumer's gather becomes identity. */
int polyq_layer_permute_rows(polyq_layer* layer, const int32_t* row_perm);

/* Section 4.3 merge rule, index side: gather_out[p] =
 * producer_basis^-1[consumer_perm[p]] where the producer emits
 * emitted[i] = y[producer_basis[i]].  All arrays host int32 [n]; both inputs
 * must be permutations.  The consumer then reads xs[p] = emitted[gather[p]]. */
int polyq_permute_merge(const int32_t* producer_basis,
                        const int32_t* consumer_perm, int64_t n,
                        int32_t* gather_out);

/* Section 4.4 graph-based permutation planning.  The model is a static DAG
 * whose edges are activations and whose nodes are: */
#define POLYQ_NODE_SOURCE_FIXED 0 /* no inputs; emits its output in natural order */
#define POLYQ_NODE_SOURCE_FREE 1  /* no inputs; emits in any order at no cost
                                     (e.g. an embedding table with permuted columns) */
#define POLYQ_NODE_LINEAR 2       /* in[0] = x; reads x in any order through its
                                     gather and emits any order by permuting its
                                     output rows; `perm` = id of its clustering
                                     permutation in the perms table */
#define POLYQ_NODE_ELEMENTWISE 3  /* 1..3 inputs and the output share one order
                                     (norms, activations, products, residual adds) */
#define POLYQ_NODE_BOUNDARY 4     /* inputs read in natural order; the output, if
                                     any, is natural (graph outputs, rotary q/k) */
#define POLYQ_NODE_ATTENTION 5    /* in = q, k, v: q and k natural; the output keeps
                                     v's order when both have the same width (the
                                     kernel maps channels to heads through it),
                                     otherwise v is read and the output written in
                                     natural order */

typedef struct {
  int32_t kind;   /* POLYQ_NODE_* */
  int32_t n_in;   /* inputs used in `in` (0..3) */
  int32_t in[3];  /* input edge ids */
  int32_t out;    /* output edge id, or -1 */
  int32_t perm;   /* POLYQ_NODE_LINEAR: permutation id; otherwise -1 */
} polyq_plan_node;

/* Assign a channel order ("basis") to every edge so that the explicit
 * activation shuffles the graph needs cost the least modelled traffic
 * (Section 4.4; the traffic model is Section 5.4's A16 read + write, 4 bytes
 * per channel per shuffle).  Edges joined by elementwise nodes (and by an
 * attention node that keeps v's order) form regions that share one order;
 * each region takes, among the natural order and the permutations of the
 * linears reading it, the one with the smallest cost: one shuffle per
 * distinct (edge, order wanted by a consumer) that differs from the region's
 * order, shared by every consumer of that edge wanting that order, plus one
 * per fixed-order producer that differs.  Ties go to the natural order, then
 * to the lowest permutation id.  Permutations with equal contents count as
 * one order, and an identity permutation as the natural order.
 *   nodes [n_nodes], edge_dims [n_edges] (channels of each edge, >= 1).
 *   perms [n_perms]: host int32 arrays, perms[i] of length perm_lens[i] (a
 *   permutation; a linear's permutation must be as long as its input edge).
 *   labels [n_edges] (out): -1 = natural order, else the id of the
 *   permutation p (the smallest id with p's contents): the edge carries
 *   emitted[i] = natural[p[i]].
 *   bytes_per_token (out, may be NULL): the plan's modelled traffic.
 * A linear then reads its input through polyq_permute_merge(label of its
 * input edge, its permutation) (identity when equal) and has its rows
 * permuted to its output edge's label (polyq_layer_permute_rows). */
int polyq_plan_graph(const polyq_plan_node* nodes, int32_t n_nodes, const int64_t* edge_dims,
                     int32_t n_edges, const int32_t* const* perms, const int64_t* perm_lens,
                     int32_t n_perms, int32_t* labels, int64_t* bytes_per_token);

/* Fill a device-layer descriptor from a host layer and the device copies of
 * its packed bytes and meta (uploaded by the caller from polyq_layer_export
 * with meta_stride = polyq_info.meta_stride) and an optional device gather
 * vector (NULL = identity). */
int polyq_dev_layer_fill(const polyq_layer* layer, const uint8_t* packed_dev,
                         const uint32_t* meta_dev, const int32_t* gather_dev,
                         polyq_dev_layer* out);

/* Device scratch bytes polyq_linear_gemv needs for this layer and batch on
 * the current device (it grows with N and with the device's SM count). */
int polyq_gemv_workspace_bytes(const polyq_dev_layer* layer, int batch,
                               size_t* bytes);

/* Decode GEMV (Section 4.1 factorisation; Section 4.2 blocks in one launch):
 *   y[b][n] = residual[b][n] + sum_p x[b][gather[p]] * W'[n][p]
 * x: device bf16 [batch][K] (the activation in its producer's basis), any
 * finite values.  The kernel multiplies fp16 copies of the gathered x with the
 * decoded codes and accumulates in fp32.  Before the fp16 rounding each
 * 64-channel group of a 2/3/4/8-bit block (each step of 128 channels of a
 * 16-bit block) and batch row is scaled by the power of two that brings its
 * largest |x| into [2^14, 2^15); its result is scaled back in fp32.  So the
 * copies are exact whatever the activations' absolute scale, except for
 * values more than about 2^20 below their group's largest, which lose low
 * bits as fp16 subnormals (each by at most 2^-31 of that largest value).  batch in 1..4; y: device fp32 [batch][N];
 * residual: device fp32 [batch][N] or NULL (y may alias residual; y must not
 * overlap x or the workspace).  y is
 * first set to the residual (or zero), then each of the few pieces a row's
 * sum is split into is added with an fp32 atomic addition, so the last bits
 * of y may differ from run to run.  workspace: device scratch of at least
 * polyq_gemv_workspace_bytes(), 256-byte aligned, zero-filled before its
 * first use; its first 4 bytes are a status word that stays zero unless a
 * bounded device wait gave up (then zero it again).  A workspace may serve
 * consecutive calls on one stream but not calls that run at the same time.
 * Two kernel launches (activation pre-pass, streaming kernel). */
int polyq_linear_gemv(const polyq_dev_layer* layer, const void* x, int batch,
                      float* y, const float* residual, void* workspace,
                      size_t workspace_bytes, void* stream);

/* Scratch, in bytes, compiled into the library for polyq_linear_gemv_noalloc
 * (1 MiB).  A call needs 256 bytes plus one activation record per step of K
 * (1184 bytes per 512 channels at batch 1, 1376 bytes per 128 channels at
 * batch 4), so every layer with K <= 65536 fits at any batch and any mix of
 * widths; N does not matter (see polyq_gemv_workspace_bytes). */
#define POLYQ_NOALLOC_SCRATCH_BYTES (1u << 20)

/* polyq_linear_gemv without a workspace argument: it allocates no device
 * memory and takes none from the caller.  The paper has no counterpart; this
 * is for callers that cannot allocate, such as a plugin living inside a host
 * program that owns all device memory through its own pool and hands out no
 * allocation hook, or a latency-bound loop that may not take the device-wide
 * synchronisation that cudaMalloc and cudaFree can cause.
 *
 * The scratch is one fixed array of POLYQ_NOALLOC_SCRATCH_BYTES compiled into
 * this library; each device that loads the library keeps its copy until the
 * process exits.  The first call on a device, with that device current, looks
 * up the array's device address once (cudaGetSymbolAddress); make that first
 * call before any stream capture on that device.  Every call on a device uses
 * the same array, so calls whose kernels may overlap on the GPU (different
 * streams, or different host threads without ordering) race and corrupt each
 * other's results; serialise them, e.g. on one stream.  The call's first
 * kernel zeroes the scratch's status word once the previous kernel on the
 * stream has finished, and writes every record before the second kernel reads
 * it, so nothing left by an earlier call leaks into a later one.  A bounded
 * device wait that gives up sets the status word and leaves y incomplete:
 * read it with polyq_noalloc_status after the call and before the next
 * no-allocation call on the same device.
 * Arguments and results are those of polyq_linear_gemv.  Returns
 * POLYQ_ENOMEM, touching nothing, when the layer and batch need more than
 * POLYQ_NOALLOC_SCRATCH_BYTES (see polyq_gemv_workspace_bytes). */
int polyq_linear_gemv_noalloc(const polyq_dev_layer* layer, const void* x, int batch,
                              float* y, const float* residual, void* stream);

/* Status word of the current device's no-allocation scratch after the work
 * queued on `stream` (a 4-byte copy to the host and a wait for the stream; no
 * allocation): the status of the last polyq_linear_gemv_noalloc call on this
 * device, decoded as polyq_workspace_status does (POLYQ_ETIMEOUT when a
 * bounded device wait gave up, with *status naming the wait).  The paper has
 * no counterpart. */
int polyq_noalloc_status(int* status, void* stream);

/* Device scratch bytes polyq_linear_gemv_group needs for these layers
 * (same rules as polyq_gemv_workspace_bytes). */
int polyq_gemv_group_workspace_bytes(const polyq_dev_layer* const* layers,
                                     int n, int batch, size_t* bytes);

/* Several independent decode GEMVs (the Section 4.1 product of each layer)
 * in one pair of launches, e.g. q/k/v or gate/up of a decoder layer, which
 * read the same activation.  layers[i], xs[i], ys[i], residuals[i] (the
 * array itself and each entry may be NULL) have the meaning they have in
 * polyq_linear_gemv; 1 <= n <= POLYQ_MAX_GROUP; all layers share `batch`
 * and one workspace of polyq_gemv_group_workspace_bytes().  Outputs must not
 * overlap each other or any input. */
int polyq_linear_gemv_group(const polyq_dev_layer* const* layers, int n,
                            const void* const* xs, int batch, float* const* ys,
                            const float* const* residuals, void* workspace,
                            size_t workspace_bytes, void* stream);

/* Activation input of polyq_linear_gemv_input: the glue of a decoder layer
 * (the residual stream's RMSNorm, SiLU(gate) * up, or a plain rounding to
 * bf16) fused into the GEMV's record pre-pass.  These are elementwise up to
 * a per-row scale, so they commute with the channel permutations
 * (Section 4.3) and run on the gathered values.  Every kind produces the bf16
 * activation x[b][k] that polyq_linear_gemv would take:
 *   POLYQ_X_BF16      x = a                      a: bf16 [batch][K]
 *   POLYQ_X_F32       x = bf16_rn(a)             a: fp32 [batch][K]
 *   POLYQ_X_RMSNORM   x = bf16_rn(a[b][k] / sqrt(mean_k(a[b][k]^2) + eps))
 *                                                a: fp32 [batch][K], unit gain
 *   POLYQ_X_SILU_MUL  x = bf16_rn(a / (1 + exp(-a)) * b)
 *                                                a, b: fp32 [batch][K]
 * bf16_rn rounds the fp32 result to nearest even.  x_out (optional, device
 * bf16 [batch][K]) receives x as computed, in source order. */
#define POLYQ_X_BF16 0
#define POLYQ_X_F32 1
#define POLYQ_X_RMSNORM 2
#define POLYQ_X_SILU_MUL 3
typedef struct {
  int32_t kind;      /* POLYQ_X_* */
  float eps;         /* POLYQ_X_RMSNORM only */
  const void* a;     /* device input, see kind */
  const float* b;    /* device fp32 [batch][K] for POLYQ_X_SILU_MUL, else NULL */
  uint16_t* x_out;   /* device bf16 [batch][K] or NULL */
} polyq_gemv_input;

/* polyq_linear_gemv_group with every layer reading the one input `in`
 * (all layers must have the same K).  Workspace, outputs and residuals as
 * for polyq_linear_gemv_group. */
int polyq_linear_gemv_input(const polyq_dev_layer* const* layers, int n,
                            const polyq_gemv_input* in, int batch, float* const* ys,
                            const float* const* residuals, void* workspace,
                            size_t workspace_bytes, void* stream);

/* ---- chained decode GEMVs in one persistent launch ----
 * A decoder's decode step is a chain of dependent GEMV phases (q/k/v, o,
 * gate/up, down, then the next layer's q/k/v, ...), each the product of
 * Section 4.1 for one to POLYQ_MAX_GROUP layers that share an input.  A chain runs all
 * of its phases in one launch: one CTA per resident slot (three per SM)
 * streams the packed weights of every phase through its TMA ring without
 * stopping at phase boundaries.  Between phases the consumer warps of all
 * CTAs meet at a grid-wide barrier (phase p+1 reads what phase p wrote),
 * then build the phase's activation records in the workspace, one per CTA.
 * Work items of a phase are (layer, 64-row tile, step) in tile-major order,
 * split into contiguous ranges of equal modelled cost; each tile piece adds
 * its rows into y with fp32 atomics (the order of those additions varies
 * from run to run).  Every device-side wait is bounded; on a timeout the
 * kernel records a status and returns. */
typedef struct polyq_gemv_chain polyq_gemv_chain; /* opaque, host-owned */

typedef struct {
  int32_t n_layers;                              /* 1..POLYQ_MAX_GROUP */
  const polyq_dev_layer* layers[POLYQ_MAX_GROUP];
  polyq_gemv_input in;    /* the phase's input and its transform (as for
                             polyq_linear_gemv_input); with POLYQ_X_BF16 a
                             non-NULL xs[i] overrides in.a for layer i */
  const void* xs[POLYQ_MAX_GROUP];
  float* ys[POLYQ_MAX_GROUP];                    /* fp32 [batch][N_i] */
  const float* residuals[POLYQ_MAX_GROUP];       /* NULL = none; may equal ys[i] */
} polyq_gemv_phase;


/* Build a chain of n_phases phases (1..65536) at one batch size (1..4).
 * The phase descriptors and the layer descriptors are copied (device memory
 * they point to must stay valid while the chain is used).  Rules, checked
 * here (POLYQ_EINVAL):
 *   - every layer of a phase has the phase input's width K;
 *   - a phase's outputs do not overlap its inputs (a residual may be the
 *     output itself: y += W'x in place);
 *   - the outputs of phase p+1 other than in-place ones overlap nothing that
 *     phase p reads or writes (they are initialised while phase p runs).
 * *out owns a host plan; upload it to device memory with
 * polyq_gemv_chain_upload before launching. */
int polyq_gemv_chain_create(const polyq_gemv_phase* phases, int n_phases, int batch,
                            polyq_gemv_chain** out);

/* Bytes of device memory the chain's plan needs (tensor maps, block tables
 * and per-CTA work ranges for the current device). */
/* Bytes of the workspace a launch of the chain needs: a status word, the
 * grid-barrier and launch counters, one record-ready counter per phase and
 * the activation records of the largest phase. */
int polyq_gemv_chain_workspace_bytes(const polyq_gemv_chain* chain, size_t* bytes);

int polyq_gemv_chain_plan_bytes(const polyq_gemv_chain* chain, size_t* bytes);

/* Copy the plan into plan_dev (device memory of at least
 * polyq_gemv_chain_plan_bytes, owned by the caller) with a
 * copy on `stream` (the call waits for it); the chain then launches from
 * plan_dev.  plan_dev must be 128-byte aligned. */
int polyq_gemv_chain_upload(polyq_gemv_chain* chain, void* plan_dev, size_t bytes,
                            void* stream);

/* Run every phase of the chain, in order, in one cooperative launch on
 * `stream`.  workspace: device, 256-byte aligned, at least
 * polyq_gemv_chain_workspace_bytes, zero-filled before first use and then
 * kept for this chain (its counters carry over from launch to launch); one
 * workspace serves consecutive launches on one stream but not launches that
 * run at the same time.  Its first 4 bytes are a status word that stays zero
 * unless a bounded wait gave up (then zero the whole workspace again).
 * Launch errors (including a device that cannot hold every CTA at once) are
 * POLYQ_ECUDA. */
int polyq_linear_gemv_chain(const polyq_gemv_chain* chain, void* workspace,
                            size_t workspace_bytes, void* stream);

void polyq_gemv_chain_free(polyq_gemv_chain* chain);

/* Read the status word of a GEMV, GEMM or chain workspace (its first 4 bytes)
 * after the work queued on `stream`: a copy to the host and a wait for the
 * stream.  *status = 0 and POLYQ_OK when no bounded device wait gave up;
 * otherwise *status names the wait (1 a consumer's wait for a stage's data,
 * 2 a producer's wait for a free stage, 3 a chained launch's grid barrier,
 * 4 a chained launch's wait for a phase's records) and the call returns
 * POLYQ_ETIMEOUT.  The kernels that gave up returned normally, so the
 * context stays usable; zero the workspace before using it again.  The GEMM
 * workspace keeps its status word in its last 256 bytes: pass that address
 * (workspace + polyq_gemm_workspace_bytes() - 256). */
int polyq_workspace_status(const void* workspace, int* status, void* stream);

/* Device scratch bytes polyq_linear_gemm needs for this layer and M. */
int polyq_gemm_workspace_bytes(const polyq_dev_layer* layer, int64_t M,
                               size_t* bytes);

/* Prefill GEMM (the same product for M tokens, Section 5.5 prefill):
 *   Y[m][n] = sum_p X[m][gather[p]] * W'[n][p]
 * X: device bf16 [M][K], any finite values; Y: device fp32 [M][N], 16-byte
 * aligned (else POLYQ_EINVAL); workspace as for the GEMV (its status word in
 * its last 256 bytes).  Weights are dequantised to fp16 tiles in shared
 * memory and multiplied on the tcgen05 tensor cores with fp32 accumulation in
 * tensor memory.  X is gathered and converted to fp16 first, each row scaled
 * by the power of two that brings its largest |x| into [2^14, 2^15) (scaled
 * back in the epilogue), so the conversion is exact at any absolute scale
 * except for values more than about 2^28 below their row's largest; the
 * product is then within fp16 rounding of each weight. */
int polyq_linear_gemm(const polyq_dev_layer* layer, const void* X, int64_t M,
                      float* Y, void* workspace, size_t workspace_bytes,
                      void* stream);

/* Test aid: unpack the integer codes of every row into codes [N][K]
 * (device uint16, clustered order; for 16-bit channels the fp16 bit pattern).
 * Must equal the host-side codes bit for bit. */
int polyq_unpack_codes(const polyq_dev_layer* layer, uint16_t* codes,
                       void* stream);

/* Utility: round a double to the nearest fp16 (ties to even); returns the
 * fp16 bit pattern.  The packer's scale rounding. */
uint16_t polyq_f64_to_f16(double v);

#ifdef __cplusplus
}
#endif
#endif /* POLYQ_H */
