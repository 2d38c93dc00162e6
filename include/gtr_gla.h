/*
 * gtr_gla.h -- C ABI of the GB300 (sm_103a) chunkwise gated-linear-attention
 * forward: the token mixer of GTR ("GTR: Gated Token Recurrence for Efficient
 * Dense Prediction").
 *
 * Operation (Sec. 3.1, "Key-only gated recurrence"; value-side decay fixed to
 * one, Sec. 3.1 and App. C.3), per batch b and head h, along one scan order:
 *
 *     S_0 = 0,   S_t = Diag(exp(g_t)) S_{t-1} + k_t^T v_t,   o_t = q_t S_t
 *
 * with q_t, k_t, g_t in R^{1 x Dk}, v_t, o_t in R^{1 x Dv}, S_t in R^{Dk x Dv}.
 * g_t = log(gamma_t) is the learned per-key-channel log-decay the operator takes
 * as input (Sec. 3.3: "the same queries, keys, values, and learned
 * log-decays").  The paper's output factor d_k^{-1/2} is not applied: fold it
 * into k (or q) before the call.
 *
 * Scan orders (Sec. 3.1, "Directional scanning"): the T = grid_h * grid_w
 * tokens of a patch grid are stored in spatial row-major order
 * (t = y * grid_w + x).  The recurrence visits them in one of four raster
 * orders, one sequence per image with the state carried across rows/columns;
 * each output is written back at its token's spatial position (the block
 * "restores the original spatial order"):
 *     ROW_FWD  left-to-right:  position s visits t = s
 *     ROW_REV  right-to-left:  t = T-1-s          (exact reversal of ROW_FWD)
 *     COL_FWD  top-to-bottom:  t = (s mod grid_h) * grid_w + s div grid_h
 *     COL_REV  bottom-to-top:  COL_FWD applied to T-1-s (exact reversal)
 *
 * Schedule (Sec. 3.3 and App. C.3): chunks of C = 64 scan positions; the
 * in-chunk cumulative log-decay, the chunk summaries U_c, the boundary-state
 * carry S_[c+1] = Diag(d_c) S_[c] + U_c and the intra-chunk gated scores are
 * computed on the GPU; the scan permutation is applied inside the loads and
 * the output store.  The result equals the recurrence up to floating-point
 * rounding.
 *
 * Common argument rules (every entry point below):
 *   - q, k, log_gate : [B, T, H, Dk]  element type `dtype`, contiguous.
 *     v, out         : [B, T, H, Dv]  element type `dtype`, contiguous.
 *     final_state    : [B, H, Dk, Dv] float32, contiguous, or NULL (not written).
 *     All tensor pointers are device pointers unless stated otherwise, owned by
 *     the caller, 16-byte aligned, and `out` / `final_state` must not overlap
 *     the inputs.
 *   - log_gate must be <= 0 or -inf; values below -1e4 act as -1e4, which is
 *     gamma = 0 exactly in float32.  NaN inputs give NaN outputs.
 *   - B, H, grid_h, grid_w >= 1 (B*H*T == 0 is allowed only as B == 0 or H == 0,
 *     which launches nothing); 1 <= Dk, Dv <= 128.
 *   - The call is asynchronous on `stream`: it validates, enqueues kernels and
 *     returns.  Validation failures return before anything is enqueued.
 *     Launch failures return GTR_ERR_CUDA.  Conditions the device detects
 *     (a bounded wait that gave up) are recorded in a per-device status word
 *     and reported by gtr_gla_sync_status().
 *   - Allocation and synchronisation: gtr_gla_fwd, gtr_gla_fwd_sched and
 *     gtr_gla_fwd_gated keep an internal per-device workspace for the split
 *     and balanced schedules.  The first call that needs it, and any later
 *     call that needs more, allocates it with cudaMalloc (and frees the
 *     smaller one with cudaFree, which synchronises the device); calls made
 *     while their stream is being captured never touch it and run the
 *     round-robin schedule instead (gtr_gla_last_schedule reports both the
 *     schedule that ran and the one that was planned).  gtr_gla_fwd_host
 *     creates two streams and a set of events on its first call per device.
 *     Every other entry point allocates no device memory and does not
 *     synchronise: the _ws and _noalloc forms are the ones to capture in a
 *     CUDA graph with every schedule.  No entry point reads device data on the
 *     host except gtr_gla_sync_status.
 */
#ifndef GTR_GLA_H
#define GTR_GLA_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    GTR_OK = 0,
    GTR_ERR_INVALID_ARG = 1,  /* null / misaligned pointer, bad size or enum value   */
    GTR_ERR_UNSUPPORTED = 2,  /* well-formed, but the requested schedule cannot run  */
    GTR_ERR_WORKSPACE = 3,    /* workspace missing or smaller than required          */
    GTR_ERR_CUDA = 4,         /* a CUDA call failed; see gtr_last_cuda_error()       */
    GTR_ERR_TIMEOUT = 5       /* a bounded device-side wait gave up                  */
} gtr_status_t;

typedef enum { GTR_F32 = 0, GTR_F16 = 1, GTR_BF16 = 2 } gtr_dtype_t;

typedef enum {
    GTR_SCAN_ROW_FWD = 0,     /* left-to-right  */
    GTR_SCAN_ROW_REV = 1,     /* right-to-left  */
    GTR_SCAN_COL_FWD = 2,     /* top-to-bottom  */
    GTR_SCAN_COL_REV = 3      /* bottom-to-top  */
} gtr_scan_t;

/* Kernel schedule.  AUTO picks the fastest schedule that supports the
 * arguments.  SIMT is the plain fp32 CUDA-core recurrence (any dtype, any
 * shape within the common rules; the float32 path).  TC is the tensor-core
 * chunkwise schedule (tcgen05 MMAs, TMEM accumulators, TMA loads):
 * fp16/bf16 only, with the shape rules of gtr_gla_tc_supported(). */
typedef enum { GTR_SCHED_AUTO = 0, GTR_SCHED_SIMT = 1, GTR_SCHED_TC = 2 } gtr_schedule_t;

/* Forward of the token mixer with the AUTO schedule (argument rules above).
 * Returns GTR_OK once the work is enqueued on `stream`.  When few, long
 * sequences would leave most SMs idle, the tensor-core schedule splits each
 * sequence into segments of equal length but the last, which may run past the
 * sequence over all-zero chunks (a first pass stores every segment's end state
 * from zero and its total decay, the second pass starts each segment from the
 * fold of the earlier ones: the state carry of Eq. chunk_boundary_main applied
 * across segments).  Those summaries live in an internal per-device workspace
 * that this call allocates (cudaMalloc) the first time a problem needs it and
 * grows outside stream capture; under capture the call never touches it and
 * runs the schedule unsplit (gtr_gla_last_schedule then reports GTR_RAN_TC
 * against a planned GTR_RAN_TC_SPLIT).  Callers that manage memory themselves
 * use gtr_gla_fwd_ws. */
gtr_status_t gtr_gla_fwd(const void *q, const void *k, const void *v, const void *log_gate,
                         int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                         gtr_scan_t scan_order, gtr_dtype_t dtype,
                         void *out, float *final_state, cudaStream_t stream);

/* Same as gtr_gla_fwd with an explicit schedule.  Requesting a schedule that
 * cannot run these arguments returns GTR_ERR_UNSUPPORTED (never a silent
 * fallback). */
gtr_status_t gtr_gla_fwd_sched(const void *q, const void *k, const void *v,
                               const void *log_gate, int B, int H, int grid_h, int grid_w,
                               int Dk, int Dv, gtr_scan_t scan_order, gtr_dtype_t dtype,
                               void *out, float *final_state, gtr_schedule_t schedule,
                               cudaStream_t stream);

/* Bytes of workspace gtr_gla_fwd_ws needs for these arguments on the current
 * device: the segment summaries of the split schedule (B*H*(segments-1)*(Dk'*Dv'
 * + Dk') floats, Dk' and Dv' rounded up to multiples of 64), or, for the
 * balanced schedule (gtr_gla_balanced_plan), one 64 x 64 fp32 hand-off state and
 * one 64-bit flag per SM; 0 when the call needs neither (the SIMT schedule, or
 * whole sequences dealt round-robin) or the arguments are invalid.  Both depend
 * on the device's SM count. */
size_t gtr_gla_workspace_bytes(int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                               gtr_dtype_t dtype);

/* The sequence split the tensor-core schedule would use for these shapes on a
 * device with n_sm SMs: *nseg segments per sequence of *seg_len 64-token chunks
 * each (the last segment may run past the sequence over all-zero padding
 * chunks; *nseg == 1: unsplit, *seg_len = the chunk count).  Host arithmetic
 * only: no device is queried, so it answers for any SM count.  The split is the
 * chunkwise state carry (Eq. chunk_boundary_main) applied across segments; the
 * segment length minimises a cost model of the split's critical path measured
 * on a GB300.  Returns GTR_ERR_INVALID_ARG for invalid shapes, n_sm < 1 or
 * NULL outputs (the outputs are then not written). */
gtr_status_t gtr_gla_split_plan(int B, int H, int grid_h, int grid_w, int Dk, int Dv, int n_sm,
                                int *nseg, int *seg_len);

/* 1 when the tensor-core schedule balances these shapes on a device with n_sm SMs,
 * else 0 (also for invalid shapes or n_sm < 1).  Balanced: Dk <= 64, no sequence
 * split, more (sequence, 64-column value slice) units than SMs, and a round-robin
 * deal of whole units would give the busiest SM at least 1.1 times the chunks of an
 * even split; every
 * CTA then takes an equal contiguous range of the units' chunks, and a unit cut by
 * a range boundary continues from the state (Eq. chunk_boundary_main) the CTA
 * before it handed over through the workspace.  Host arithmetic only. */
int gtr_gla_balanced_plan(int B, int H, int grid_h, int grid_w, int Dk, int Dv, int n_sm);

/* The chunks one CTA of the balanced schedule processes, in its order, computed on
 * the host by the kernel's own decode (no device is used).  n_units (sequence,
 * value slice) units of n_chunks 64-token chunks each, in unit order, are cut into
 * `grid` equal contiguous ranges (1 <= grid <= n_units, so a range is at least one
 * unit long).  CTA `cta` (0 <= cta < grid) first runs the head of the unit its
 * range ends in (chunks 0 .. *head - 1, from a zero state; the state after them is
 * handed to CTA cta + 1), then its whole units, then the tail of the unit its range
 * starts in, from the state CTA cta - 1 handed over (Eq. chunk_boundary_main across
 * CTAs).  Writes min(count, cap) entries of 4 ints: unit, chunk, start (1 where a
 * unit's state is set: chunk 0, or the tail's first chunk) and hand-in (1 at the
 * tail's first chunk); *head receives the head run's length.  Returns the CTA's
 * chunk count, or -1 for invalid arguments (entries may be NULL when cap is 0;
 * head must not be NULL). */
int gtr_gla_balanced_walk(int n_units, int n_chunks, int grid, int cta, int *entries, int cap, int *head);

/* Introspection of the scan-order gather (Sec. 3.1, directional scanning): the
 * TMA boxes of 64-token chunk c of a sequence on a grid_h x grid_w patch grid,
 * computed on the host by the same code the kernel's producer runs.  The
 * tensor-core schedule loads a chunk as these boxes unless gtr_gla_chunk_walk
 * returns 1 for it (column-order chunks inside the sequence load as one walk).
 * Writes min(count, cap) boxes of 4 ints to `boxes`:
 * rows (1-64), first row of the chunk's 64-row shared-memory tile, and the two
 * token coordinates of the box's first row (row orders: token index, 0; column
 * orders: column x, row y; x == grid_w marks a box that lies wholly outside the
 * tensor and loads zeros).  Chunks at or past the sequence's end are the
 * all-zero padding chunks of a split's last segment.  Returns the chunk's box
 * count, or -1 for invalid arguments.  No device is used. */
int gtr_gla_chunk_boxes(int grid_h, int grid_w, gtr_scan_t scan_order, int c, int *boxes, int cap);

/* Whether the tensor-core schedule loads 64-token chunk c as one walk (Sec. 3.1,
 * directional scanning): for a column order and a chunk wholly inside the
 * sequence, each tensor's 64 tokens come in one TMA im2col load that starts at
 * grid column *x, row *y (the chunk's first walk position; reverse orders load the
 * forward range their chunk covers) and runs down that column and on into the
 * next ones.  Returns 1 and sets *x, *y in that case; 0 when the chunk loads as
 * the boxes of gtr_gla_chunk_boxes (row orders; chunks reaching past either end of
 * the sequence); -1 for invalid arguments (x and y must not be NULL).  Computed on
 * the host by the producer's own test; no device is used. */
int gtr_gla_chunk_walk(int grid_h, int grid_w, gtr_scan_t scan_order, int c, int *x, int *y);

/* gtr_gla_fwd with a caller-owned device workspace of workspace_bytes >=
 * gtr_gla_workspace_bytes() bytes, 256-byte aligned (may be NULL when that is
 * 0).  The call allocates nothing and does not synchronise.  Returns
 * GTR_ERR_WORKSPACE when the workspace is missing or too small.  Calls that
 * overlap on the GPU must not share a workspace. */
gtr_status_t gtr_gla_fwd_ws(const void *q, const void *k, const void *v, const void *log_gate,
                            int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                            gtr_scan_t scan_order, gtr_dtype_t dtype, void *out,
                            float *final_state, void *workspace, size_t workspace_bytes,
                            cudaStream_t stream);

/* The mixer followed by its output gate (Sec. 3.1): instead of o, `out`
 * receives u = SiLU(r) * RMSNorm(o) per head, where `gate` holds the gate's
 * pre-activation r = x W_r ([B, T, H, Dv], same dtype and layout as v) and
 * RMSNorm(o)_j = o_j / sqrt(mean over the head's Dv outputs of o^2 + eps) *
 * norm_weight[j] (`norm_weight`: Dv fp32 values on the device, shared by the
 * heads; eps >= 0).  App. C.3 fuses this epilogue into the mixer kernel's
 * output stores.  Here the tensor-core schedule does so (u rounded once, from
 * the fp32 outputs) for launches of few sequences with Dk, Dv <= 64 (at most half
 * as many B*H units as SMs), where it saves a launch; otherwise a second kernel
 * applies it to `out` in place right after the mixer (o is rounded to the dtype
 * in between), reading o back while it is still in L2: on GB300 that was measured
 * 1.14-1.26x faster than the fused stores for large batches, whose extra work
 * lands on the mixer's critical chain.  final_state is the mixer's state as in
 * gtr_gla_fwd.  `gate` and `norm_weight` must be 16-byte
 * aligned and `gate` must not overlap `out`.  Allocation, workspace and errors
 * as gtr_gla_fwd. */
gtr_status_t gtr_gla_fwd_gated(const void *q, const void *k, const void *v, const void *log_gate,
                               const void *gate, const float *norm_weight, float eps, int B, int H,
                               int grid_h, int grid_w, int Dk, int Dv, gtr_scan_t scan_order,
                               gtr_dtype_t dtype, void *out, float *final_state, cudaStream_t stream);

/* gtr_gla_fwd_gated with a caller-owned device workspace, as gtr_gla_fwd_ws:
 * workspace_bytes >= gtr_gla_workspace_bytes() (the gate needs none of its
 * own), 256-byte aligned, NULL allowed when that is 0.  Allocates nothing and
 * does not synchronise, so it may be captured into a CUDA graph with the split
 * schedule (gtr_gla_fwd_gated under capture runs unsplit).  Returns
 * GTR_ERR_WORKSPACE when the workspace is missing or too small; other
 * arguments and errors as gtr_gla_fwd_gated. */
gtr_status_t gtr_gla_fwd_gated_ws(const void *q, const void *k, const void *v, const void *log_gate,
                                  const void *gate, const float *norm_weight, float eps, int B, int H,
                                  int grid_h, int grid_w, int Dk, int Dv, gtr_scan_t scan_order,
                                  gtr_dtype_t dtype, void *out, float *final_state, void *workspace,
                                  size_t workspace_bytes, cudaStream_t stream);

/* Spatial SwiGLU between its two projections (Sec. 3.1, Eq. spatial_swiglu):
 *   out = SiLU(X W_g) * DWConv3x3(X W_v),
 * the step the deployed S-SwiGLU kernel fuses (Sec. 4).  `gate` = X W_g and
 * `value` = X W_v are [B, T, F] with T = grid_h * grid_w tokens in spatial
 * row-major order and in_stride elements from one token to the next (F for
 * separate tensors, 2F when both halves of one [B, T, 2F] projection output
 * are passed, value = gate + F).  The value branch is convolved per channel on
 * the grid_h x grid_w grid with zero padding: weight[f][i][j] (fp32, [F][3][3])
 * multiplies the value at row offset i - 1 and column offset j - 1 (the
 * cross-correlation of a depthwise 2-D convolution layer), plus bias[f] (fp32
 * [F], or NULL for none); the product with SiLU(gate) is accumulated in fp32
 * and rounded once to the dtype.  out: [B, T, F] contiguous, same dtype; it
 * must not overlap gate or value.  gate, value and out 16-byte aligned, F and
 * in_stride multiples of 8 elements (4 for fp32); grid_w <= 254.  Device
 * pointers; allocates nothing and does not synchronise (capturable).
 * Returns GTR_ERR_INVALID_ARG / GTR_ERR_UNSUPPORTED before any launch; a
 * device-side wait that gives up is reported by gtr_gla_sync_status. */
gtr_status_t gtr_sswiglu_dwconv(const void *gate, const void *value, long long in_stride,
                                const float *weight, const float *bias, int B, int grid_h,
                                int grid_w, int F, gtr_dtype_t dtype, void *out, cudaStream_t stream);

/* The mixer with its retention gate computed inside the kernel (Sec. 3.1, the key-wise
 * retention gate gamma_t = sigmoid(x_t W_1 W_2 + b)^(1/tau) with a rank-r factorisation of
 * the gate projection): instead of a stored log_gate, the kernel reads the rank-r projection
 * a = x W_1 of every token and forms
 *
 *     g[b,t,h,:] = logsigmoid(a[b,t,:] W2[h] + bias[h]) / tau
 *
 * per chunk: Z = a W2 by a tensor-core product, the log-sigmoid in fp32, g rounded to fp16,
 * then the schedule of gtr_gla_fwd.  The gate tensor ([B, T, H, Dk], 2 Dk bytes per
 * token-head) is never written or read; a costs 2 r bytes per token for all heads.
 *   a_low     : [B, T, rank], element type `dtype`, contiguous, 16-byte aligned.
 *   w2        : [H, rank, Dk], element type `dtype`, contiguous, 16-byte aligned.
 *   gate_bias : [H, Dk] float32, contiguous, 16-byte aligned.
 *   tau       : > 0 (the paper uses 16).
 * q, k, v, out, final_state and the other arguments as gtr_gla_fwd.  Tensor-core
 * schedule only: fp16 or bf16, rank == 16 (the paper's rank), Dk a multiple of 8 up to 64,
 * Dv a multiple of 8 up to 128, and T = grid_h * grid_w > 192; other well-formed
 * arguments return GTR_ERR_UNSUPPORTED.  Sequences are dealt whole to the SMs (no split, no
 * balanced ranges): allocates nothing and does not synchronise (capturable).
 * Errors as gtr_gla_fwd; gtr_gla_last_schedule reports GTR_RAN_TC. */
gtr_status_t gtr_gla_fwd_lowrank_gate(const void *q, const void *k, const void *v, const void *a_low,
                                      const void *w2, const float *gate_bias, float tau, int rank,
                                      int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                                      gtr_scan_t scan_order, gtr_dtype_t dtype, void *out,
                                      float *final_state, cudaStream_t stream);

/* Size of the fixed device scratch array behind gtr_gla_fwd_noalloc.  The
 * library holds one such array on every GPU where it is loaded, from the
 * module's load until the process exits.  What a call keeps there is bounded by
 * the device's SM count n_sm:
 *   - split schedule: B*H*(segments-1) summaries of (Dk'*Dv' + Dk') floats
 *     (Dk', Dv' rounded up to 64), and the split keeps B*H*nv*segments <= n_sm
 *     with nv = Dv'/64, so at most floor(n_sm/nv) * (Dk'*Dv' + Dk') * 4 bytes,
 *     which is largest for Dk = 128, Dv <= 64: n_sm * 33,280 bytes;
 *   - balanced schedule: n_sm * (64*64*4 + 8) = n_sm * 16,392 bytes.
 * So 8 MiB covers every problem on devices of up to 252 SMs (a 152-SM GB300
 * needs at most 5.06 MB); on larger devices a problem over the limit returns
 * GTR_ERR_WORKSPACE. */
#define GTR_GLA_NOALLOC_SCRATCH_BYTES (8u << 20)

/* gtr_gla_fwd for callers that must not allocate device memory on the call
 * path.  One example is an engine that reserves all of HBM for its own pool at
 * start-up.  Another is a latency-critical loop: cudaFree synchronises the
 * whole device, and cudaMalloc can.  gtr_gla_fwd may cudaMalloc its internal
 * workspace, and gtr_gla_fwd_ws needs a buffer that the caller owns.  This
 * call uses neither.  The paper has no counterpart; it changes only where the
 * segment summaries of the split schedule are kept.
 *
 * Arguments, results and errors are those of gtr_gla_fwd.  The summaries go to
 * a fixed array of GTR_GLA_NOALLOC_SCRATCH_BYTES in this library.  A problem
 * whose gtr_gla_workspace_bytes() exceeds that returns GTR_ERR_WORKSPACE before
 * anything is launched.  The call allocates no device memory and does not
 * synchronise.
 *
 * Set-up: the first call on each device looks up the array's device address
 * (cudaGetSymbolAddress, with that device current).  Make that first call
 * before capturing any stream on that device; a failed lookup returns
 * GTR_ERR_CUDA.
 *
 * Every call on a device shares the one array, and it keeps what the last call
 * wrote.  Nothing in it must start at zero: the first kernel of a call writes
 * every summary that the call's second kernel reads.  Calls whose kernels
 * overlap on the GPU race on the array and give wrong results, for example
 * calls on two streams with no ordering between them.  Order them on one
 * stream or with events. */
gtr_status_t gtr_gla_fwd_noalloc(const void *q, const void *k, const void *v, const void *log_gate,
                                 int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                                 gtr_scan_t scan_order, gtr_dtype_t dtype, void *out,
                                 float *final_state, cudaStream_t stream);

/* 1 when the tensor-core schedule supports these arguments, else 0: fp16 or
 * bf16, Dk and Dv each a multiple of 8 up to 128 (processed in 64-channel key
 * halves and 64-column value slices, a narrower last one zero-padded on
 * load); any grid. */
int gtr_gla_tc_supported(int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                         gtr_scan_t scan_order, gtr_dtype_t dtype);

/* Bytes of device memory gtr_gla_fwd_host needs as `dev_buffer` (inputs,
 * output and final state staged on the device, each 256-byte aligned). */
size_t gtr_gla_host_buffer_bytes(int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                                 gtr_dtype_t dtype, int with_final_state);

/* End-to-end forward from HOST memory: copies q, k, v, log_gate (host
 * pointers, same layouts as above; pinned memory makes the copies
 * asynchronous) into `dev_buffer` (caller-owned device memory of at least
 * gtr_gla_host_buffer_bytes() bytes), runs gtr_gla_fwd on `stream`, and
 * copies `out` (and `final_state` when non-NULL) back to the host pointers.
 * The batch is processed in up to four pieces so that uploads, compute and
 * downloads overlap: the uploads and downloads run on two internal streams of
 * the current device (created with a set of events on its first call and kept
 * until exit), forked from and joined back into `stream` with events, so the
 * call is ordered on `stream` like any other work: synchronise it before
 * reading the results.  Calls from several host threads are serialised.
 * Errors as gtr_gla_fwd, plus GTR_ERR_WORKSPACE when dev_buffer is NULL or
 * too small. */
gtr_status_t gtr_gla_fwd_host(const void *q_host, const void *k_host, const void *v_host,
                              const void *log_gate_host, int B, int H, int grid_h, int grid_w,
                              int Dk, int Dv, gtr_scan_t scan_order, gtr_dtype_t dtype,
                              void *out_host, float *final_state_host, void *dev_buffer,
                              size_t dev_buffer_bytes, cudaStream_t stream);

/* Synchronises `stream`, then returns and clears the device status word of the
 * current device (GTR_OK when no device-side condition was recorded,
 * GTR_ERR_TIMEOUT when a bounded wait gave up), or GTR_ERR_CUDA when the
 * synchronisation itself failed.  Every device-side wait gives up after 1 s;
 * the kernel then drains its copies, frees its tensor memory and returns, so
 * the context stays usable (the outputs of that call are undefined).  Test
 * hook for this path: with the environment variable GTR_GLA_TEST_DROP_LOAD=1
 * the tensor-core schedule withholds one chunk's load in its first CTA, so the
 * call reports GTR_ERR_TIMEOUT (no fault is involved). */
gtr_status_t gtr_gla_sync_status(cudaStream_t stream);

/* Schedules a forward call can run (gtr_gla_last_schedule). */
typedef enum {
    GTR_RAN_NONE = 0,         /* nothing launched (no call yet on this thread, or B*H == 0)      */
    GTR_RAN_SIMT = 1,         /* fp32 CUDA-core recurrence                                        */
    GTR_RAN_TC = 2,           /* tensor cores, whole sequences dealt round-robin to the SMs       */
    GTR_RAN_TC_SPLIT = 3,     /* tensor cores, sequences split into segments (two launches)       */
    GTR_RAN_TC_BALANCED = 4   /* tensor cores, equal chunk ranges per SM with state hand-offs     */
} gtr_ran_t;

/* What the last successful forward call (gtr_gla_fwd, _sched, _ws, _gated,
 * _gated_ws, _noalloc; gtr_gla_fwd_host: its last piece) of this host thread
 * enqueued: *ran receives the schedule that was launched and *planned the one
 * the library would have chosen with enough workspace.  They differ when the
 * split or balanced schedule was dropped for lack of workspace, for example
 * gtr_gla_fwd under stream capture before its internal workspace had grown to
 * the size the problem needs.  Either pointer may be NULL.  Host state only:
 * nothing is launched or synchronised. */
gtr_status_t gtr_gla_last_schedule(int *ran, int *planned);

/* Static, NUL-terminated description of a status code. */
const char *gtr_status_string(gtr_status_t status);

/* The cudaError_t value behind the last GTR_ERR_CUDA returned on this host
 * thread (0 when none). */
int gtr_last_cuda_error(void);

/* Library version, MAJOR * 10000 + MINOR * 100 + PATCH. */
int gtr_version(void);

#ifdef __cplusplus
}
#endif

#endif /* GTR_GLA_H */
