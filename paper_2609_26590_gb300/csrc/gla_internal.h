// gla_internal.h -- declarations shared by the translation units of the GB300
// GLA library (host side only; kernels live in their own .cu files).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace gtr {

// One forward call, as validated by the C ABI (include/gtr_gla.h).
struct Problem {
    const void *q, *k, *v, *g;  // [B,T,H,Dk] x3, [B,T,H,Dv]
    void *out;                  // [B,T,H,Dv]
    float *final_state;         // [B,H,Dk,Dv] or nullptr
    int B, H, grid_h, grid_w, Dk, Dv;
    int order;                  // gtr_scan_t
    int dtype;                  // gtr_dtype_t
    long long T;                // grid_h * grid_w
};

// Output gate of Sec. 3.1, u = SiLU(r) * RMSNorm(o) per head (RMSNorm over Dv
// with a weight vector of Dv entries shared by the heads).
struct Gate {
    const void *r;    // [B,T,H,Dv] gate pre-activation x W_r, input dtype
    const float *w;   // [Dv] RMSNorm weight
    float eps;
};

// Plain fp32 CUDA-core recurrence (gla_simt.cu).  Any dtype, Dk, Dv <= 128.
cudaError_t launch_simt(const Problem &p, cudaStream_t stream);
// The gate applied in place to a finished output (gla_simt.cu, CUDA cores; any
// dtype, Dv <= 128): 16-byte vectors per lane, a row's lanes reduce its RMS.
cudaError_t launch_gate_epilogue(const Problem &p, const Gate &gate, cudaStream_t stream);

// Tensor-core chunkwise schedule (gla_tc.cu).
bool tc_supported(const Problem &p);
// The TMA boxes the tensor-core producer loads for chunk c (the kernel's own
// enumeration, run on the host): up to cap boxes of 4 ints (rows, shared-memory row,
// coordinate 2, coordinate 3); returns how many the chunk has.
int tc_chunk_boxes(int order, int T, int grid_h, int grid_w, int c, int *boxes, int cap);
int tc_chunk_walk(int order, int T, int grid_h, int c, int *x0, int *y0);
// The balanced schedule's walk of CTA cta of grid over n_units units of N chunks: entries of
// (unit, chunk, start, hand-in), *head = the head run's length; returns the chunk count.
int tc_balanced_walk(int n_units, int N, int grid, int cta, int *entries, int cap, int *head);
// Segments per sequence and chunks per segment the tensor-core schedule uses for
// this problem on a device with n_sm SMs (host arithmetic only; nseg 1: unsplit).
void tc_split_plan(const Problem &p, int n_sm, int *nseg, int *seg_len);
// Scratch the tensor-core schedule uses for this problem on the current device:
// per-segment summaries when it splits sequences (few, long ones), hand-off states and
// flags when it balances chunk ranges (tc_balanced_plan), else 0.
size_t tc_workspace_bytes(const Problem &p);
// 1 when the tensor-core schedule gives every CTA an equal contiguous range of chunks
// (more units than SMs, a round-robin deal at least 1.1 times an even split's share) on a device
// with n_sm SMs; its workspace then holds one hand-off state and flag per SM.
int tc_balanced_plan(const Problem &p, int n_sm);
// Which schedule a launch ran, and which one it would have run with enough workspace
// (values of gtr_ran_t in include/gtr_gla.h).
struct Ran {
    int ran = 0, planned = 0;
};
enum : int { kRanNone = 0, kRanSimt = 1, kRanTc = 2, kRanTcSplit = 3, kRanTcBalanced = 4 };
// Launches the schedule; it splits sequences or balances ranges only when `workspace`
// holds at least tc_workspace_bytes(p) bytes (256-byte aligned), else it deals whole
// sequences round-robin.  *ran (may be null) receives what was launched and planned.  With
// `gate`, launches whose rows fit one thread pair (Dk, Dv <= 64) and are not balanced apply
// the output gate in the kernel's stores and set *gate_fused; otherwise the caller applies it.
cudaError_t launch_tc(const Problem &p, cudaStream_t stream, void *workspace, size_t workspace_bytes,
                      Ran *ran = nullptr, const Gate *gate = nullptr, bool *gate_fused = nullptr);

// The retention gate computed inside the mixer (Sec. 3.1): g = logsigmoid(a W2 + b) / tau from
// the rank-r projection a = x W1 instead of a stored g.
struct GateSource {
    const void *a_low;   // [B, T, r] in the problem's dtype
    const void *w2;      // [H, r, Dk] in the problem's dtype
    const float *bias;   // [H, Dk]
    float tau;
};
// Whether launch_tc_gate takes these shapes: the tensor-core dtypes, Dk <= 64 (one key half),
// rank 16, and at least four 64-token chunks per sequence.
bool tc_gate_supported(const Problem &p, int rank);
// The tensor-core schedule with the gate producer (whole sequences dealt round-robin; the
// problem's g pointer is not used).
cudaError_t launch_tc_gate(const Problem &p, const GateSource &gs, cudaStream_t stream, Ran *ran = nullptr);

// Device status word of the current device (set by bounded device waits).
cudaError_t read_and_clear_device_status(unsigned int *status);

// The driver's cuTensorMapEncodeTiled (as void *; null when the driver lacks it).
void *tensor_map_encoder();

// Spatial SwiGLU between its projections (sswiglu.cu): out = SiLU(gate) * DWConv3x3(value).
struct SwProblem {
    const void *gate, *value;   // [B, T, F] at in_stride elements per token
    long long in_stride;
    const float *weight;        // [F][3][3]
    const float *bias;          // [F] or null
    void *out;                  // [B, T, F], F elements per token
    int B, grid_h, grid_w, F;
    int dtype;                  // 0 f32, 1 f16, 2 bf16
};
// Grids the kernel takes (a tile's box spans the grid width plus the halo).
bool sswiglu_supported(const SwProblem &p);
cudaError_t launch_sswiglu(const SwProblem &p, cudaStream_t stream);
// Status word of the S-SwiGLU kernel's bounded wait (kStatusTimeout).
cudaError_t read_and_clear_sswiglu_status(unsigned int *status);

enum : unsigned int { kStatusTimeout = 1u };

}  // namespace gtr
