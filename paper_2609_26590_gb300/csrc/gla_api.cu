// gla_api.cu -- the C ABI of include/gtr_gla.h: argument validation, schedule
// dispatch, the host-memory entry point and status reporting.  No kernel code;
// one device array, the scratch of gtr_gla_fwd_noalloc.
#include <cstdint>
#include <cstring>
#include <mutex>
#include <vector>

#include "gla_internal.h"
#include "gtr_gla.h"

// Segment summaries of gtr_gla_fwd_noalloc, for callers that may not allocate
// device memory.  Every device that loads this library holds one copy until the
// process exits.  Host code reaches it only through the address that
// noalloc_scratch() looks up.
static __device__ __align__(256) unsigned char g_noalloc_scratch[GTR_GLA_NOALLOC_SCRATCH_BYTES];

namespace {

thread_local int t_last_cuda_error = 0;
thread_local gtr::Ran t_last_ran;  // schedule of this thread's last successful forward call

gtr_status_t nothing_launched() {
    t_last_ran = gtr::Ran{};
    return GTR_OK;
}

constexpr size_t kAlign = 16;
constexpr int kMaxHeadDim = 128;

bool aligned(const void *p) { return (reinterpret_cast<uintptr_t>(p) % kAlign) == 0; }

size_t elem_size(int dtype) { return dtype == GTR_F32 ? 4 : 2; }

bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
    if (a == nullptr || b == nullptr || na == 0 || nb == 0) return false;
    auto pa = reinterpret_cast<uintptr_t>(a), pb = reinterpret_cast<uintptr_t>(b);
    return pa < pb + nb && pb < pa + na;
}

gtr_status_t cuda_fail(cudaError_t e) {
    t_last_cuda_error = static_cast<int>(e);
    return GTR_ERR_CUDA;
}

// Shape / enum checks shared by every entry point.
gtr_status_t check_shape(int B, int H, int grid_h, int grid_w, int Dk, int Dv, int order,
                         int dtype) {
    if (B < 0 || H < 0 || grid_h < 1 || grid_w < 1) return GTR_ERR_INVALID_ARG;
    if (Dk < 1 || Dv < 1 || Dk > kMaxHeadDim || Dv > kMaxHeadDim) return GTR_ERR_INVALID_ARG;
    if (order < GTR_SCAN_ROW_FWD || order > GTR_SCAN_COL_REV) return GTR_ERR_INVALID_ARG;
    if (dtype < GTR_F32 || dtype > GTR_BF16) return GTR_ERR_INVALID_ARG;
    const long long T = (long long)grid_h * grid_w;
    if (T > 0x7fffffffLL) return GTR_ERR_INVALID_ARG;
    if ((long long)B * H > 0x7fffffffLL) return GTR_ERR_INVALID_ARG;
    const long long D = Dk > Dv ? Dk : Dv;
    // every element offset must fit in int64 with room to spare
    if ((long long)B * T > (1LL << 40) / ((long long)H * D + 1)) return GTR_ERR_INVALID_ARG;
    return GTR_OK;
}

gtr_status_t make_problem(const void *q, const void *k, const void *v, const void *g, int B,
                          int H, int grid_h, int grid_w, int Dk, int Dv, int order, int dtype,
                          void *out, float *final_state, gtr::Problem *p) {
    gtr_status_t st = check_shape(B, H, grid_h, grid_w, Dk, Dv, order, dtype);
    if (st != GTR_OK) return st;
    const long long T = (long long)grid_h * grid_w;
    if (B == 0 || H == 0) {  // nothing is read or written: pointers may be null
        *p = gtr::Problem{q, k, v, g, out, final_state, B, H, grid_h, grid_w, Dk, Dv, order, dtype, T};
        return GTR_OK;
    }
    if (!q || !k || !v || !g || !out) return GTR_ERR_INVALID_ARG;
    if (!aligned(q) || !aligned(k) || !aligned(v) || !aligned(g) || !aligned(out) ||
        !aligned(final_state))
        return GTR_ERR_INVALID_ARG;
    const size_t es = elem_size(dtype);
    const size_t nk = (size_t)B * T * H * Dk * es, nv = (size_t)B * T * H * Dv * es;
    const size_t nfs = (size_t)B * H * Dk * Dv * sizeof(float);
    const void *ins[4] = {q, k, v, g};
    const size_t ins_n[4] = {nk, nk, nv, nk};
    for (int i = 0; i < 4; ++i) {
        if (overlaps(out, nv, ins[i], ins_n[i])) return GTR_ERR_INVALID_ARG;
        if (overlaps(final_state, nfs, ins[i], ins_n[i])) return GTR_ERR_INVALID_ARG;
    }
    if (overlaps(out, nv, final_state, nfs)) return GTR_ERR_INVALID_ARG;
    *p = gtr::Problem{q, k, v, g, out, final_state, B, H, grid_h, grid_w, Dk, Dv, order, dtype, T};
    return GTR_OK;
}

size_t round_up(size_t n, size_t a) { return (n + a - 1) / a * a; }

// Internal per-device workspace of gtr_gla_fwd (segment summaries of the split
// schedule).  It grows, outside stream capture, to the largest size asked for and
// is kept until exit.  A call whose stream is being captured never uses it, so no
// captured graph refers to memory that a later growth frees.
struct DeviceWorkspace {
    void *ptr = nullptr;
    size_t bytes = 0;
};
std::mutex g_ws_mutex;
std::vector<DeviceWorkspace> g_ws;

void *internal_workspace(size_t need, cudaStream_t stream, size_t *got) {
    *got = 0;
    if (need == 0) return nullptr;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) return nullptr;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
    std::lock_guard<std::mutex> lock(g_ws_mutex);
    if ((size_t)dev >= g_ws.size()) g_ws.resize(dev + 1);
    DeviceWorkspace &w = g_ws[dev];
    if (w.bytes < need) {
        if (w.ptr != nullptr && cudaFree(w.ptr) != cudaSuccess) return nullptr;  // waits for its users
        w.ptr = nullptr;
        w.bytes = 0;
        if (cudaMalloc(&w.ptr, need) != cudaSuccess) {
            w.ptr = nullptr;
            cudaGetLastError();  // the schedule runs unsplit instead
            return nullptr;
        }
        w.bytes = need;
    }
    *got = w.bytes;
    return w.ptr;
}

// Device address of g_noalloc_scratch on the current device, looked up on the
// first call per device and kept (null: not looked up yet).
std::mutex g_noalloc_mutex;
std::vector<void *> g_noalloc_ptr;

cudaError_t noalloc_scratch(void **ptr) {
    *ptr = nullptr;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if ((size_t)dev >= g_noalloc_ptr.size()) g_noalloc_ptr.resize(dev + 1, nullptr);
    if (g_noalloc_ptr[dev] == nullptr) {
        void *addr = nullptr;
        e = cudaGetSymbolAddress(&addr, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = addr;
    }
    *ptr = g_noalloc_ptr[dev];
    return cudaSuccess;
}

// Per-device streams and events of gtr_gla_fwd_host's pipeline (created on first
// use and kept; calls are serialised by g_pipe_mutex, so the events are reused).
constexpr int kPipePieces = 4;
struct HostPipe {
    bool ready = false;
    cudaStream_t up = nullptr, down = nullptr;
    cudaEvent_t fork = nullptr, join = nullptr;
    cudaEvent_t in[kPipePieces] = {}, done[kPipePieces] = {};
};
std::mutex g_pipe_mutex;
std::vector<HostPipe> g_pipe;

cudaError_t host_pipe(HostPipe **out) {  // caller holds g_pipe_mutex
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if ((size_t)dev >= g_pipe.size()) g_pipe.resize(dev + 1);
    HostPipe &hp = g_pipe[dev];
    if (!hp.ready) {
        const unsigned ef = cudaEventDisableTiming;
        if ((e = cudaStreamCreateWithFlags(&hp.up, cudaStreamNonBlocking)) != cudaSuccess ||
            (e = cudaStreamCreateWithFlags(&hp.down, cudaStreamNonBlocking)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&hp.fork, ef)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&hp.join, ef)) != cudaSuccess)
            return e;
        for (int j = 0; j < kPipePieces; ++j)
            if ((e = cudaEventCreateWithFlags(&hp.in[j], ef)) != cudaSuccess ||
                (e = cudaEventCreateWithFlags(&hp.done[j], ef)) != cudaSuccess)
                return e;
        hp.ready = true;
    }
    *out = &hp;
    return cudaSuccess;
}

// Dispatch of one validated, non-empty problem; `ws` null means the internal workspace.
gtr_status_t dispatch(const gtr::Problem &p, gtr_schedule_t schedule, void *ws, size_t ws_bytes, bool own_ws,
                      cudaStream_t stream, const gtr::Gate *gate = nullptr, bool *gate_fused = nullptr) {
    if (gate_fused) *gate_fused = false;
    cudaError_t e;
    const bool tc = gtr::tc_supported(p);
    gtr::Ran r;
    if (schedule == GTR_SCHED_SIMT || (schedule == GTR_SCHED_AUTO && !tc)) {
        e = gtr::launch_simt(p, stream);
        r.ran = r.planned = gtr::kRanSimt;
    } else {
        if (!tc) return GTR_ERR_UNSUPPORTED;
        if (!own_ws) ws = internal_workspace(gtr::tc_workspace_bytes(p), stream, &ws_bytes);
        e = gtr::launch_tc(p, stream, ws, ws_bytes, &r, gate, gate_fused);
    }
    if (e != cudaSuccess) return cuda_fail(e);
    t_last_ran = r;
    return GTR_OK;
}

}  // namespace

extern "C" {

gtr_status_t gtr_gla_fwd_sched(const void *q, const void *k, const void *v, const void *log_gate,
                               int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                               gtr_scan_t scan_order, gtr_dtype_t dtype, void *out,
                               float *final_state, gtr_schedule_t schedule, cudaStream_t stream) {
    gtr::Problem p;
    gtr_status_t st = make_problem(q, k, v, log_gate, B, H, grid_h, grid_w, Dk, Dv, scan_order,
                                   dtype, out, final_state, &p);
    if (st != GTR_OK) return st;
    if (schedule < GTR_SCHED_AUTO || schedule > GTR_SCHED_TC) return GTR_ERR_INVALID_ARG;
    if (B == 0 || H == 0) return nothing_launched();
    return dispatch(p, schedule, nullptr, 0, false, stream);
}

size_t gtr_gla_workspace_bytes(int B, int H, int grid_h, int grid_w, int Dk, int Dv, gtr_dtype_t dtype) {
    if (check_shape(B, H, grid_h, grid_w, Dk, Dv, 0, dtype) != GTR_OK || B == 0 || H == 0) return 0;
    gtr::Problem p{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, B, H, grid_h, grid_w,
                   Dk, Dv, 0, dtype, (long long)grid_h * grid_w};
    return gtr::tc_supported(p) ? gtr::tc_workspace_bytes(p) : 0;
}

int gtr_gla_chunk_boxes(int grid_h, int grid_w, gtr_scan_t scan_order, int c, int *boxes, int cap) {
    if (grid_h < 1 || grid_w < 1 || (long long)grid_h * grid_w > 0x7fffffffLL) return -1;
    if (scan_order < GTR_SCAN_ROW_FWD || scan_order > GTR_SCAN_COL_REV || c < 0 || cap < 0) return -1;
    if (cap > 0 && boxes == nullptr) return -1;
    const long long T = (long long)grid_h * grid_w;
    if ((long long)c * 64 > T + (1LL << 24)) return -1;  // far past the sequence: no schedule asks
    return gtr::tc_chunk_boxes(scan_order, static_cast<int>(T), grid_h, grid_w, c, boxes, cap);
}

int gtr_gla_chunk_walk(int grid_h, int grid_w, gtr_scan_t scan_order, int c, int *x, int *y) {
    if (grid_h < 1 || grid_w < 1 || (long long)grid_h * grid_w > 0x7fffffffLL) return -1;
    if (scan_order < GTR_SCAN_ROW_FWD || scan_order > GTR_SCAN_COL_REV || c < 0 || !x || !y) return -1;
    const long long T = (long long)grid_h * grid_w;
    if ((long long)c * 64 > T + (1LL << 24)) return -1;  // far past the sequence: no schedule asks
    return gtr::tc_chunk_walk(scan_order, static_cast<int>(T), grid_h, c, x, y);
}

int gtr_gla_balanced_walk(int n_units, int n_chunks, int grid, int cta, int *entries, int cap, int *head) {
    if (n_units < 1 || n_chunks < 1 || grid < 1 || grid > n_units || cta < 0 || cta >= grid) return -1;
    if ((long long)n_units * n_chunks > 0x7fffffffLL || cap < 0 || (cap > 0 && entries == nullptr) || !head) return -1;
    return gtr::tc_balanced_walk(n_units, n_chunks, grid, cta, entries, cap, head);
}

gtr_status_t gtr_gla_split_plan(int B, int H, int grid_h, int grid_w, int Dk, int Dv, int n_sm, int *nseg,
                                int *seg_len) {
    if (!nseg || !seg_len || n_sm < 1) return GTR_ERR_INVALID_ARG;
    const gtr_status_t st = check_shape(B, H, grid_h, grid_w, Dk, Dv, 0, GTR_F16);
    if (st != GTR_OK) return st;
    gtr::Problem p{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, B, H, grid_h, grid_w,
                   Dk, Dv, 0, GTR_F16, (long long)grid_h * grid_w};
    if (B == 0 || H == 0) {
        *nseg = 1;
        *seg_len = static_cast<int>((p.T + 63) / 64);
        return GTR_OK;
    }
    gtr::tc_split_plan(p, n_sm, nseg, seg_len);
    return GTR_OK;
}

int gtr_gla_balanced_plan(int B, int H, int grid_h, int grid_w, int Dk, int Dv, int n_sm) {
    if (n_sm < 1 || check_shape(B, H, grid_h, grid_w, Dk, Dv, 0, GTR_F16) != GTR_OK || B == 0 || H == 0) return 0;
    gtr::Problem p{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, B, H, grid_h, grid_w,
                   Dk, Dv, 0, GTR_F16, (long long)grid_h * grid_w};
    return gtr::tc_balanced_plan(p, n_sm);
}

gtr_status_t gtr_gla_fwd_ws(const void *q, const void *k, const void *v, const void *log_gate, int B,
                            int H, int grid_h, int grid_w, int Dk, int Dv, gtr_scan_t scan_order,
                            gtr_dtype_t dtype, void *out, float *final_state, void *workspace,
                            size_t workspace_bytes, cudaStream_t stream) {
    gtr::Problem p;
    gtr_status_t st = make_problem(q, k, v, log_gate, B, H, grid_h, grid_w, Dk, Dv, scan_order,
                                   dtype, out, final_state, &p);
    if (st != GTR_OK) return st;
    if ((reinterpret_cast<uintptr_t>(workspace) % 256) != 0) return GTR_ERR_INVALID_ARG;
    if (B == 0 || H == 0) return nothing_launched();
    const size_t need = gtr_gla_workspace_bytes(B, H, grid_h, grid_w, Dk, Dv, dtype);
    if (need > 0 && (workspace == nullptr || workspace_bytes < need)) return GTR_ERR_WORKSPACE;
    return dispatch(p, GTR_SCHED_AUTO, workspace, workspace_bytes, true, stream);
}

}  // extern "C"

namespace {

// The mixer, then the gate over its output in place (the output is still in L2 for
// workloads that fit there); `own_ws`: the caller's workspace, else the internal one.
gtr_status_t gated(const void *q, const void *k, const void *v, const void *log_gate, const void *gate,
                   const float *norm_weight, float eps, int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                   gtr_scan_t scan_order, gtr_dtype_t dtype, void *out, float *final_state, void *ws,
                   size_t ws_bytes, bool own_ws, cudaStream_t stream) {
    gtr::Problem p;
    gtr_status_t st = make_problem(q, k, v, log_gate, B, H, grid_h, grid_w, Dk, Dv, scan_order,
                                   dtype, out, final_state, &p);
    if (st != GTR_OK) return st;
    if (!(eps >= 0.f) || !(eps < 3.0e38f)) return GTR_ERR_INVALID_ARG;  // also rejects NaN
    if (B == 0 || H == 0) return nothing_launched();
    if (!gate || !norm_weight || !aligned(gate) || !aligned(norm_weight)) return GTR_ERR_INVALID_ARG;
    const size_t nv = (size_t)B * p.T * H * Dv * elem_size(dtype);
    if (overlaps(out, nv, gate, nv)) return GTR_ERR_INVALID_ARG;
    if (own_ws) {
        const size_t need = gtr_gla_workspace_bytes(B, H, grid_h, grid_w, Dk, Dv, dtype);
        if (need > 0 && (ws == nullptr || ws_bytes < need)) return GTR_ERR_WORKSPACE;
    }
    // the tensor-core schedule applies the gate in its stores where a row's outputs stay in one
    // CTA (Dk, Dv <= 64, not balanced); otherwise a second kernel applies it to `out` in place
    const gtr::Gate g{gate, norm_weight, eps};
    bool fused = false;
    st = dispatch(p, GTR_SCHED_AUTO, ws, ws_bytes, own_ws, stream, &g, &fused);
    if (st != GTR_OK) return st;
    if (fused) return GTR_OK;
    const cudaError_t e = gtr::launch_gate_epilogue(p, g, stream);
    if (e != cudaSuccess) return cuda_fail(e);
    return GTR_OK;
}

}  // namespace

extern "C" {

gtr_status_t gtr_gla_fwd_gated(const void *q, const void *k, const void *v, const void *log_gate,
                               const void *gate, const float *norm_weight, float eps, int B, int H,
                               int grid_h, int grid_w, int Dk, int Dv, gtr_scan_t scan_order,
                               gtr_dtype_t dtype, void *out, float *final_state, cudaStream_t stream) {
    return gated(q, k, v, log_gate, gate, norm_weight, eps, B, H, grid_h, grid_w, Dk, Dv, scan_order, dtype,
                 out, final_state, nullptr, 0, false, stream);
}

gtr_status_t gtr_gla_fwd_gated_ws(const void *q, const void *k, const void *v, const void *log_gate,
                                  const void *gate, const float *norm_weight, float eps, int B, int H,
                                  int grid_h, int grid_w, int Dk, int Dv, gtr_scan_t scan_order,
                                  gtr_dtype_t dtype, void *out, float *final_state, void *workspace,
                                  size_t workspace_bytes, cudaStream_t stream) {
    return gated(q, k, v, log_gate, gate, norm_weight, eps, B, H, grid_h, grid_w, Dk, Dv, scan_order, dtype,
                 out, final_state, workspace, workspace_bytes, true, stream);
}

gtr_status_t gtr_gla_fwd_noalloc(const void *q, const void *k, const void *v, const void *log_gate,
                                 int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                                 gtr_scan_t scan_order, gtr_dtype_t dtype, void *out,
                                 float *final_state, cudaStream_t stream) {
    gtr::Problem p;
    gtr_status_t st = make_problem(q, k, v, log_gate, B, H, grid_h, grid_w, Dk, Dv, scan_order,
                                   dtype, out, final_state, &p);
    if (st != GTR_OK) return st;
    if (B == 0 || H == 0) return nothing_launched();
    if (gtr_gla_workspace_bytes(B, H, grid_h, grid_w, Dk, Dv, dtype) > GTR_GLA_NOALLOC_SCRATCH_BYTES)
        return GTR_ERR_WORKSPACE;
    void *scratch = nullptr;
    const cudaError_t e = noalloc_scratch(&scratch);
    if (e != cudaSuccess) return cuda_fail(e);
    // The summary pass writes every summary the output pass reads, so what an
    // earlier call left in the array is never read and nothing is cleared.
    return dispatch(p, GTR_SCHED_AUTO, scratch, GTR_GLA_NOALLOC_SCRATCH_BYTES, true, stream);
}

gtr_status_t gtr_gla_fwd_lowrank_gate(const void *q, const void *k, const void *v, const void *a_low,
                                      const void *w2, const float *gate_bias, float tau, int rank, int B, int H,
                                      int grid_h, int grid_w, int Dk, int Dv, gtr_scan_t scan_order,
                                      gtr_dtype_t dtype, void *out, float *final_state, cudaStream_t stream) {
    // the common checks with q standing in for the unused log_gate; a_low, w2 and the bias are
    // checked below with their own extents
    gtr::Problem p;
    gtr_status_t st = make_problem(q, k, v, q, B, H, grid_h, grid_w, Dk, Dv, scan_order, dtype, out, final_state, &p);
    if (st != GTR_OK) return st;
    if (!(tau > 0.f) || !(tau < 3.0e38f)) return GTR_ERR_INVALID_ARG;  // also rejects NaN
    if (rank < 1) return GTR_ERR_INVALID_ARG;
    if (B == 0 || H == 0) return nothing_launched();
    if (!a_low || !w2 || !gate_bias || !aligned(a_low) || !aligned(w2) || !aligned(gate_bias)) return GTR_ERR_INVALID_ARG;
    const size_t es = elem_size(dtype);
    const size_t na = (size_t)B * p.T * rank * es, nw = (size_t)H * rank * Dk * es, nb = (size_t)H * Dk * 4;
    const size_t nv = (size_t)B * p.T * H * Dv * es, nfs = (size_t)B * H * Dk * Dv * 4;
    const void *extra[3] = {a_low, w2, gate_bias};
    const size_t extra_n[3] = {na, nw, nb};
    for (int i = 0; i < 3; ++i)
        if (overlaps(out, nv, extra[i], extra_n[i]) || overlaps(final_state, nfs, extra[i], extra_n[i]))
            return GTR_ERR_INVALID_ARG;
    if (!gtr::tc_gate_supported(p, rank)) return GTR_ERR_UNSUPPORTED;
    gtr::Ran r;
    const cudaError_t e = gtr::launch_tc_gate(p, gtr::GateSource{a_low, w2, gate_bias, tau}, stream, &r);
    if (e != cudaSuccess) return cuda_fail(e);
    t_last_ran = r;
    return GTR_OK;
}

gtr_status_t gtr_gla_fwd(const void *q, const void *k, const void *v, const void *log_gate, int B,
                         int H, int grid_h, int grid_w, int Dk, int Dv, gtr_scan_t scan_order,
                         gtr_dtype_t dtype, void *out, float *final_state, cudaStream_t stream) {
    return gtr_gla_fwd_sched(q, k, v, log_gate, B, H, grid_h, grid_w, Dk, Dv, scan_order, dtype,
                             out, final_state, GTR_SCHED_AUTO, stream);
}

int gtr_gla_tc_supported(int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                         gtr_scan_t scan_order, gtr_dtype_t dtype) {
    if (check_shape(B, H, grid_h, grid_w, Dk, Dv, scan_order, dtype) != GTR_OK) return 0;
    gtr::Problem p{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, B, H, grid_h, grid_w,
                   Dk, Dv, scan_order, dtype, (long long)grid_h * grid_w};
    return gtr::tc_supported(p) ? 1 : 0;
}

size_t gtr_gla_host_buffer_bytes(int B, int H, int grid_h, int grid_w, int Dk, int Dv,
                                 gtr_dtype_t dtype, int with_final_state) {
    if (check_shape(B, H, grid_h, grid_w, Dk, Dv, 0, dtype) != GTR_OK) return 0;
    const size_t T = (size_t)grid_h * grid_w, es = elem_size(dtype);
    const size_t nk = round_up((size_t)B * T * H * Dk * es, 256);
    const size_t nv = round_up((size_t)B * T * H * Dv * es, 256);
    const size_t nfs = with_final_state ? round_up((size_t)B * H * Dk * Dv * 4, 256) : 0;
    return 3 * nk + 2 * nv + nfs;
}

gtr_status_t gtr_gla_fwd_host(const void *q_host, const void *k_host, const void *v_host,
                              const void *log_gate_host, int B, int H, int grid_h, int grid_w,
                              int Dk, int Dv, gtr_scan_t scan_order, gtr_dtype_t dtype,
                              void *out_host, float *final_state_host, void *dev_buffer,
                              size_t dev_buffer_bytes, cudaStream_t stream) {
    gtr_status_t st = check_shape(B, H, grid_h, grid_w, Dk, Dv, scan_order, dtype);
    if (st != GTR_OK) return st;
    if (!q_host || !k_host || !v_host || !log_gate_host || !out_host) return GTR_ERR_INVALID_ARG;
    const int with_fs = final_state_host != nullptr;
    const size_t need = gtr_gla_host_buffer_bytes(B, H, grid_h, grid_w, Dk, Dv, dtype, with_fs);
    if (dev_buffer == nullptr || dev_buffer_bytes < need) return GTR_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(dev_buffer) % 256) != 0) return GTR_ERR_INVALID_ARG;
    if (B == 0 || H == 0) return nothing_launched();
    const size_t T = (size_t)grid_h * grid_w, es = elem_size(dtype);
    const size_t bk = (size_t)B * T * H * Dk * es, bv = (size_t)B * T * H * Dv * es;
    char *base = static_cast<char *>(dev_buffer);
    char *dq = base, *dk = dq + round_up(bk, 256), *dg = dk + round_up(bk, 256);
    char *dv = dg + round_up(bk, 256), *dout = dv + round_up(bv, 256);
    float *dfs = with_fs ? reinterpret_cast<float *>(dout + round_up(bv, 256)) : nullptr;
    // Batch pieces in a pipeline: piece j's uploads (stream `up`) overlap piece j-1's
    // forward (the caller's stream) and piece j-2's downloads (stream `down`); events
    // fork the two internal streams off the caller's stream and join them back.
    HostPipe *hp = nullptr;
    std::lock_guard<std::mutex> lock(g_pipe_mutex);
    cudaError_t e = host_pipe(&hp);
    if (e != cudaSuccess) return cuda_fail(e);
    const int P = B < kPipePieces ? B : kPipePieces;
    const size_t row_k = T * H * Dk * es, row_v = T * H * Dv * es, row_fs = (size_t)H * Dk * Dv * 4;
    if ((e = cudaEventRecord(hp->fork, stream)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(hp->up, hp->fork, 0)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(hp->down, hp->fork, 0)) != cudaSuccess)
        return cuda_fail(e);
    for (int j = 0; j < P; ++j) {
        const size_t b0 = (size_t)B * j / P, nb = (size_t)B * (j + 1) / P - b0;
        const size_t ok0 = b0 * row_k, ov0 = b0 * row_v, nk = nb * row_k, nvb = nb * row_v;
        if ((e = cudaMemcpyAsync(dq + ok0, static_cast<const char *>(q_host) + ok0, nk, cudaMemcpyHostToDevice, hp->up)) != cudaSuccess ||
            (e = cudaMemcpyAsync(dk + ok0, static_cast<const char *>(k_host) + ok0, nk, cudaMemcpyHostToDevice, hp->up)) != cudaSuccess ||
            (e = cudaMemcpyAsync(dg + ok0, static_cast<const char *>(log_gate_host) + ok0, nk, cudaMemcpyHostToDevice, hp->up)) != cudaSuccess ||
            (e = cudaMemcpyAsync(dv + ov0, static_cast<const char *>(v_host) + ov0, nvb, cudaMemcpyHostToDevice, hp->up)) != cudaSuccess ||
            (e = cudaEventRecord(hp->in[j], hp->up)) != cudaSuccess ||
            (e = cudaStreamWaitEvent(stream, hp->in[j], 0)) != cudaSuccess)
            return cuda_fail(e);
        st = gtr_gla_fwd(dq + ok0, dk + ok0, dv + ov0, dg + ok0, static_cast<int>(nb), H, grid_h, grid_w, Dk, Dv,
                         scan_order, dtype, dout + ov0, with_fs ? dfs + b0 * row_fs / 4 : nullptr, stream);
        if (st != GTR_OK) return st;
        if ((e = cudaEventRecord(hp->done[j], stream)) != cudaSuccess ||
            (e = cudaStreamWaitEvent(hp->down, hp->done[j], 0)) != cudaSuccess ||
            (e = cudaMemcpyAsync(static_cast<char *>(out_host) + ov0, dout + ov0, nvb, cudaMemcpyDeviceToHost, hp->down)) != cudaSuccess)
            return cuda_fail(e);
        if (with_fs && (e = cudaMemcpyAsync(reinterpret_cast<char *>(final_state_host) + b0 * row_fs,
                                            reinterpret_cast<char *>(dfs) + b0 * row_fs, nb * row_fs,
                                            cudaMemcpyDeviceToHost, hp->down)) != cudaSuccess)
            return cuda_fail(e);
    }
    if ((e = cudaEventRecord(hp->join, hp->down)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(stream, hp->join, 0)) != cudaSuccess)
        return cuda_fail(e);
    return GTR_OK;
}

gtr_status_t gtr_gla_sync_status(cudaStream_t stream) {
    cudaError_t e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_fail(e);
    unsigned int word = 0, sw = 0;
    e = gtr::read_and_clear_device_status(&word);
    if (e != cudaSuccess) return cuda_fail(e);
    e = gtr::read_and_clear_sswiglu_status(&sw);
    if (e != cudaSuccess) return cuda_fail(e);
    if ((word | sw) & gtr::kStatusTimeout) return GTR_ERR_TIMEOUT;
    return GTR_OK;
}

gtr_status_t gtr_sswiglu_dwconv(const void *gate, const void *value, long long in_stride, const float *weight,
                                const float *bias, int B, int grid_h, int grid_w, int F, gtr_dtype_t dtype,
                                void *out, cudaStream_t stream) {
    if (dtype < GTR_F32 || dtype > GTR_BF16) return GTR_ERR_INVALID_ARG;
    if (B < 0 || grid_h < 1 || grid_w < 1 || F < 1) return GTR_ERR_INVALID_ARG;
    const long long es = elem_size(dtype), vec = 16 / es;
    const long long T = (long long)grid_h * grid_w;
    if (F % vec != 0 || in_stride < F || (in_stride * es) % 16 != 0) return GTR_ERR_INVALID_ARG;
    if (T > 0x7fffffffLL || (long long)B * T > (1LL << 40) / (in_stride + 1)) return GTR_ERR_INVALID_ARG;
    if (B == 0) return GTR_OK;
    if (!gate || !value || !weight || !out || !aligned(gate) || !aligned(value) || !aligned(out))
        return GTR_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(weight) & 3u) || (bias && (reinterpret_cast<uintptr_t>(bias) & 3u)))
        return GTR_ERR_INVALID_ARG;
    // the output must not overlap the inputs (the convolution reads neighbouring tokens)
    const size_t in_bytes = (size_t)((B * T - 1) * in_stride + F) * es, out_bytes = (size_t)(B * T * F) * es;
    if (overlaps(out, out_bytes, gate, in_bytes) || overlaps(out, out_bytes, value, in_bytes))
        return GTR_ERR_INVALID_ARG;
    gtr::SwProblem p{gate, value, in_stride, weight, bias, out, B, grid_h, grid_w, F, (int)dtype};
    if (!gtr::sswiglu_supported(p)) return GTR_ERR_UNSUPPORTED;
    const cudaError_t e = gtr::launch_sswiglu(p, stream);
    if (e != cudaSuccess) return cuda_fail(e);
    return GTR_OK;
}

const char *gtr_status_string(gtr_status_t status) {
    switch (status) {
    case GTR_OK: return "ok";
    case GTR_ERR_INVALID_ARG: return "invalid argument";
    case GTR_ERR_UNSUPPORTED: return "unsupported by the requested schedule";
    case GTR_ERR_WORKSPACE: return "workspace missing or too small";
    case GTR_ERR_CUDA: return "CUDA error";
    case GTR_ERR_TIMEOUT: return "device-side wait timed out";
    default: return "unknown status";
    }
}

int gtr_last_cuda_error(void) { return t_last_cuda_error; }

gtr_status_t gtr_gla_last_schedule(int *ran, int *planned) {
    if (ran) *ran = t_last_ran.ran;
    if (planned) *planned = t_last_ran.planned;
    return GTR_OK;
}

int gtr_version(void) { return 100; }

}  // extern "C"
