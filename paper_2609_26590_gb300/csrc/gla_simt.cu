// gla_simt.cu -- plain fp32 CUDA-core token recurrence.
//
// Sec. 3.1 ("Key-only gated recurrence"): S_t = Diag(gamma_t) S_{t-1} + k_t^T v_t,
// o_t = q_t S_t, walked token by token along the scan order of Sec. 3.1
// ("Directional scanning").  This is the float32 path (the tensor-core schedule
// cannot hold a 1e-5 relative error) and the path for shapes the tensor-core
// schedule does not take.
//
// Mapping: one CTA of 256 threads per (b, h, block of 16 value columns).  Thread
// (r, j) owns column j of S over the r-th sixteenth of the Dk rows in registers, so
// the state update is thread-local and the readout o_t[j] = sum_i q_t[i] S[i][j] is
// sixteen partial sums, added after every block of 16 tokens through shared memory
// (one barrier per block, not per token); the per-token chain of a thread is short
// (2 to 8 rows), which is what bounds this latency-bound recurrence.  q_t, k_t, gamma_t and v_t of the next
// block are loaded into registers while the current block runs, then staged in
// shared memory and read as broadcasts.  The permutation is applied when loading
// (gather) and when storing o_t (scatter back to the spatial position).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "gla_internal.h"

namespace gtr {
namespace {

constexpr int kTok = 16;       // tokens staged per block
constexpr int kCols = 16;      // value columns per CTA
constexpr int kGroups = 16;    // row groups of S per column
constexpr int kSimtThreads = kCols * kGroups;

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__half x) { return __half2float(x); }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __half from_f32<__half>(float x) { return __float2half_rn(x); }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

// Spatial token visited at scan position s (Sec. 3.1 "Directional scanning").
__device__ __forceinline__ long long scan_token(int order, long long gh, long long gw,
                                                long long T, long long s) {
    switch (order) {
    case 0: return s;
    case 1: return T - 1 - s;
    case 2: return (s % gh) * gw + s / gh;
    default: {
        long long u = T - 1 - s;
        return (u % gh) * gw + u / gh;
    }
    }
}

template <int DKM, typename E>
__global__ void __launch_bounds__(kSimtThreads) gla_simt_kernel(Problem p) {
    constexpr int RPT = DKM / kGroups;                 // rows of S per thread
    constexpr int NQ = kTok * DKM / kSimtThreads;      // staged q / k / gamma values per thread
    constexpr int NV = kTok * kCols / kSimtThreads;    // staged v values per thread
    __shared__ __align__(16) float sq[kTok][DKM];
    __shared__ __align__(16) float sk[kTok][DKM];
    __shared__ __align__(16) float sgam[kTok][DKM];
    __shared__ float sv[kTok][kCols];
    __shared__ float po[kGroups][kTok][kCols];          // partial readouts of the block
    __shared__ long long stok[kTok];

    const int bh = blockIdx.x;
    const int b = bh / p.H, h = bh % p.H;
    const int c0 = blockIdx.y * kCols;
    const int tid = threadIdx.x;
    const int cj = tid % kCols, grp = tid / kCols;     // column and row quarter owned
    const long long T = p.T;
    const int Dk = p.Dk, Dv = p.Dv, H = p.H;
    const E *q = static_cast<const E *>(p.q);
    const E *k = static_cast<const E *>(p.k);
    const E *v = static_cast<const E *>(p.v);
    const E *g = static_cast<const E *>(p.g);
    E *out = static_cast<E *>(p.out);

    // one block's inputs in registers (zeros / gamma = 1 past the sequence and past Dk, Dv:
    // padding contributes nothing)
    float rq[NQ], rk[NQ], rg[NQ], rv[NV];
    long long rt = 0;
    auto load_block = [&](long long s0) {
        const int n = (int)((T - s0) < kTok ? (T - s0) : kTok);
#pragma unroll
        for (int m = 0; m < NQ; ++m) {
            const int idx = tid + m * kSimtThreads, j = idx / DKM, i = idx % DKM;
            float qv = 0.f, kv = 0.f, gam = 1.f;
            if (j < n && i < Dk) {
                const long long off = (((long long)b * T + scan_token(p.order, p.grid_h, p.grid_w, T, s0 + j)) * H + h) * Dk + i;
                qv = to_f32(q[off]);
                kv = to_f32(k[off]);
                float lg = to_f32(g[off]);
                lg = lg < -1.0e4f ? -1.0e4f : lg;  // gamma = 0 below -1e4; NaN stays NaN
                gam = expf(lg);
            }
            rq[m] = qv;
            rk[m] = kv;
            rg[m] = gam;
        }
#pragma unroll
        for (int m = 0; m < NV; ++m) {
            const int idx = tid + m * kSimtThreads, j = idx / kCols, c = idx % kCols;
            float vv = 0.f;
            if (j < n && c0 + c < Dv)
                vv = to_f32(v[(((long long)b * T + scan_token(p.order, p.grid_h, p.grid_w, T, s0 + j)) * H + h) * Dv + c0 + c]);
            rv[m] = vv;
        }
        rt = tid < n ? scan_token(p.order, p.grid_h, p.grid_w, T, s0 + tid) : 0;
    };

    float S[RPT];
#pragma unroll
    for (int i = 0; i < RPT; ++i) S[i] = 0.f;

    load_block(0);
    for (long long s0 = 0; s0 < T; s0 += kTok) {
        const int n = (int)((T - s0) < kTok ? (T - s0) : kTok);
        __syncthreads();  // the previous block's shared values and partials are consumed
#pragma unroll
        for (int m = 0; m < NQ; ++m) {
            const int idx = tid + m * kSimtThreads;
            sq[idx / DKM][idx % DKM] = rq[m];
            sk[idx / DKM][idx % DKM] = rk[m];
            sgam[idx / DKM][idx % DKM] = rg[m];
        }
#pragma unroll
        for (int m = 0; m < NV; ++m) {
            const int idx = tid + m * kSimtThreads;
            sv[idx / kCols][idx % kCols] = rv[m];
        }
        if (tid < kTok) stok[tid] = rt;
        __syncthreads();
        if (s0 + kTok < T) load_block(s0 + kTok);  // in flight while this block runs
        for (int j = 0; j < n; ++j) {
            const float vj = sv[j][cj];
            float o0 = 0.f, o1 = 0.f;
#pragma unroll
            for (int i = 0; i < RPT; i += 2) {
                const int r = grp * RPT + i;
                S[i] = fmaf(sgam[j][r], S[i], sk[j][r] * vj);
                S[i + 1] = fmaf(sgam[j][r + 1], S[i + 1], sk[j][r + 1] * vj);
                o0 = fmaf(sq[j][r], S[i], o0);
                o1 = fmaf(sq[j][r + 1], S[i + 1], o1);
            }
            po[grp][j][cj] = o0 + o1;
        }
        __syncthreads();
        // the block's outputs: sum over the row groups, scattered to the spatial tokens
        for (int idx = tid; idx < n * kCols; idx += kSimtThreads) {
            const int j = idx / kCols, c = idx % kCols;
            if (c0 + c < Dv) {
                float o = 0.f;
#pragma unroll
                for (int r = 0; r < kGroups; ++r) o += po[r][j][c];
                out[(((long long)b * T + stok[j]) * H + h) * Dv + c0 + c] = from_f32<E>(o);
            }
        }
    }
    const int col = c0 + cj;
    if (p.final_state != nullptr && col < Dv) {
        float *fs = p.final_state + ((long long)b * H + h) * Dk * Dv;
#pragma unroll
        for (int i = 0; i < RPT; ++i)
            if (grp * RPT + i < Dk) fs[(long long)(grp * RPT + i) * Dv + col] = S[i];
    }
}

template <typename T>
cudaError_t launch_typed(const Problem &p, cudaStream_t stream) {
    dim3 grid((unsigned)(p.B * p.H), (unsigned)((p.Dv + kCols - 1) / kCols));
    if (p.Dk <= 32) {
        gla_simt_kernel<32, T><<<grid, kSimtThreads, 0, stream>>>(p);
    } else if (p.Dk <= 64) {
        gla_simt_kernel<64, T><<<grid, kSimtThreads, 0, stream>>>(p);
    } else {
        gla_simt_kernel<128, T><<<grid, kSimtThreads, 0, stream>>>(p);
    }
    return cudaGetLastError();
}

// Output gate of Sec. 3.1 applied in place: one warp per (token, head) row of
// Dv <= 128 outputs; lane j takes columns j, j + 32, j + 64, j + 96.
template <typename E>
__global__ void __launch_bounds__(256) gate_epilogue_kernel(E *out, const E *r, const float *w, float eps,
                                                            long long rows, int Dv) {
    const long long row = static_cast<long long>(blockIdx.x) * 8 + (threadIdx.x >> 5);
    if (row >= rows) return;
    const int lane = threadIdx.x & 31;
    E *o_row = out + row * Dv;
    const E *r_row = r + row * Dv;
    float o[4];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int col = lane + 32 * i;
        o[i] = col < Dv ? to_f32(o_row[col]) : 0.f;
        ss += o[i] * o[i];
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, m);
    const float inv = rsqrtf(ss / static_cast<float>(Dv) + eps);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int col = lane + 32 * i;
        if (col < Dv) {
            const float z = to_f32(r_row[col]);
            const float silu = __fdividef(z, 1.f + __expf(-z));
            o_row[col] = from_f32<E>(silu * o[i] * inv * w[col]);
        }
    }
}

// The same gate for 16-byte vectors: LPR = Dv / VEC lanes per row, each moving
// VEC = 16 / sizeof(E) contiguous values (coalesced 16-byte loads and stores).
template <typename E, int LPR>
__global__ void __launch_bounds__(256) gate_epilogue_vec_kernel(E *out, const E *r, const float *w, float eps,
                                                                long long rows) {
    constexpr int VEC = 16 / static_cast<int>(sizeof(E));
    constexpr int Dv = LPR * VEC;
    const long long gid = static_cast<long long>(blockIdx.x) * 256 + threadIdx.x;
    const long long row = gid / LPR;
    const int part = static_cast<int>(gid % LPR);
    const bool live = row < rows;
    const size_t off = static_cast<size_t>(live ? row : 0) * Dv + static_cast<size_t>(part) * VEC;
    uint4 ov = live ? *reinterpret_cast<const uint4 *>(out + off) : make_uint4(0u, 0u, 0u, 0u);
    const uint4 rv = live ? *reinterpret_cast<const uint4 *>(r + off) : make_uint4(0u, 0u, 0u, 0u);
    const E *oe = reinterpret_cast<const E *>(&ov);
    const E *re = reinterpret_cast<const E *>(&rv);
    float o[VEC];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
        o[i] = to_f32(oe[i]);
        ss += o[i] * o[i];
    }
#pragma unroll
    for (int m = LPR / 2; m >= 1; m >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, m);
    const float inv = rsqrtf(ss / static_cast<float>(Dv) + eps);
    uint4 uv;
    E *ue = reinterpret_cast<E *>(&uv);
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
        const float z = to_f32(re[i]);
        ue[i] = from_f32<E>(__fdividef(z, 1.f + __expf(-z)) * o[i] * inv * w[part * VEC + i]);
    }
    if (live) *reinterpret_cast<uint4 *>(out + off) = uv;
}

template <typename E, int LPR>
cudaError_t launch_gate_vec(E *out, const E *r, const float *w, float eps, long long rows, cudaStream_t stream) {
    const long long blocks = (rows * LPR + 255) / 256;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
    gate_epilogue_vec_kernel<E, LPR><<<static_cast<unsigned>(blocks), 256, 0, stream>>>(out, r, w, eps, rows);
    return cudaGetLastError();
}

template <typename E>
cudaError_t launch_gate_typed(const Problem &p, const Gate &gate, cudaStream_t stream) {
    const long long rows = static_cast<long long>(p.B) * p.T * p.H;
    E *out = static_cast<E *>(p.out);
    const E *r = static_cast<const E *>(gate.r);
    constexpr int VEC = 16 / static_cast<int>(sizeof(E));
    // rows of a 16-byte-multiple width take the vector kernel (row starts stay 16-byte aligned)
    switch (p.Dv % VEC == 0 ? p.Dv / VEC : 0) {
    case 1: return launch_gate_vec<E, 1>(out, r, gate.w, gate.eps, rows, stream);
    case 2: return launch_gate_vec<E, 2>(out, r, gate.w, gate.eps, rows, stream);
    case 4: return launch_gate_vec<E, 4>(out, r, gate.w, gate.eps, rows, stream);
    case 8: return launch_gate_vec<E, 8>(out, r, gate.w, gate.eps, rows, stream);
    case 16: return launch_gate_vec<E, 16>(out, r, gate.w, gate.eps, rows, stream);
    case 32: return launch_gate_vec<E, 32>(out, r, gate.w, gate.eps, rows, stream);
    default: break;
    }
    const long long blocks = (rows + 7) / 8;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
    gate_epilogue_kernel<E><<<static_cast<unsigned>(blocks), 256, 0, stream>>>(out, r, gate.w, gate.eps, rows, p.Dv);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gate_epilogue(const Problem &p, const Gate &gate, cudaStream_t stream) {
    if (p.dtype == 0) return launch_gate_typed<float>(p, gate, stream);
    if (p.dtype == 1) return launch_gate_typed<__half>(p, gate, stream);
    return launch_gate_typed<__nv_bfloat16>(p, gate, stream);
}

cudaError_t launch_simt(const Problem &p, cudaStream_t stream) {
    switch (p.dtype) {
    case 0: return launch_typed<float>(p, stream);
    case 1: return launch_typed<__half>(p, stream);
    default: return launch_typed<__nv_bfloat16>(p, stream);
    }
}

}  // namespace gtr
