// gla_simt.cu -- plain fp32 CUDA-core token recurrence.
//
// Sec. 3.1 ("Key-only gated recurrence"): S_t = Diag(gamma_t) S_{t-1} + k_t^T v_t,
// o_t = q_t S_t, walked token by token along the scan order of Sec. 3.1
// ("Directional scanning").  This is the float32 path (the tensor-core schedule
// cannot hold a 1e-5 relative error) and the path for shapes the tensor-core
// schedule does not take.
//
// Mapping: one CTA of 64 threads per (b, h, block of 64 value columns).  Thread
// j owns column j of S (all Dk rows) in registers, so the state update and the
// readout o_t[j] = sum_i q_t[i] S[i][j] are thread-local; q_t, k_t and gamma_t
// are staged in shared memory for 16 tokens at a time and read as broadcasts.
// The permutation is applied when staging (gather) and when storing o_t
// (scatter back to the spatial position).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "gla_internal.h"

namespace gtr {
namespace {

constexpr int kTok = 16;    // tokens staged per step
constexpr int kCols = 64;   // value columns per CTA (= threads per CTA)

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
__global__ void __launch_bounds__(kCols) gla_simt_kernel(Problem p) {
    __shared__ __align__(16) float sq[kTok][DKM];
    __shared__ __align__(16) float sk[kTok][DKM];
    __shared__ __align__(16) float sgam[kTok][DKM];
    __shared__ float sv[kTok][kCols];
    __shared__ long long stok[kTok];

    const int bh = blockIdx.x;
    const int b = bh / p.H, h = bh % p.H;
    const int c0 = blockIdx.y * kCols;
    const int tid = threadIdx.x;
    const int col = c0 + tid;
    const long long T = p.T;
    const int Dk = p.Dk, Dv = p.Dv, H = p.H;
    const E *q = static_cast<const E *>(p.q);
    const E *k = static_cast<const E *>(p.k);
    const E *v = static_cast<const E *>(p.v);
    const E *g = static_cast<const E *>(p.g);
    E *out = static_cast<E *>(p.out);

    float S[DKM];
#pragma unroll
    for (int i = 0; i < DKM; ++i) S[i] = 0.f;

    for (long long s0 = 0; s0 < T; s0 += kTok) {
        const int n = (int)((T - s0) < kTok ? (T - s0) : kTok);
        __syncthreads();  // readers of the previous step are done
        if (tid < kTok) stok[tid] = tid < n ? scan_token(p.order, p.grid_h, p.grid_w, T, s0 + tid) : 0;
        __syncthreads();
        for (int idx = tid; idx < kTok * DKM; idx += kCols) {
            const int j = idx / DKM, i = idx % DKM;
            float qv = 0.f, kv = 0.f, gam = 1.f;  // padding rows/channels contribute nothing
            if (j < n && i < Dk) {
                const long long off = (((long long)b * T + stok[j]) * H + h) * Dk + i;
                qv = to_f32(q[off]);
                kv = to_f32(k[off]);
                float lg = to_f32(g[off]);
                lg = lg < -1.0e4f ? -1.0e4f : lg;  // gamma = 0 below -1e4; NaN stays NaN
                gam = expf(lg);
            }
            sq[j][i] = qv;
            sk[j][i] = kv;
            sgam[j][i] = gam;
        }
        for (int idx = tid; idx < kTok * kCols; idx += kCols) {
            const int j = idx / kCols, c = idx % kCols;
            float vv = 0.f;
            if (j < n && c0 + c < Dv) vv = to_f32(v[(((long long)b * T + stok[j]) * H + h) * Dv + c0 + c]);
            sv[j][c] = vv;
        }
        __syncthreads();
        for (int j = 0; j < n; ++j) {
            const float vj = sv[j][tid];
            float o = 0.f;
#pragma unroll
            for (int i = 0; i < DKM; ++i) {
                S[i] = fmaf(sgam[j][i], S[i], sk[j][i] * vj);
                o = fmaf(sq[j][i], S[i], o);
            }
            if (col < Dv) out[(((long long)b * T + stok[j]) * H + h) * Dv + col] = from_f32<E>(o);
        }
    }
    if (p.final_state != nullptr && col < Dv) {
        float *fs = p.final_state + ((long long)b * H + h) * Dk * Dv;
#pragma unroll
        for (int i = 0; i < DKM; ++i)
            if (i < Dk) fs[(long long)i * Dv + col] = S[i];
    }
}

template <typename T>
cudaError_t launch_typed(const Problem &p, cudaStream_t stream) {
    dim3 grid((unsigned)(p.B * p.H), (unsigned)((p.Dv + kCols - 1) / kCols));
    if (p.Dk <= 32) {
        gla_simt_kernel<32, T><<<grid, kCols, 0, stream>>>(p);
    } else if (p.Dk <= 64) {
        gla_simt_kernel<64, T><<<grid, kCols, 0, stream>>>(p);
    } else {
        gla_simt_kernel<128, T><<<grid, kCols, 0, stream>>>(p);
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_simt(const Problem &p, cudaStream_t stream) {
    switch (p.dtype) {
    case 0: return launch_typed<float>(p, stream);
    case 1: return launch_typed<__half>(p, stream);
    default: return launch_typed<__nv_bfloat16>(p, stream);
    }
}

}  // namespace gtr
