// gla_tc.cu -- tensor-core chunkwise schedule of the GTR token mixer for sm_103a.
//
// Method (Sec. 3.3, Eq. chunk_boundary_main and the chunk-output formula after
// it; chunk size C = 64 as in App. C.3).  For chunk c of a (b, h) sequence, with
// in-chunk scan position r and A_r = sum_{m<=r} g_m (per key channel):
//   o_r      = (q_r . e^{A_r}) S_[c] + sum_{j<=r} (sum_i q_ri k_ji e^{A_ri - A_ji}) v_j
//   U_c      = sum_r (k_r . e^{A_last - A_r})^T v_r,   d_c = e^{A_last}
//   S_[c+1]  = Diag(d_c) S_[c] + U_c
// One CTA walks all chunks of one (b, h) sequence (single pass: every input is
// read once and o, S_final written once; S stays on chip between chunks).
//
// Warp roles (320 threads):
//   warp 0      TMA producer: 8-row boxes of q, k, v, g gathered in scan order
//               (the scan permutation is applied in the box coordinates).
//   warp 1      TMEM allocator + single-thread tcgen05 MMA issuer.
//   warps 2-5   "gen" warpgroup: in-chunk prefix sum of the log-gates (fp32,
//               log2 domain), then the decay-scaled MMA operands.
//   warps 6-9   "epi" warpgroup: reads accumulators from TMEM, applies the
//               causal mask, carries the fp32 state S in registers, converts
//               and stores o through TMA (scatter back to spatial order).
//
// Intra-chunk scores: e^{A_r - A_j} is split at the mid-chunk reference
// A_mid = A_31 as e^{A_r - A_mid} e^{A_mid - A_j}.  Both factors lie within
// 2^{+-M}, M = max_i max(-A_mid, A_mid - A_last) (log2 units); when M <= 100 the
// two scaled operands are exact enough in tf32 and P = Q^ K^^T runs on the tensor
// core (kind::tf32).  Otherwise (extreme decay, e.g. gamma = 0) the chunk's scores
// are computed exactly by the gen warpgroup with per-element exponentials.
// All other operands carry factors <= 1 and are fp16 (kind::f16):
//   U = Kbar^T V   (Kbar = k e^{A_last - A}),  O = Qtil S + P V  (Qtil = q e^{A}).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <mutex>
#include <type_traits>

#include "gla_internal.h"
#include "tc_ptx.cuh"

namespace gtr {

__device__ unsigned int g_device_status;

namespace {

using namespace ptx;

constexpr int kC = 64;                    // chunk length
constexpr int kD = 64;                    // Dk = Dv handled by this kernel
constexpr int kStages = 3;                // input stage ring
constexpr int kTile16 = kC * kD * 2;      // one 64 x 64 16-bit tile (SW128, 128-byte rows)
constexpr int kTile32 = kC * kD * 4;      // one 64 x 64 fp32 tile (two 32-column K-blocks)
constexpr int kThreads = 320;
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // bounded waits give up after 1 s
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kGateMinLog2 = -1.0e4f * 1.4426950408889634f;  // g < -1e4 acts as -1e4
constexpr float kMaxRefExp = 100.0f;      // tf32 score path bound (log2 units)

enum : uint32_t { kModeTF32 = 0, kModeExact = 1 };

// Shared-memory map (byte offsets from a 1024-aligned base).
constexpr int kOffStage = 0;                                   // kStages x {q,k,v,g}
constexpr int kStageBytes = 4 * kTile16;
constexpr int kOffOp = kOffStage + kStages * kStageBytes;      // 2 x {Q^, K^} tf32
constexpr int kOpBytes = 2 * kTile32;
constexpr int kOffS = kOffOp + 2 * kOpBytes;                   // 2 x S (fp16, MN-major)
constexpr int kOffO = kOffS + 2 * kTile16;                     // 2 x O staging
constexpr int kOffDecay = kOffO + 2 * kTile16;                 // kStages x 64 fp32
constexpr int kOffMode = kOffDecay + kStages * kD * 4;         // kStages x u32
constexpr int kOffTot = kOffMode + 64;                         // 2 x 4 x 64 fp32 quarter totals
constexpr int kOffBar = kOffTot + 2 * 4 * kD * 4;              // mbarriers
constexpr int kNumBars = 32;
constexpr int kOffMisc = kOffBar + kNumBars * 8;               // tmem base, abort flag
constexpr int kSmemBytes = kOffMisc + 64 + 1024;               // + alignment slack

// mbarrier indices
enum {
    BAR_FULL = 0,                 // [kStages] TMA -> gen
    BAR_EMPTY = BAR_FULL + kStages,  // [kStages] MMA (O done) -> producer
    BAR_OPND = BAR_EMPTY + kStages,  // [2] gen -> MMA (operands ready)
    BAR_OPFREE = BAR_OPND + 2,       // [2] MMA (P done) -> gen (Q^/K^ buffers free)
    BAR_PFULL = BAR_OPFREE + 2,      // [2] MMA -> epi (P accumulator ready)
    BAR_UFULL = BAR_PFULL + 2,       // [2] MMA -> epi (U accumulator ready)
    BAR_OFULL = BAR_UFULL + 2,       // [2] MMA -> epi (O accumulator ready)
    BAR_PREADY = BAR_OFULL + 2,      // [2] epi -> MMA (masked fp16 P in smem)
    BAR_SREADY = BAR_PREADY + 2,     // [2] epi -> MMA (S_[c] fp16 in smem)
    BAR_TFREE_P = BAR_SREADY + 2,    // [2] epi -> MMA (TMEM P drained)
    BAR_TFREE_U = BAR_TFREE_P + 2,   // [2]
    BAR_TFREE_O = BAR_TFREE_U + 2,   // [2]
    BAR_DONE = BAR_TFREE_O + 2,      // MMA: all issued MMAs completed
    BAR_COUNT
};
static_assert(BAR_COUNT <= kNumBars, "barrier space");

// TMEM columns (fp32 accumulators, M = 64 layout)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColP = 0, kColU = 128, kColO = 256;

struct TmaMaps {
    CUtensorMap q, k, v, g, o;
};

struct TcParams {
    TmaMaps maps;
    float *final_state;
    int H, grid_h, grid_w, order, n_chunks;
    int T;
};

// ---------------------------------------------------------------- small helpers
__device__ __forceinline__ uint32_t sw128(uint32_t row, uint32_t byte) {
    return row * 128u + ((((byte >> 4) ^ (row & 7u)) << 4) | (byte & 15u));
}
// 64 x 64 fp32 tile stored as two K-blocks of 32 columns (8 KB each)
__device__ __forceinline__ uint32_t off32(uint32_t row, uint32_t col) {
    return (col >> 5) * 8192u + sw128(row, (col & 31u) * 4u);
}
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}

template <typename E> struct Pack;
template <> struct Pack<__half> {
    static __device__ __forceinline__ float2 load(const uint8_t *p) {
        return __half22float2(*reinterpret_cast<const __half2 *>(p));
    }
    static __device__ __forceinline__ uint32_t from2(float a, float b) {
        __half2 h = __floats2half2_rn(a, b);
        return *reinterpret_cast<uint32_t *>(&h);
    }
};
template <> struct Pack<__nv_bfloat16> {
    static __device__ __forceinline__ float2 load(const uint8_t *p) {
        return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(p));
    }
    static __device__ __forceinline__ uint32_t from2(float a, float b) {
        __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
        return *reinterpret_cast<uint32_t *>(&h);
    }
};
__device__ __forceinline__ uint32_t half2_bits(float a, float b) {
    __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&h);
}

__device__ __forceinline__ void record_timeout(volatile uint32_t *abort_flag) {
    *abort_flag = 1u;
    atomicOr(&g_device_status, kStatusTimeout);
}

// TMA box coordinates of 8-row group `grp` of chunk `c` (scan positions
// 64c + 8grp .. +7, in smem rows 8grp .. 8grp+7).  Row orders use maps with dims
// (D, H, T, 1, B); column orders (D, H, W, Hg, B).  Reverse orders address the
// reversed range, so smem row rho holds scan position 64c + 63 - rho.  Returns
// false when the whole group lies outside the sequence.
__device__ __forceinline__ bool group_coords(int order, int T, int grid_h, int c, int grp,
                                             int &x2, int &x3) {
    const int rev = order & 1;
    if ((order >> 1) == 0) {  // row orders: token index along dim 2
        int t0 = rev ? (T - kC * (c + 1) + 8 * grp) : (kC * c + 8 * grp);
        x2 = t0;
        x3 = 0;
        return rev ? (t0 + 8 > 0) : (t0 < T);
    }
    // column orders: position u in the top-to-bottom column walk -> (x = u / Hg, y = u % Hg)
    int u0 = rev ? (T - kC * (c + 1) + 8 * grp) : (kC * c + 8 * grp);
    if (u0 < 0 || u0 >= T) {  // entirely outside: point past the last column (zero fill)
        x2 = T / grid_h;
        x3 = 0;
        return false;
    }
    x2 = u0 / grid_h;
    x3 = u0 % grid_h;
    return true;
}

template <typename E>
__global__ void __launch_bounds__(kThreads, 1) gla_tc_kernel(const __grid_constant__ TcParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
    volatile uint32_t *tmem_base_s = reinterpret_cast<volatile uint32_t *>(smem + kOffMisc);
    volatile uint32_t *abort_flag = reinterpret_cast<volatile uint32_t *>(smem + kOffMisc + 4);
    float *decay_s = reinterpret_cast<float *>(smem + kOffDecay);
    volatile uint32_t *mode_s = reinterpret_cast<volatile uint32_t *>(smem + kOffMode);
    float *tot_s = reinterpret_cast<float *>(smem + kOffTot);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int bh = blockIdx.x;
    const int b = bh / p.H, h = bh % p.H;
    const int N = p.n_chunks;
    const int rev = p.order & 1;

    if (threadIdx.x == 0) {
        *abort_flag = 0u;
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&bars[BAR_FULL + i], 1);
            mbar_init(&bars[BAR_EMPTY + i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars[BAR_OPND + i], 4);
            mbar_init(&bars[BAR_OPFREE + i], 1);
            mbar_init(&bars[BAR_PFULL + i], 1);
            mbar_init(&bars[BAR_UFULL + i], 1);
            mbar_init(&bars[BAR_OFULL + i], 1);
            mbar_init(&bars[BAR_PREADY + i], 4);
            mbar_init(&bars[BAR_SREADY + i], 4);
            mbar_init(&bars[BAR_TFREE_P + i], 4);
            mbar_init(&bars[BAR_TFREE_U + i], 4);
            mbar_init(&bars[BAR_TFREE_O + i], 4);
        }
        mbar_init(&bars[BAR_DONE], 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(const_cast<uint32_t *>(tmem_base_s), kTmemCols);
        tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&p.maps.q);
        tma_prefetch_desc(&p.maps.k);
        tma_prefetch_desc(&p.maps.v);
        tma_prefetch_desc(&p.maps.g);
        tma_prefetch_desc(&p.maps.o);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_base_s;

    if (warp == 0) {
        // ======================================================= TMA producer
        if (lane == 0) {
            int issued = 0;
            for (int c = 0; c < N; ++c) {
                const int s = c % kStages;
                if (!mbar_wait(&bars[BAR_EMPTY + s], ((c / kStages) & 1) ^ 1, abort_flag,
                               kWaitLimitNs)) {
                    record_timeout(abort_flag);
                    break;
                }
                uint8_t *st = smem + kOffStage + s * kStageBytes;
                mbar_arrive_expect_tx(&bars[BAR_FULL + s], kStageBytes);
                for (int grp = 0; grp < 8; ++grp) {
                    int x2, x3;
                    group_coords(p.order, p.T, p.grid_h, c, grp, x2, x3);
                    const uint32_t o = grp * 1024;
                    tma_load_5d(st + 0 * kTile16 + o, &p.maps.q, &bars[BAR_FULL + s], 0, h, x2, x3, b);
                    tma_load_5d(st + 1 * kTile16 + o, &p.maps.k, &bars[BAR_FULL + s], 0, h, x2, x3, b);
                    tma_load_5d(st + 2 * kTile16 + o, &p.maps.v, &bars[BAR_FULL + s], 0, h, x2, x3, b);
                    tma_load_5d(st + 3 * kTile16 + o, &p.maps.g, &bars[BAR_FULL + s], 0, h, x2, x3, b);
                }
                ++issued;
            }
            // never leave the CTA while loads are in flight into its shared memory
            if (*abort_flag) {
                for (int c = (issued > kStages ? issued - kStages : 0); c < issued; ++c)
                    mbar_wait(&bars[BAR_FULL + c % kStages], (c / kStages) & 1, nullptr, kWaitLimitNs);
            }
        }
    } else if (warp == 1) {
        // ======================================================= MMA issuer
        if (lane == 0) {
            const uint32_t idesc_p = instr_desc(kFmtTF32, 64, 64, 0, 0);
            const uint32_t idesc_u = instr_desc(kFmtF16, 64, 64, 1, 1);
            const uint32_t idesc_o = instr_desc(kFmtF16, 64, 64, 0, 1);
            const uint32_t sbase = smem_u32(smem);
            bool ok = true;
            auto issue_pu = [&](int c) -> bool {
                const int s = c % kStages, bb = c & 1;
                const uint32_t ph = (c >> 1) & 1;
                if (!mbar_wait(&bars[BAR_OPND + bb], ph, abort_flag, kWaitLimitNs)) return false;
                const uint32_t mode = mode_s[s];
                if (mode == kModeTF32) {
                    if (!mbar_wait(&bars[BAR_TFREE_P + bb], ph ^ 1, abort_flag, kWaitLimitNs)) return false;
                    tc_fence_after();
                    const uint32_t qh = sbase + kOffOp + bb * kOpBytes, kh = qh + kTile32;
                    for (int ks = 0; ks < 8; ++ks) {
                        const uint32_t off = (ks >> 2) * 8192 + (ks & 3) * 32;
                        mma_tf32_ss(tmem + kColP + bb * 64, smem_desc(qh + off, 16, 1024, kLayoutSw128),
                                    smem_desc(kh + off, 16, 1024, kLayoutSw128), idesc_p, ks > 0);
                    }
                    mma_commit(&bars[BAR_PFULL + bb]);
                    mma_commit(&bars[BAR_OPFREE + bb]);
                } else {
                    mbar_arrive(&bars[BAR_PFULL + bb]);
                    mbar_arrive(&bars[BAR_OPFREE + bb]);
                }
                if (!mbar_wait(&bars[BAR_TFREE_U + bb], ph ^ 1, abort_flag, kWaitLimitNs)) return false;
                tc_fence_after();
                const uint32_t st = sbase + kOffStage + s * kStageBytes;
                const uint32_t kb = st + 1 * kTile16, vv = st + 2 * kTile16;
                for (int ks = 0; ks < 4; ++ks) {
                    mma_f16_ss(tmem + kColU + bb * 64, smem_desc(kb + ks * 2048, 8192, 1024, kLayoutSw128),
                               smem_desc(vv + ks * 2048, 8192, 1024, kLayoutSw128), idesc_u, ks > 0);
                }
                mma_commit(&bars[BAR_UFULL + bb]);
                return true;
            };
            if (N > 0) ok = issue_pu(0);
            for (int c = 0; c < N && ok; ++c) {
                if (c + 1 < N && !(ok = issue_pu(c + 1))) break;
                const int s = c % kStages, bb = c & 1;
                const uint32_t ph = (c >> 1) & 1;
                if (!mbar_wait(&bars[BAR_PREADY + bb], ph, abort_flag, kWaitLimitNs) ||
                    !mbar_wait(&bars[BAR_SREADY + bb], ph, abort_flag, kWaitLimitNs) ||
                    !mbar_wait(&bars[BAR_TFREE_O + bb], ph ^ 1, abort_flag, kWaitLimitNs)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t st = sbase + kOffStage + s * kStageBytes;
                const uint32_t qt = st, vv = st + 2 * kTile16, pp = st + 3 * kTile16;
                const uint32_t ss = sbase + kOffS + bb * kTile16;
                const uint32_t dcol = tmem + kColO + bb * 64;
                for (int ks = 0; ks < 4; ++ks)  // O = Qtil S_[c]
                    mma_f16_ss(dcol, smem_desc(qt + ks * 32, 16, 1024, kLayoutSw128),
                               smem_desc(ss + ks * 2048, 8192, 1024, kLayoutSw128), idesc_o, ks > 0);
                for (int ks = 0; ks < 4; ++ks)  // O += P V
                    mma_f16_ss(dcol, smem_desc(pp + ks * 32, 16, 1024, kLayoutSw128),
                               smem_desc(vv + ks * 2048, 8192, 1024, kLayoutSw128), idesc_o, 1);
                mma_commit(&bars[BAR_OFULL + bb]);
                mma_commit(&bars[BAR_EMPTY + s]);
            }
            if (!ok) record_timeout(abort_flag);
            // all MMAs this thread issued must finish before TMEM is released
            mma_commit(&bars[BAR_DONE]);
            mbar_wait(&bars[BAR_DONE], 0, nullptr, kWaitLimitNs);
        }
    } else if (warp < 6) {
        // ======================================================= gen warpgroup
        const int tq = warp - 2;          // scan positions 16 tq .. 16 tq + 15
        const int ch = 2 * lane;          // key channels ch, ch + 1
        const int tg = threadIdx.x - 64;  // 0..127
        for (int c = 0; c < N; ++c) {
            const int s = c % kStages, bb = c & 1;
            if (!mbar_wait(&bars[BAR_FULL + s], (c / kStages) & 1, abort_flag, kWaitLimitNs) ||
                !mbar_wait(&bars[BAR_OPFREE + bb], ((c >> 1) & 1) ^ 1, abort_flag, kWaitLimitNs)) {
                record_timeout(abort_flag);
                break;
            }
            uint8_t *st = smem + kOffStage + s * kStageBytes;
            uint8_t *tq_ = st, *tk = st + kTile16, *tv = st + 2 * kTile16, *tgate = st + 3 * kTile16;
            // -- in-chunk cumulative log-decay (log2 units), Sec. 3.3: A_r = sum_{m<=r} g_m
            float2 a[16];
            float2 run = make_float2(0.f, 0.f);
#pragma unroll
            for (int t = 0; t < 16; ++t) {
                const int r = 16 * tq + t;
                const int rho = rev ? 63 - r : r;
                float2 g2 = Pack<E>::load(tgate + sw128(rho, ch * 2));
                float x = g2.x * kLog2e, y = g2.y * kLog2e;
                x = x < kGateMinLog2 ? kGateMinLog2 : x;
                y = y < kGateMinLog2 ? kGateMinLog2 : y;
                run.x += x;
                run.y += y;
                a[t] = run;
            }
            float *tot = tot_s + bb * 4 * kD;  // double-buffered: chunk c+1 may write while c is read
            *reinterpret_cast<float2 *>(tot + tq * kD + ch) = run;
            named_barrier_sync(1, 128);
            float2 off = make_float2(0.f, 0.f), amid, alast;
            {
                const float2 t0 = *reinterpret_cast<const float2 *>(tot + 0 * kD + ch);
                const float2 t1 = *reinterpret_cast<const float2 *>(tot + 1 * kD + ch);
                const float2 t2 = *reinterpret_cast<const float2 *>(tot + 2 * kD + ch);
                const float2 t3 = *reinterpret_cast<const float2 *>(tot + 3 * kD + ch);
                if (tq > 0) { off.x += t0.x; off.y += t0.y; }
                if (tq > 1) { off.x += t1.x; off.y += t1.y; }
                if (tq > 2) { off.x += t2.x; off.y += t2.y; }
                amid = make_float2(t0.x + t1.x, t0.y + t1.y);
                alast = make_float2(amid.x + t2.x + t3.x, amid.y + t2.y + t3.y);
            }
#pragma unroll
            for (int t = 0; t < 16; ++t) { a[t].x += off.x; a[t].y += off.y; }
            // -- score-path selection: largest |exponent| of the mid-chunk split
            float m = fmaxf(fmaxf(-amid.x, amid.x - alast.x), fmaxf(-amid.y, amid.y - alast.y));
            if (m != m) m = 1e30f;  // NaN gates: exact path (propagates NaN)
            const uint32_t mbits = __reduce_max_sync(0xffffffffu, __float_as_uint(fmaxf(m, 0.f)));
            const uint32_t mode = (__uint_as_float(mbits) <= kMaxRefExp) ? kModeTF32 : kModeExact;
            if (tq == 3) {
                decay_s[s * kD + ch] = ex2(alast.x);
                decay_s[s * kD + ch + 1] = ex2(alast.y);
            }
            if (tg == 0) mode_s[s] = mode;
            if (mode == kModeTF32) {
                uint8_t *qh = smem + kOffOp + bb * kOpBytes, *kh = qh + kTile32;
                const float c1x = ex2(amid.x), c1y = ex2(amid.y);                    // <= 1
                const float c2x = ex2(alast.x - amid.x), c2y = ex2(alast.y - amid.y);  // <= 1
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    const int r = 16 * tq + t;
                    const int rho = rev ? 63 - r : r;
                    const float ex = a[t].x - amid.x, ey = a[t].y - amid.y;
                    const float fqx = ex2(ex), fqy = ex2(ey), fkx = ex2(-ex), fky = ex2(-ey);
                    const uint32_t o16 = sw128(rho, ch * 2);
                    const float2 q2 = Pack<E>::load(tq_ + o16);
                    const float2 k2 = Pack<E>::load(tk + o16);
                    const float qx = q2.x * fqx, qy = q2.y * fqy, kx = k2.x * fkx, ky = k2.y * fky;
                    *reinterpret_cast<float2 *>(qh + off32(rho, ch)) = make_float2(to_tf32(qx), to_tf32(qy));
                    *reinterpret_cast<float2 *>(kh + off32(rho, ch)) = make_float2(to_tf32(kx), to_tf32(ky));
                    *reinterpret_cast<uint32_t *>(tq_ + o16) = half2_bits(qx * c1x, qy * c1y);
                    *reinterpret_cast<uint32_t *>(tk + o16) = half2_bits(kx * c2x, ky * c2y);
                }
            } else {
                // exact scores: P[rho][sigma] = sum_i q_i k_i 2^{a_r,i - a_j,i} for j <= r
                float *as = reinterpret_cast<float *>(smem + kOffOp + bb * kOpBytes);  // [64][64] by rho
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    const int r = 16 * tq + t;
                    const int rho = rev ? 63 - r : r;
                    *reinterpret_cast<float2 *>(as + rho * kD + ch) = a[t];
                }
                named_barrier_sync(1, 128);
                {
                    const int rho = tg >> 1, half = tg & 1;
                    const int r = rev ? 63 - rho : rho;
                    uint32_t packed[16];
                    for (int jj = 0; jj < 32; jj += 2) {
                        float pv[2];
                        for (int u = 0; u < 2; ++u) {
                            const int sig = half * 32 + jj + u;
                            const int j = rev ? 63 - sig : sig;
                            float acc = 0.f;
                            if (j <= r) {
                                for (int i = 0; i < kD; i += 2) {
                                    const float2 qi = Pack<E>::load(tq_ + sw128(rho, i * 2));
                                    const float2 ki = Pack<E>::load(tk + sw128(sig, i * 2));
                                    acc += qi.x * ki.x * ex2(as[rho * kD + i] - as[sig * kD + i]);
                                    acc += qi.y * ki.y * ex2(as[rho * kD + i + 1] - as[sig * kD + i + 1]);
                                }
                            }
                            pv[u] = acc;
                        }
                        packed[jj >> 1] = half2_bits(pv[0], pv[1]);
                    }
                    for (int jj = 0; jj < 16; ++jj)
                        *reinterpret_cast<uint32_t *>(tgate + sw128(rho, (half * 32 + 2 * jj) * 2)) = packed[jj];
                }
                named_barrier_sync(1, 128);
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    const int r = 16 * tq + t;
                    const int rho = rev ? 63 - r : r;
                    const uint32_t o16 = sw128(rho, ch * 2);
                    const float2 q2 = Pack<E>::load(tq_ + o16);
                    const float2 k2 = Pack<E>::load(tk + o16);
                    *reinterpret_cast<uint32_t *>(tq_ + o16) =
                        half2_bits(q2.x * ex2(a[t].x), q2.y * ex2(a[t].y));
                    *reinterpret_cast<uint32_t *>(tk + o16) =
                        half2_bits(k2.x * ex2(alast.x - a[t].x), k2.y * ex2(alast.y - a[t].y));
                }
            }
            // bf16 inputs: values become fp16 MMA operands (exact for |v| in the fp16 normal range)
            if constexpr (std::is_same<E, __nv_bfloat16>::value) {
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    uint4 *pv = reinterpret_cast<uint4 *>(tv) + tg * 4 + u;
                    uint4 w = *pv;
                    uint32_t *wp = reinterpret_cast<uint32_t *>(&w);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 f = __bfloat1622float2(*reinterpret_cast<__nv_bfloat162 *>(&wp[e]));
                        wp[e] = half2_bits(f.x, f.y);
                    }
                    *pv = w;
                }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_OPND + bb]);
        }
    } else {
        // ======================================================= epi warpgroup
        const int qd = warp & 3;                     // TMEM sub-partition of this warp
        const bool has_row = lane < 16;              // M = 64 layout: 16 rows per sub-partition
        const int row = qd * 16 + (lane & 15);       // accumulator row (token rho or channel i)
        const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
        const bool elected = (warp == 6 && lane == 0);
        float S[kD];
#pragma unroll
        for (int j = 0; j < kD; ++j) S[j] = 0.f;
        // S_[0] = 0
        {
            const int te = threadIdx.x - 192;
            uint4 z = make_uint4(0, 0, 0, 0);
            for (int i = te; i < kTile16 / 16; i += 128)
                reinterpret_cast<uint4 *>(smem + kOffS)[i] = z;
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_SREADY + 0]);
        }
        bool ok = true;
        for (int c = 0; c < N; ++c) {
            const int s = c % kStages, bb = c & 1;
            const uint32_t ph = (c >> 1) & 1;
            uint8_t *st = smem + kOffStage + s * kStageBytes;
            if (!mbar_wait(&bars[BAR_PFULL + bb], ph, abort_flag, kWaitLimitNs)) { ok = false; break; }
            const uint32_t mode = mode_s[s];
            const float dc = decay_s[s * kD + row];
            if (mode == kModeTF32) {
                tc_fence_after();
                uint8_t *pt = st + 3 * kTile16;
#pragma unroll
                for (int cb = 0; cb < 4; ++cb) {
                    uint32_t r[16];
                    tmem_ld_32x32b_x16(tmem + lane_base + kColP + bb * 64 + cb * 16, r);
                    tmem_ld_wait();
                    if (has_row) {
                        uint32_t w[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            const int s0 = cb * 16 + 2 * e;
                            const bool k0 = rev ? (s0 >= row) : (s0 <= row);
                            const bool k1 = rev ? (s0 + 1 >= row) : (s0 + 1 <= row);
                            w[e] = half2_bits(k0 ? __uint_as_float(r[2 * e]) : 0.f,
                                              k1 ? __uint_as_float(r[2 * e + 1]) : 0.f);
                        }
                        *reinterpret_cast<uint4 *>(pt + sw128(row, cb * 32)) = make_uint4(w[0], w[1], w[2], w[3]);
                        *reinterpret_cast<uint4 *>(pt + sw128(row, cb * 32 + 16)) = make_uint4(w[4], w[5], w[6], w[7]);
                    }
                }
            }
            // arrived every chunk (also when the exact path skipped the P accumulator)
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_TFREE_P + bb]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_PREADY + bb]);
            // -- state carry: S_[c+1] = Diag(d_c) S_[c] + U_c
            if (!mbar_wait(&bars[BAR_UFULL + bb], ph, abort_flag, kWaitLimitNs)) { ok = false; break; }
            tc_fence_after();
#pragma unroll
            for (int cb = 0; cb < 4; ++cb) {
                uint32_t r[16];
                tmem_ld_32x32b_x16(tmem + lane_base + kColU + bb * 64 + cb * 16, r);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 16; ++e) S[cb * 16 + e] = fmaf(dc, S[cb * 16 + e], __uint_as_float(r[e]));
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_TFREE_U + bb]);
            if (c + 1 < N) {
                uint8_t *sb = smem + kOffS + ((c + 1) & 1) * kTile16;
                if (has_row) {
#pragma unroll
                    for (int cb = 0; cb < 8; ++cb) {
                        uint32_t w[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) w[e] = half2_bits(S[cb * 8 + 2 * e], S[cb * 8 + 2 * e + 1]);
                        *reinterpret_cast<uint4 *>(sb + sw128(row, cb * 16)) = make_uint4(w[0], w[1], w[2], w[3]);
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&bars[BAR_SREADY + ((c + 1) & 1)]);
            }
            // -- output: TMEM -> dtype -> smem -> TMA store in spatial order
            if (!mbar_wait(&bars[BAR_OFULL + bb], ph, abort_flag, kWaitLimitNs)) { ok = false; break; }
            if (elected) tma_store_wait_read<1>();
            named_barrier_sync(2, 128);
            tc_fence_after();
            uint8_t *ob = smem + kOffO + bb * kTile16;
#pragma unroll
            for (int cb = 0; cb < 4; ++cb) {
                uint32_t r[16];
                tmem_ld_32x32b_x16(tmem + lane_base + kColO + bb * 64 + cb * 16, r);
                tmem_ld_wait();
                if (has_row) {
                    uint32_t w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        w[e] = Pack<E>::from2(__uint_as_float(r[2 * e]), __uint_as_float(r[2 * e + 1]));
                    *reinterpret_cast<uint4 *>(ob + sw128(row, cb * 32)) = make_uint4(w[0], w[1], w[2], w[3]);
                    *reinterpret_cast<uint4 *>(ob + sw128(row, cb * 32 + 16)) = make_uint4(w[4], w[5], w[6], w[7]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_TFREE_O + bb]);
            fence_proxy_async_smem();
            named_barrier_sync(2, 128);
            if (elected) {
                for (int grp = 0; grp < 8; ++grp) {
                    int x2, x3;
                    if (group_coords(p.order, p.T, p.grid_h, c, grp, x2, x3))
                        tma_store_5d(&p.maps.o, ob + grp * 1024, 0, h, x2, x3, b);
                }
                tma_store_commit();
            }
        }
        if (!ok) record_timeout(abort_flag);
        if (ok && p.final_state != nullptr && has_row) {
            float4 *dst = reinterpret_cast<float4 *>(p.final_state + ((size_t)bh * kD + row) * kD);
#pragma unroll
            for (int j = 0; j < kD / 4; ++j) dst[j] = make_float4(S[4 * j], S[4 * j + 1], S[4 * j + 2], S[4 * j + 3]);
        }
        if (elected) tma_store_wait_all<0>();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void *f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}

// dims (D, H, T, 1, B) for row orders, (D, H, W, Hg, B) for column orders; box 8 rows.
bool encode_map(CUtensorMap *m, const void *ptr, int dtype, const Problem &p, int D) {
    auto enc = get_encode();
    if (!enc) return false;
    const cuuint64_t es = 2;
    const bool col = (p.order >> 1) != 0;
    cuuint64_t dims[5], strides[4];
    cuuint32_t box[5], estr[5] = {1, 1, 1, 1, 1};
    dims[0] = D;
    dims[1] = p.H;
    strides[0] = (cuuint64_t)D * es;
    strides[1] = (cuuint64_t)p.H * D * es;
    if (!col) {
        dims[2] = p.T;
        dims[3] = 1;
        strides[2] = (cuuint64_t)p.T * p.H * D * es;
        box[2] = 8;
        box[3] = 1;
    } else {
        dims[2] = p.grid_w;
        dims[3] = p.grid_h;
        strides[2] = (cuuint64_t)p.grid_w * p.H * D * es;
        box[2] = 1;
        box[3] = 8;
    }
    dims[4] = p.B;
    strides[3] = (cuuint64_t)p.T * p.H * D * es;
    box[0] = 64;
    box[1] = 1;
    box[4] = 1;
    const CUtensorMapDataType dt =
        dtype == 1 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    CUresult r = enc(m, dt, 5, const_cast<void *>(ptr), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace

bool tc_supported(const Problem &p) {
    if (p.dtype != 1 && p.dtype != 2) return false;      // fp16 / bf16 operands only
    if (p.Dk != kD || p.Dv != kD) return false;
    if (p.T % 8 != 0) return false;                       // 8-row boxes never straddle the end
    if ((p.order >> 1) != 0 && p.grid_h % 8 != 0) return false;  // 8-row groups inside one column
    if (p.T > (1 << 30)) return false;
    return get_encode() != nullptr;
}

cudaError_t launch_tc(const Problem &p, cudaStream_t stream) {
    TcParams tp;
    if (!encode_map(&tp.maps.q, p.q, p.dtype, p, kD) || !encode_map(&tp.maps.k, p.k, p.dtype, p, kD) ||
        !encode_map(&tp.maps.v, p.v, p.dtype, p, kD) || !encode_map(&tp.maps.g, p.g, p.dtype, p, kD) ||
        !encode_map(&tp.maps.o, p.out, p.dtype, p, kD))
        return cudaErrorInvalidValue;
    tp.final_state = p.final_state;
    tp.H = p.H;
    tp.grid_h = p.grid_h;
    tp.grid_w = p.grid_w;
    tp.order = p.order;
    tp.T = static_cast<int>(p.T);
    tp.n_chunks = static_cast<int>((p.T + kC - 1) / kC);
    const dim3 grid(static_cast<unsigned>(p.B * p.H));
    cudaError_t e;
    if (p.dtype == 1) {
        e = cudaFuncSetAttribute(gla_tc_kernel<__half>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
        if (e != cudaSuccess) return e;
        gla_tc_kernel<__half><<<grid, kThreads, kSmemBytes, stream>>>(tp);
    } else {
        e = cudaFuncSetAttribute(gla_tc_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemBytes);
        if (e != cudaSuccess) return e;
        gla_tc_kernel<__nv_bfloat16><<<grid, kThreads, kSmemBytes, stream>>>(tp);
    }
    return cudaGetLastError();
}

cudaError_t read_and_clear_device_status(unsigned int *status) {
    cudaError_t e = cudaMemcpyFromSymbol(status, g_device_status, sizeof(unsigned int));
    if (e != cudaSuccess) return e;
    const unsigned int zero = 0;
    return cudaMemcpyToSymbol(g_device_status, &zero, sizeof(unsigned int));
}

}  // namespace gtr
