// sswiglu.cu -- Spatial SwiGLU between its two projections (Sec. 3.1, Eq.
// spatial_swiglu): Z = SiLU(X W_g) * DWConv3x3(X W_v) on the patch grid, the
// step the deployed S-SwiGLU kernel fuses (Sec. 4).
//
// Memory-bound: per token it reads F gate and F value elements and writes F
// outputs.  Work is cut into tiles of R grid rows x one 128-byte channel slice
// (64 channels at 16 bits, 32 at fp32) of one image, one CTA of 256 threads per
// tile, two CTAs per SM (up to 108 KB of shared memory each), so that one CTA's
// TMA loads overlap the other's arithmetic.  (A persistent CTA per SM with two
// stages, or two persistent CTAs per SM, measured 3-29 % slower on a GB300: a
// CTA-wide barrier per tile idles its warps.)  A tile's value box covers rows
// y0-1 .. y0+R and columns -1 .. W of the slice: it starts at -1 on both grid
// axes and runs one past the last row and column, where the tensor map returns
// zeros, which is exactly the convolution's zero padding; the gate box covers the
// tile's own tokens.  Each thread owns one 8-byte channel group (4 channels at 16
// bits, 2 at fp32; its 9 taps and bias in registers) and walks strips of 4 rows
// down one column of the tile with the 3 x 3 window of values in registers: per
// output row it reads one new tile row of three values and the gate from shared
// memory, accumulates in fp32 and stores 8 bytes.  (The window cut the
// instructions per output element by about a third against re-reading all nine
// values per token: 1.40x faster on GTR-L at 640^2, 1.13x on GTR-X at 1280^2, with
// identical output bits.)  Neighbouring row tiles re-read their halo rows, which L2
// serves.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <atomic>
#include <cstdint>
#include <cstring>

#include "gla_internal.h"
#include "tc_ptx.cuh"

namespace gtr {

__device__ unsigned int g_sswiglu_status;

namespace {

using namespace ptx;

constexpr int kSwThreads = 256;
constexpr int kSwStageBudget = 108 * 1024;        // a tile's boxes (two CTAs per SM)
constexpr int kSwSmemBudget = 2 * kSwStageBudget;  // wide grids: one CTA per SM
constexpr int kSwMaxRows = 32;
constexpr uint64_t kSwWaitNs = 1000000000ull;     // 1 s: a tile's copies never take that long

struct SwParams {
    CUtensorMap vmap;       // value tensor: dims (F, W, Hg, B), box (slice, W + 2, rows + 2, 1)
    CUtensorMap gmap;       // gate tensor: same dims, box (slice, W, rows, 1)
    void *out;
    const float *weight;
    const float *bias;
    int grid_h, grid_w, F, rows, ntile_y, ntile_f, ntiles;
    uint32_t vbytes, gbytes;  // bytes of the value box and of the gate box
};

struct TilePos {
    int f0, y0, b;
};
template <int SLICE>
__device__ __forceinline__ TilePos tile_pos(const SwParams &p, int t) {
    const int tf = t % p.ntile_f, rest = t / p.ntile_f;
    return {tf * SLICE, (rest % p.ntile_y) * p.rows, rest / p.ntile_y};
}

// TMA loads of the CTA's tile (one thread): the value box with its halo, then the
// gate box.  Always inlined: the tensor maps are addressed in the kernel's
// parameter space.
__device__ __forceinline__ void issue_tile(const SwParams &p, uint8_t *smem, uint64_t *full, const TilePos &tp) {
    mbar_arrive_expect_tx(full, p.vbytes + p.gbytes);
    tma_load_4d(smem, &p.vmap, full, tp.f0, -1, tp.y0 - 1, tp.b);
    tma_load_4d(smem + p.vbytes, &p.gmap, full, tp.f0, 0, tp.y0, tp.b);
}

template <typename E> struct Vec8;
template <> struct Vec8<float> {
    static constexpr int n = 2;
    static __device__ __forceinline__ void unpack(uint2 q, float (&v)[2]) {
        v[0] = __uint_as_float(q.x);
        v[1] = __uint_as_float(q.y);
    }
    static __device__ __forceinline__ uint2 pack(const float (&v)[2]) {
        return make_uint2(__float_as_uint(v[0]), __float_as_uint(v[1]));
    }
};
template <> struct Vec8<__half> {
    static constexpr int n = 4;
    static __device__ __forceinline__ void unpack(uint2 q, float (&v)[4]) {
        const float2 a = __half22float2(*reinterpret_cast<const __half2 *>(&q.x));
        const float2 b = __half22float2(*reinterpret_cast<const __half2 *>(&q.y));
        v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
    }
    static __device__ __forceinline__ uint2 pack(const float (&v)[4]) {
        const __half2 a = __floats2half2_rn(v[0], v[1]), b = __floats2half2_rn(v[2], v[3]);
        return make_uint2(*reinterpret_cast<const uint32_t *>(&a), *reinterpret_cast<const uint32_t *>(&b));
    }
};
template <> struct Vec8<__nv_bfloat16> {
    static constexpr int n = 4;
    static __device__ __forceinline__ void unpack(uint2 q, float (&v)[4]) {
        v[0] = __uint_as_float(q.x << 16); v[1] = __uint_as_float(q.x & 0xFFFF0000u);
        v[2] = __uint_as_float(q.y << 16); v[3] = __uint_as_float(q.y & 0xFFFF0000u);
    }
    static __device__ __forceinline__ uint2 pack(const float (&v)[4]) {
        const __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
        return make_uint2(*reinterpret_cast<const uint32_t *>(&a), *reinterpret_cast<const uint32_t *>(&b));
    }
};

template <typename E>
__global__ void __launch_bounds__(kSwThreads, 2) sswiglu_kernel(const __grid_constant__ SwParams p) {
    constexpr int N = Vec8<E>::n;           // elements per 8 bytes
    constexpr int SLICE = 16 * N;           // channels per tile: 128 bytes, sixteen groups
    constexpr int RB = 4;                   // rows per strip piece
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
    __shared__ uint64_t full;
    const int W = p.grid_w;
    // one tile per CTA (the grid has one CTA per tile)
    const TilePos tp = tile_pos<SLICE>(p, static_cast<int>(blockIdx.x));
    if (threadIdx.x == 0) {
        mbar_init(&full, 1);
        fence_mbar_init();
        issue_tile(p, smem, &full, tp);
    }
    __syncthreads();
    const int cg = static_cast<int>(threadIdx.x & 15u);
    E *out = static_cast<E *>(p.out);
    const long long T = (long long)p.grid_h * W;
    {
        const int fc = tp.f0 + cg * N;
        const bool live = fc < p.F;
        const int R = p.grid_h - tp.y0 < p.rows ? p.grid_h - tp.y0 : p.rows;
        float w[9][N], bs[N];
#pragma unroll
        for (int e = 0; e < N; ++e) {
#pragma unroll
            for (int q = 0; q < 9; ++q) w[q][e] = live ? p.weight[(size_t)(fc + e) * 9 + q] : 0.f;
            bs[e] = (live && p.bias != nullptr) ? p.bias[fc + e] : 0.f;
        }
        const bool ok = mbar_wait(&full, 0, nullptr, kSwWaitNs);
        if (__syncthreads_or(!ok)) {
            if (threadIdx.x == 0) {  // never leave while the copies may still land
                atomicOr(&g_sswiglu_status, kStatusTimeout);
                mbar_wait(&full, 0, nullptr, kSwWaitNs);
            }
            __syncthreads();
            return;
        }
        const uint8_t *vt = smem;
        const uint8_t *gt = vt + p.vbytes;
        const int nrb = (R + RB - 1) / RB;
        // items: (column x, row block) pairs; each walks RB rows down its column with a
        // 3 x 3 window of values in registers (one new tile row of 3 values per output row)
        for (int it = static_cast<int>(threadIdx.x >> 4); it < W * nrb; it += kSwThreads / 16) {
            const int x = it % W, r0 = (it / W) * RB;
            float win[3][3][N];
#pragma unroll
            for (int i = 0; i < 2; ++i)
#pragma unroll
                for (int j = 0; j < 3; ++j)
                    Vec8<E>::unpack(*reinterpret_cast<const uint2 *>(
                                        vt + ((size_t)(r0 + i) * (W + 2) + (x + j)) * 128 + cg * 8),
                                    win[i][j]);
#pragma unroll
            for (int rr = 0; rr < RB; ++rr) {
                const int r = r0 + rr;
                if (r >= R) break;
                // tile rows r, r + 1, r + 2 sit in window slots rr % 3, (rr + 1) % 3, (rr + 2) % 3
#pragma unroll
                for (int j = 0; j < 3; ++j)
                    Vec8<E>::unpack(*reinterpret_cast<const uint2 *>(
                                        vt + ((size_t)(r + 2) * (W + 2) + (x + j)) * 128 + cg * 8),
                                    win[(rr + 2) % 3][j]);
                float acc[N];
#pragma unroll
                for (int e = 0; e < N; ++e) acc[e] = bs[e];
#pragma unroll
                for (int i = 0; i < 3; ++i)
#pragma unroll
                    for (int j = 0; j < 3; ++j)
#pragma unroll
                        for (int e = 0; e < N; ++e) acc[e] = fmaf(w[3 * i + j][e], win[(rr + i) % 3][j][e], acc[e]);
                if (live) {
                    float g[N], z[N];
                    Vec8<E>::unpack(*reinterpret_cast<const uint2 *>(gt + ((size_t)r * W + x) * 128 + cg * 8), g);
#pragma unroll
                    for (int e = 0; e < N; ++e) z[e] = __fdividef(g[e], 1.f + __expf(-g[e])) * acc[e];
                    const long long tok = (long long)tp.b * T + (long long)(tp.y0 + r) * W + x;
                    *reinterpret_cast<uint2 *>(out + tok * p.F + fc) = Vec8<E>::pack(z);
                }
            }
        }
    }
}

int elem_bytes(int dtype) { return dtype == 0 ? 4 : 2; }

// Shared memory of one stage for `rows` grid rows: the value box (rows + 2) x (W + 2)
// and the gate box rows x W, 128 bytes a token.
size_t stage_bytes(int rows, int W) { return 128u * ((size_t)(rows + 2) * (W + 2) + (size_t)rows * W); }

// Rows per tile: the most rows (up to kSwMaxRows and the grid's height) whose boxes
// fit kSwStageBudget (two CTAs per SM), else, for grids too wide for one row there,
// kSwSmemBudget (one CTA per SM); 0 when not even one row fits.
int tile_rows(const SwProblem &p) {
    for (int pass = 0; pass < 2; ++pass) {
        const size_t budget = pass == 0 ? kSwStageBudget : kSwSmemBudget;
        int r = 0;
        while (r < kSwMaxRows && r < p.grid_h && stage_bytes(r + 1, p.grid_w) <= budget) ++r;
        if (r >= 1) return r;
    }
    return 0;
}

template <typename E>
cudaError_t launch_typed(const SwParams &sp, unsigned grid, size_t smem, cudaStream_t stream) {
    static std::atomic<unsigned long long> set_on_devices(0);
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(set_on_devices.load(std::memory_order_relaxed) & bit)) {
        e = cudaFuncSetAttribute(sswiglu_kernel<E>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSwSmemBudget + 256));
        if (e != cudaSuccess) return e;
        set_on_devices.fetch_or(bit);
    }
    sswiglu_kernel<E><<<grid, kSwThreads, smem, stream>>>(sp);
    return cudaGetLastError();
}

bool encode(CUtensorMap *m, const SwProblem &p, const void *base, int box_w, int box_h) {
    auto enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensor_map_encoder());
    if (!enc) return false;
    const int es = elem_bytes(p.dtype);
    const cuuint64_t row = static_cast<cuuint64_t>(p.in_stride) * es;
    const cuuint64_t T = static_cast<cuuint64_t>(p.grid_h) * p.grid_w;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(p.F), static_cast<cuuint64_t>(p.grid_w),
                          static_cast<cuuint64_t>(p.grid_h), static_cast<cuuint64_t>(p.B)};
    cuuint64_t strides[3] = {row, row * p.grid_w, row * T};
    cuuint32_t box[4] = {static_cast<cuuint32_t>(128 / es), static_cast<cuuint32_t>(box_w),
                         static_cast<cuuint32_t>(box_h), 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUtensorMapDataType dt = p.dtype == 0 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
                                   : p.dtype == 1 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                                  : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    return enc(m, dt, 4, const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool sswiglu_supported(const SwProblem &p) {
    // the value box spans the grid width plus the halo in one TMA dimension (at most
    // 256 elements), and a stage of at least one row must fit the shared memory
    return p.grid_w + 2 <= 256 && tile_rows(p) >= 1 && tensor_map_encoder() != nullptr;
}

cudaError_t launch_sswiglu(const SwProblem &p, cudaStream_t stream) {
    if (!sswiglu_supported(p)) return cudaErrorInvalidValue;
    const int slice = 128 / elem_bytes(p.dtype);
    SwParams sp;
    std::memset(&sp, 0, sizeof(sp));
    sp.rows = tile_rows(p);
    sp.out = p.out;
    sp.weight = p.weight;
    sp.bias = p.bias;
    sp.grid_h = p.grid_h;
    sp.grid_w = p.grid_w;
    sp.F = p.F;
    sp.ntile_y = (p.grid_h + sp.rows - 1) / sp.rows;
    sp.ntile_f = (p.F + slice - 1) / slice;
    const long long tiles = (long long)p.B * sp.ntile_y * sp.ntile_f;
    if (tiles <= 0 || tiles > 0x7fffffffLL) return cudaErrorInvalidValue;
    sp.ntiles = static_cast<int>(tiles);
    sp.vbytes = static_cast<uint32_t>(128u * (size_t)(sp.rows + 2) * (p.grid_w + 2));
    sp.gbytes = static_cast<uint32_t>(128u * (size_t)sp.rows * p.grid_w);
    if (!encode(&sp.vmap, p, p.value, p.grid_w + 2, sp.rows + 2) || !encode(&sp.gmap, p, p.gate, p.grid_w, sp.rows))
        return cudaErrorInvalidValue;
    const unsigned grid = static_cast<unsigned>(tiles);  // one CTA per tile
    const size_t smem = (size_t)sp.vbytes + sp.gbytes + 128;
    if (p.dtype == 0) return launch_typed<float>(sp, grid, smem, stream);
    if (p.dtype == 1) return launch_typed<__half>(sp, grid, smem, stream);
    return launch_typed<__nv_bfloat16>(sp, grid, smem, stream);
}

cudaError_t read_and_clear_sswiglu_status(unsigned int *status) {
    cudaError_t e = cudaMemcpyFromSymbol(status, g_sswiglu_status, sizeof(unsigned int));
    if (e != cudaSuccess) return e;
    const unsigned int zero = 0;
    return cudaMemcpyToSymbol(g_sswiglu_status, &zero, sizeof(unsigned int));
}

}  // namespace gtr
