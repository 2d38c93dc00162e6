// gla_tc.cu -- tensor-core chunkwise schedule of the GTR token mixer for sm_103a.
//
// Method (Sec. 3.3, Eq. chunk_boundary_main and the chunk-output formula after
// it; chunk size C = 64 as in App. C.3).  For chunk c of a (b, h) sequence, with
// in-chunk scan position r and A_r = sum_{m<=r} g_m (per key channel):
//   o_r      = (q_r . e^{A_r}) S_[c] + sum_{j<=r} (sum_i q_ri k_ji e^{A_ri - A_ji}) v_j
//   U_c      = sum_r (k_r . e^{A_last - A_r})^T v_r,   d_c = e^{A_last}
//   S_[c+1]  = Diag(d_c) S_[c] + U_c
// A persistent CTA per SM walks all chunks of its (b, h) sequences as one stream
// (single pass: q, k, v, g are read once, o and S_final written once; S stays on
// chip between chunks, and the pipeline does not drain between sequences).
//
// Per chunk, tensor-core products (tcgen05.mma, fp32 accumulators in TMEM):
//   A = L G          in-chunk cumulative log-decay: L is the 64x64 triangle of
//                    ones in scan order, G the gate tile as loaded (exact products)
//   P = Q^ K^^T      intra-chunk scores with e^{A_r - A_j} split at the mid-chunk
//                    reference: Q^ = q e^{A_r - A_mid}, K^ = k e^{A_mid - A_j}
//   U = Kbar^T V     chunk summary, Kbar = k e^{A_last - A}
//   O = Qtil S_[c] + P V   outputs, Qtil = q e^{A}
// The split factors of P lie within 2^{+-M}, M = max_i max(-A_mid, A_mid - A_last)
// (log2 units).  M <= 8 ("fp16 mode"): Q^, K^ are fp16 and serve all products,
// because the per-channel constants c1 = e^{A_mid}, c2 = e^{A_last - A_mid} fold
// into the state: Qtil S = Q^ (Diag(c1) S) and Kbar^T V = Diag(c2) K^^T V.
// M <= 100 ("tf32 mode"): Q^, K^ are tf32 (fp32 range) for P, and Qtil, Kbar are
// written as fp16 operands.  Larger M or non-finite gates ("exact mode"): the
// chunk's log-decays and scores are computed exactly by CUDA cores.
//
// Memory: each chunk owns a 32 KB stage slot (q, k, v, g tiles) from its TMA
// load until its output product completes; the derived fp16 operands are
// written in place (Q^ or Qtil over q, K^ or Kbar over k, the masked scores P
// over g, bf16 v converted to fp16 in place), so four chunks can be in flight.
// Only the tf32 score operands use separate buffers, one per gen warpgroup, so
// that tf32-mode chunks of the two groups never wait for each other.  Row orders
// load one 64-row TMA box per tensor and chunk; column orders one im2col load per
// tensor (a map whose fastest spatial dimension is the grid row, so 64 pixels run
// down a column and on into the next).  Chunks that reach past either end of the
// sequence load one box per column segment instead, of the segment's exact height (a
// tensor map per height), and zero-fill boxes for the rows outside.  The scan
// permutation lives in the load coordinates and in the addresses of the output stores.
//
// Warp roles (512 threads, one CTA per SM; four warps per SM sub-partition, so a
// thread keeps 128 registers).  Few roles with small loops keep the hot code
// inside the SM's instruction cache:
//   warp 0       TMA producer.
//   warp 1       TMEM allocator and issuer of A(c) = L G.
//   warps 2-5    gen warpgroup 0 (even chunks): reads A, builds the operands of its
//                chunk, then masks the chunk's scores P into fp16.
//   warps 6-9    gen warpgroup 1 (odd chunks).
//   warps 10-13  epi: carries the fp32 state S in registers, writes Diag(c1) S,
//                and stores each chunk's outputs at the tokens' spatial positions
//                (GENOUT launches: the gen warpgroup that built the chunk stores them).
//   warp 14      issuer of P(c) and U(c).
//   warp 15      issuer of O(c).
// Each issuer waits only for the inputs of its own product, so the issue overhead
// of one product does not hold up the others.
// A warp reads the TMEM lanes of sub-partition (warp % 4); an M = 64 accumulator
// keeps rows 16q..16q+15 in lanes 32q..32q+15, and each thread takes one row and
// 32 of its 64 columns.
//
// Few, long sequences are split into segments (MODE kSummary computes each
// segment's end state from zero and its total decay, MODE kSplitFull starts every
// segment from the fold of the earlier ones); the last segment may run past the
// sequence over all-zero padding chunks, which leave the state unchanged.  When the
// units outnumber the SMs unevenly (MODE kBalanced), every CTA takes an equal
// contiguous range of the units' chunks: the head of the unit its range ends in comes
// first and hands its end state to the next CTA through global memory, the tail of
// the unit its range starts in comes last, from the state the CTA before handed over.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <atomic>
#include <chrono>
#include <cstdlib>
#include <cstring>
#include <list>
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
constexpr int kSlots = 4;                 // stage slots (chunks in flight)
constexpr int kTile16 = kC * kD * 2;      // 64 x 64 16-bit tile (SW128, 128-byte rows)
constexpr int kTile32 = kC * kD * 4;      // 64 x 64 fp32 tile (two 32-column K-blocks)
constexpr int kThreads = 512;
constexpr int kHeights = 15;              // TMA box heights 1 .. 7, then 8, 16, ..., 64
// Rows of the TMA box of height index hi (one tensor map per height).
__host__ __device__ constexpr int box_height(int hi) { return hi < 7 ? hi + 1 : 8 * (hi - 6); }
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // bounded waits give up after 1 s
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kGateMinLog2 = -1.0e4f * 1.4426950408889634f;  // g < -1e4 acts as -1e4
constexpr float kMaxRefF16 = 8.0f;        // fp16 score operands: factors within 2^{+-8}
constexpr float kMaxRefTF32 = 100.0f;     // tf32 score operands: factors within 2^{+-100}

enum : uint32_t { kModeF16 = 0, kModeTF32 = 1, kModeExact = 2 };
// Kernel passes: kFull (sequences whole, dealt round-robin), kSplitFull (outputs of
// segments that start from the fold of the earlier segments' summaries), kSummary (the
// summaries), kBalanced (equal contiguous chunk ranges per CTA, the state of a unit cut
// by a range boundary handed from one CTA to the next; one key half).
enum : int { kFull = 0, kSplitFull = 1, kSummary = 2, kBalanced = 3 };
constexpr int kMinSegChunks = 2;          // a split segment keeps at least this many chunks
constexpr int kMaxUnsplitChunks = 5;      // shorter sequences are never split
constexpr uint32_t kBarSin = 4;           // named barrier: epi read the folded start state (ids 1-3: gen groups, epi)

// Shared-memory map (byte offsets from a 1024-aligned base).
constexpr int kSlotBytes = 4 * kTile16;                        // q @0, k @8K, v @16K, g @24K
constexpr int kQ = 0, kK = kTile16, kV = 2 * kTile16, kG = 3 * kTile16;
constexpr int kOffSlot = 0;
constexpr int kOffOp = kOffSlot + kSlots * kSlotBytes;         // per gen group g @32K g: tf32 Q^ @0, K^ @16K
constexpr int kOffS = kOffOp + 4 * kTile32;                    // 2 x S'_[c] (fp16, MN-major)
constexpr int kOffL = kOffS + 2 * kTile16;                     // triangle of ones
constexpr int kRank = 16;                                      // rank r of the gate's low-rank projection
constexpr int kW2Bytes = kRank * kD * 2;                       // a head's W2 block: r x 64 channels, 16-bit
constexpr int kOffW2 = kOffL + kTile16;                        // gate producer: 2 x W2 (by unit parity)
constexpr int kRefFloats = 4 * kD;                             // raw A_mid, raw A_last, c1, c2
constexpr int kOffRef = kOffW2 + 2 * kW2Bytes;                 // per slot
constexpr int kOffDecay = kOffRef + kSlots * kRefFloats * 4;   // per slot, 64 fp32
constexpr int kOffMode = kOffDecay + kSlots * kD * 4;          // per slot u32 mode; 2 x 2 fp32 maxima
constexpr int kOffBar = kOffMode + 64;
constexpr int kNumBars = 40;
constexpr int kOffMisc = kOffBar + kNumBars * 8;               // tmem base, abort flag
constexpr int kSmemBytes = kOffMisc + 64 + 1024;               // + alignment slack
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

enum {
    BAR_FULL = 0,                      // [kSlots] TMA -> issuer (A)
    BAR_EMPTY = BAR_FULL + kSlots,     // [kSlots] U(c) and O(c) done (two commits) -> producer
    BAR_REFS = BAR_EMPTY + kSlots,     // [kSlots] gen -> epi: chunk constants and mode
    BAR_AFULL = BAR_REFS + kSlots,     // [2] A done -> gen
    BAR_PURDY = BAR_AFULL + 2,         // [2] P/U(c) may go: gen(c) operands in smem and A(c) read
                                       //     (4 arrivals) + epi drained U(c-2) (4 arrivals)
    BAR_PFULL = BAR_PURDY + 2,         // [2] P done -> gen
    BAR_UFULL = BAR_PFULL + 2,         // [2] U done -> epi
    BAR_ORDY = BAR_UFULL + 2,          // [2] O(c) may go: gen(c) masked P in smem and TMEM P read
                                       //     (4) + epi wrote Diag(c1) S_[c] and read O(c-2) (4)
    BAR_OFULL = BAR_ORDY + 2,          // [2] O of a virtual chunk done -> epi
    BAR_ZFULL = BAR_OFULL + 2,         // [2] gate producer: Z = a W2 done -> gen
    BAR_GRDY = BAR_ZFULL + 2,          // [2] gate producer: gates G written by the gen group (4) -> A issuer
    BAR_DONE = BAR_GRDY + 2,           // every MMA completed (teardown)
    BAR_COUNT = BAR_DONE + 1
};
static_assert(BAR_COUNT <= kNumBars, "barrier space");

constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColA = 0, kColP = 128, kColU = 256, kColO = 384;

enum { T_Q = 0, T_K = 1, T_V = 2, T_G = 3, kTensors = 4 };

// Division by a launch constant 1 <= d < 2^31 of 0 <= n < 2^31 by a multiply-high and a
// shift (Granlund and Montgomery, "Division by invariant integers using multiplication",
// 1994, Thm. 4.2): with l = ceil(log2 d) and m = floor(2^32 (2^l - d) / d) + 1, the 33-bit
// multiplier 2^32 + m satisfies 2^(32+l) < (2^32 + m) d <= 2^(32+l) + 2^l, so
// n / d = (umulhi(n, m) + n) >> l, the sum exact in 32 bits for n < 2^31.  A few
// instructions instead of an integer division's sequence: every role's per-chunk index
// arithmetic uses it, which keeps the kernel's hot code small (the SM's instruction cache
// is shared by all roles; the divisions of one decode cost a balanced launch 17 %).
struct FastDiv {
    int d;
    uint32_t m, l;
};
inline FastDiv make_fastdiv(int d) {
    if (d < 1) d = 1;
    uint32_t l = 0;
    while ((1ull << l) < static_cast<unsigned long long>(d)) ++l;
    return FastDiv{d, static_cast<uint32_t>(((1ull << 32) * ((1ull << l) - d)) / d + 1), l};
}
__host__ __device__ __forceinline__ int fdiv(int n, const FastDiv &f) {
#ifdef __CUDA_ARCH__
    const uint32_t hi = __umulhi(static_cast<uint32_t>(n), f.m);
#else
    const uint32_t hi = static_cast<uint32_t>((static_cast<uint64_t>(static_cast<uint32_t>(n)) * f.m) >> 32);
#endif
    return static_cast<int>((hi + static_cast<uint32_t>(n)) >> f.l);
}

struct TcParams {
    CUtensorMap maps[kTensors][kHeights];  // box height box_height(i)
    CUtensorMap cmaps[kTensors];           // column orders: a chunk's 64-token walk as one im2col load
    void *out;
    float *final_state;
    int H, grid_h, grid_w, order, n_chunks, T;
    int Dk, Dv;                            // multiples of 8 up to 128 (the tensors' row widths)
    int nh;                                // ceil(Dk / 64): 64-channel key halves per chunk
    int nv;                                // ceil(Dv / 64): 64-column value slices, one per CTA work unit
    int n_units;                           // work units of this launch, dealt out round-robin to the CTAs
    int seg_len;                           // chunks per segment (the last one may run past the sequence)
    int nseg;                              // segments per sequence (1: no split)
    int nsu;                               // segments per (sequence, value slice) among this launch's units
    float *summary;                        // nseg > 1: per (sequence, segment < nseg - 1) end state from zero
                                           // [Dk][Dv] and total decay [Dk], fp32
    int drop_load;                         // test hook: CTA 0 withholds its first chunk's load, so the
                                           // bounded waits run out and the call reports a timeout
    unsigned long long *flags;             // kBalanced: per CTA, == epoch once its hand-off state (in
                                           // summary, [64][64] fp32 per CTA) is written; cleared when read
    unsigned long long epoch;              // kBalanced: nonzero, new for every launch
    FastDiv fd_per, fd_nsu, fd_H, fd_gh, fd_L;  // division by L * nh, nsu, H, grid_h, L
    FastDiv bal_n;                         // kBalanced: division by the chunks per sequence
    // gate producer (maps[T_G] then load the rank-16 projection a = x W1 instead of the gates)
    CUtensorMap w2map;                     // W2 [H][r][Dk], 16-bit, box (64 channels, r rows) SW128
    const float *gbias;                    // b [H][Dk] fp32
    float tau_inv;                         // 1 / tau
    // output gate fused into the gen warpgroups' stores (GATED): u = SiLU(r) RMSNorm(o) w
    const void *gate_r;                    // r = x W_r [B][T][H][Dv], the input dtype
    const float *gate_w;                   // RMSNorm weight [Dv]
    float gate_eps;
};

// ---------------------------------------------------------------- helpers
__device__ __forceinline__ uint32_t sw128(uint32_t row, uint32_t byte) {
    return row * 128u + ((((byte >> 4) ^ (row & 7u)) << 4) | (byte & 15u));
}
__device__ __forceinline__ uint32_t off32(uint32_t row, uint32_t col) {
    return (col >> 5) * 8192u + sw128(row, (col & 31u) * 4u);
}
// SW128 operand descriptors: K-major tiles (8-row groups 1024 B apart) and
// MN-major tiles (64-element atoms 8192 B apart).  A K step of 16 elements adds
// 32 B (2 in the address field) to a K-major descriptor and 2048 B (128) to an
// MN-major one.
__device__ __forceinline__ uint64_t kdesc(uint32_t saddr) { return smem_desc(saddr, 16, 1024, kLayoutSw128); }
__device__ __forceinline__ uint64_t mndesc(uint32_t saddr) { return smem_desc(saddr, 8192, 1024, kLayoutSw128); }
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// log sigma(x) = min(x, 0) - log(1 + e), e = e^{-|x|} in (0, 1]: log(1 + e) by the fast
// logarithm (absolute error below 2^-21 on [1, 2]), or by its series e - e^2 / 2 where e < 1e-3
// (error below e^3 / 3), so that the relative error stays below 4e-4 before the gate is
// rounded to fp16.  NaN propagates; x = +inf gives 0, x = -inf gives -inf.
__device__ __forceinline__ float log_sigmoid(float x) {
    const float e = ex2(-fabsf(x) * kLog2e);
    const float l1p = e < 1.0e-3f ? e * fmaf(-0.5f, e, 1.f) : __logf(1.f + e);
    return fminf(x, 0.f) - l1p;
}
__device__ __forceinline__ float to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}
__device__ __forceinline__ uint32_t h2bits(float a, float b) {
    __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&h);
}

template <typename E> struct Elem;
template <> struct Elem<__half> {
    static constexpr uint32_t fmt = kFmtF16;
    static constexpr uint16_t one = 0x3C00;
    static __device__ __forceinline__ float2 unpack(uint32_t w) {
        return __half22float2(*reinterpret_cast<const __half2 *>(&w));
    }
    static __device__ __forceinline__ uint32_t pack(float a, float b) { return h2bits(a, b); }
};
template <> struct Elem<__nv_bfloat16> {
    static constexpr uint32_t fmt = kFmtBF16;
    static constexpr uint16_t one = 0x3F80;
    static __device__ __forceinline__ float2 unpack(uint32_t w) {
        return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w));
    }
    static __device__ __forceinline__ uint32_t pack(float a, float b) {
        __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
        return *reinterpret_cast<uint32_t *>(&h);
    }
};

__device__ __forceinline__ void record_timeout(volatile uint32_t *abort_flag) {
    *abort_flag = 1u;
    atomicOr(&g_device_status, kStatusTimeout);
}

// Smem row rho of chunk c holds walk position w0 + rho, where the walk is the
// forward scan (row-major for row orders, down the columns for column orders)
// and w0 mirrors the range for reverse orders (scan position 64c + 63 - rho).
__host__ __device__ __forceinline__ int chunk_w0(int order, int T, int c) {
    return (order & 1) ? (T - kC * (c + 1)) : kC * c;
}

// Work units are (sequence, 64-column value slice) pairs.  A CTA walks the units
// blockIdx.x, blockIdx.x + gridDim.x, ... as one stream of "virtual chunks": each
// 64-token chunk of a unit appears once per 64-channel key half (Dk = 128: twice),
// carrying that half's q, k, g and the unit's v slice.  The output is linear in the
// key channels (o = sum over halves of Qtil_a S_a + P_a V), so the halves go through
// the same per-chunk pipeline and only their O products share one accumulator.
struct StreamPos {
    int bh;      // sequence b * H + h
    int vb;      // value slice
    int c;       // chunk of the sequence
    int a;       // key half
    int seg;     // segment of the sequence
    int cl;      // chunk within the segment
    bool start;  // a run of the unit starts here: its state is set
    bool hin;    // kBalanced: the run starts from the previous CTA's hand-off state
};
// Units are (sequence, segment, value slice), the value slice fastest (the two
// slices of a sequence read the same q, k and gates); a unit covers seg_len chunks.
__device__ __forceinline__ StreamPos stream_pos(int v, int L, int nh, int lognv, const FastDiv &per, bool split,
                                                const FastDiv &nsu) {
    const int j = fdiv(v, per), rem = v - j * per.d;
    const int unit = static_cast<int>(blockIdx.x) + j * static_cast<int>(gridDim.x);
    const int rest = unit >> lognv;
    const int bh = split ? fdiv(rest, nsu) : rest;
    const int seg = split ? rest - bh * nsu.d : 0;
    const int cl = rem / nh;
    const int a = rem - cl * nh;
    return {bh, unit & ((1 << lognv) - 1), seg * L + cl, a, seg, cl, cl == 0 && a == 0, false};
}

// kBalanced: the units' chunks in order, unit by unit, cut into `grid` equal contiguous
// ranges (each at least one unit long, so no range lies inside one unit), decoded once per
// CTA (`cta`; the host runs the same code for gtr_gla_balanced_walk).  A CTA first runs the head [0, c_hi) of the unit its range ends in (from zero; its
// end state goes to the next CTA), then its whole units, then the tail [c_lo, N) of the
// unit its range starts in, from the state the previous CTA handed over at the start of
// its own run (long before).
struct BalRange {
    int base_head, base_full, base_tail;  // flattened chunk index = v + the base of v's piece
    int c_hi, t0;                         // pieces: [0, c_hi) head, [c_hi, t0) whole units, [t0, G) tail
    int G;
};
__host__ __device__ __forceinline__ BalRange bal_range(int N, int n_units, int cta, int grid) {
    const long long tot = static_cast<long long>(n_units) * N;
    const long long lo = tot * cta / grid, hi = tot * (cta + 1) / grid;
    const int u_lo = static_cast<int>(lo / N), c_lo = static_cast<int>(lo - static_cast<long long>(u_lo) * N);
    const int u_hi = static_cast<int>(hi / N), c_hi = static_cast<int>(hi - static_cast<long long>(u_hi) * N);
    const int u_first = c_lo ? u_lo + 1 : u_lo;
    BalRange r;
    r.c_hi = c_hi;
    r.t0 = c_hi + (u_hi - u_first) * N;
    r.base_head = u_hi * N;                          // head: chunk v of unit u_hi
    r.base_full = u_first * N - c_hi;                // whole units from u_first on
    r.base_tail = static_cast<int>(lo) - r.t0;       // tail: chunk c_lo + (v - t0) of unit u_lo
    r.G = static_cast<int>(hi - lo);
    return r;
}
// The piece is picked by two compares and the unit by one multiply-high division; a
// three-way branch over the pieces made every role's per-chunk decode slower and cost the
// whole kernel 10 %, and an integer division here another 17 %.
__host__ __device__ __forceinline__ StreamPos stream_pos_bal(int v, int N, int lognv, int base_head, int base_full,
                                                             int base_tail, int c_hi, int t0, const FastDiv &fn) {
    const int g = v + (v < c_hi ? base_head : (v < t0 ? base_full : base_tail));
    const int unit = fdiv(g, fn), c = g - unit * N;
    const bool hin = v == t0;  // the tail's first chunk (t0 == G when there is no tail)
    return {unit >> lognv, unit & ((1 << lognv) - 1), c, 0, 0, c, c == 0 || hin, hin};
}

// kBalanced: bounded wait for the previous CTA's hand-off flag, read with acquire semantics at
// GPU scope (the writer fenced before setting it), so the waiting thread needs no fence of its
// own, which would also wait for its output stores in flight.  Out of line: it runs once per CTA.
__device__ __noinline__ bool handoff_wait(const unsigned long long *f, unsigned long long epoch,
                                          volatile uint32_t *abort_flag) {
    bool got = ld_acquire_u64(f) == epoch;
    const uint64_t t0 = global_timer_ns();
    while (!got && !*abort_flag && global_timer_ns() - t0 < kWaitLimitNs) {
        __nanosleep(64);
        got = ld_acquire_u64(f) == epoch;
    }
    return got;
}

// Visit the TMA load boxes of one chunk: calls f(map height index, smem row, c2, c3).
// Row orders: one 64-row box at token w0 (rows outside the sequence are
// zero-filled).  Column orders: boxes for each column segment, of the segment's
// exact height (at most two: its multiple of 8 and the remainder), plus zero-fill
// boxes placed past the last column for rows outside the sequence.
//
// Runs of rows down one column (at most two zero-fill runs, then the column
// segments), each loaded as at most two boxes: its multiple of 8 and the remainder.
// One call site for f keeps the producer's issue code small.
template <typename F>
__host__ __device__ __forceinline__ void chunk_load_boxes(int order, int T, const FastDiv &gh, int grid_w, int c, F &&f) {
    const int w0 = chunk_w0(order, T, c);
    if ((order >> 1) == 0) {
        f(kHeights - 1, 0, w0, 0);
        return;
    }
    if (w0 >= T || w0 + kC <= 0) {  // a padding chunk wholly past the sequence: all zeros
        f(kHeights - 1, 0, grid_w, 0);
        return;
    }
    const int lo = w0 < 0 ? 0 : w0, hi = (w0 + kC > T) ? T : w0 + kC;
    int phase = 0, w = lo;
#pragma unroll 1
    for (;;) {
        int len, row, c2, c3;
        if (phase == 0) {  // rows before the sequence: zero-fill past the last column
            phase = 1;
            if (lo <= w0) continue;
            len = lo - w0, row = 0, c2 = grid_w, c3 = 0;
        } else if (phase == 1) {  // rows after the sequence
            phase = 2;
            if (hi >= w0 + kC) continue;
            len = w0 + kC - hi, row = hi - w0, c2 = grid_w, c3 = 0;
        } else {  // the next column segment
            if (w >= hi) break;
            const int x = fdiv(w, gh), y = w - x * gh.d;
            len = gh.d - y;
            if (len > hi - w) len = hi - w;
            row = w - w0, c2 = x, c3 = y;
            w += len;
        }
        const int len8 = len & ~7;
#pragma unroll 1
        for (int part = 0; part < 2; ++part) {
            const int n = part == 0 ? len8 : len - len8;
            if (n == 0) continue;
            f(part == 0 ? 6 + n / 8 : n - 1, row + (part == 0 ? 0 : len8), c2, c3 + (part == 0 ? 0 : len8));
        }
    }
}

// Column orders, chunk c wholly inside the sequence: its 64 tokens (down column x0 from row y0
// and on into the next columns) load as one im2col walk per tensor; returns false for row orders
// and for chunks that reach past either end, which load boxes (chunk_load_boxes).
__host__ __device__ __forceinline__ bool chunk_walk_start(int order, int T, const FastDiv &gh, int c, int *x0, int *y0) {
    const int w0 = chunk_w0(order, T, c);
    if ((order >> 1) == 0 || w0 < 0 || w0 + kC > T) return false;
    *x0 = fdiv(w0, gh);
    *y0 = w0 - *x0 * gh.d;
    return true;
}

// fp16-pair mask of score columns 2e, 2e + 1 from a bit set of kept columns
__device__ __forceinline__ uint32_t pmask(uint32_t vbits, int e) {
    return (((vbits >> (2 * e)) & 1u) ? 0x0000FFFFu : 0u) | (((vbits >> (2 * e + 1)) & 1u) ? 0xFFFF0000u : 0u);
}

// Spatial token of walk position w (-1 outside the sequence).
__device__ __forceinline__ int walk_token(int order, int T, const FastDiv &gh, int grid_w, int w) {
    if (w < 0 || w >= T) return -1;
    if ((order >> 1) == 0) return w;
    const int x = fdiv(w, gh);
    return (w - x * gh.d) * grid_w + x;
}

// Exact scores for one chunk (extreme or non-finite log-decays): serial prefix
// of the clamped gates, P[rho][sigma] = sum_i q k 2^{a_r,i - a_j,i} (j <= r) by
// CUDA cores, Qtil = q 2^{a}, Kbar = k 2^{a_last - a}, and the chunk decay.
template <typename E, typename GT>
__device__ __noinline__ void exact_chunk(uint8_t *tq, uint8_t *tk, uint8_t *tgate, float *as,
                                         float *decay, int rev, int tg, int bar_id) {
    if (tg < kD) {
        float run = 0.f;
        for (int r = 0; r < kC; ++r) {
            const int rho = rev ? kC - 1 - r : r;
            const uint16_t bits = *reinterpret_cast<const uint16_t *>(tgate + sw128(rho, tg * 2));
            float x = Elem<GT>::unpack(bits).x * kLog2e;
            x = x < kGateMinLog2 ? kGateMinLog2 : x;
            run += x;
            as[rho * kD + tg] = run;
        }
        decay[tg] = ex2(run);
    }
    named_barrier_sync(bar_id, 128);
    const int rho = tg >> 1, half = tg & 1;
    const int r = rev ? kC - 1 - rho : rho;
    uint32_t packed[16];
    for (int jj = 0; jj < 16; ++jj) {
        float pv[2];
        for (int u = 0; u < 2; ++u) {
            const int sig = half * 32 + 2 * jj + u;
            const int j = rev ? kC - 1 - sig : sig;
            float acc = 0.f;
            if (j <= r) {
                for (int i = 0; i < kD; i += 2) {
                    const float2 qi = Elem<E>::unpack(*reinterpret_cast<const uint32_t *>(tq + sw128(rho, i * 2)));
                    const float2 ki = Elem<E>::unpack(*reinterpret_cast<const uint32_t *>(tk + sw128(sig, i * 2)));
                    acc += qi.x * ki.x * ex2(as[rho * kD + i] - as[sig * kD + i]);
                    acc += qi.y * ki.y * ex2(as[rho * kD + i + 1] - as[sig * kD + i + 1]);
                }
            }
            pv[u] = acc;
        }
        packed[jj] = h2bits(pv[0], pv[1]);
    }
    const int rho_last = rev ? 0 : kC - 1;
    named_barrier_sync(bar_id, 128);  // every q/k/gate read of this chunk is done
    for (int jj = 0; jj < 16; ++jj)
        *reinterpret_cast<uint32_t *>(tgate + sw128(rho, (half * 32 + 2 * jj) * 2)) = packed[jj];
    for (int i = half * 32; i < half * 32 + 32; i += 2) {
        const uint32_t o16 = sw128(rho, i * 2);
        const float2 q2 = Elem<E>::unpack(*reinterpret_cast<const uint32_t *>(tq + o16));
        const float2 k2 = Elem<E>::unpack(*reinterpret_cast<const uint32_t *>(tk + o16));
        const float a0 = as[rho * kD + i], a1 = as[rho * kD + i + 1];
        const float l0 = as[rho_last * kD + i], l1 = as[rho_last * kD + i + 1];
        *reinterpret_cast<uint32_t *>(tq + o16) = h2bits(q2.x * ex2(a0), q2.y * ex2(a1));
        *reinterpret_cast<uint32_t *>(tk + o16) = h2bits(k2.x * ex2(l0 - a0), k2.y * ex2(l1 - a1));
    }
}

// Operands of a tf32-mode chunk (split factors beyond the fp16 range): tf32 Q^ and
// K^ for the score product in the group's operand buffer, fp16 Qtil = Q^ c1 over q and
// Kbar = K^ c2 over k.  Re-reads the thread's 32 log-decays from TMEM (A is kept
// until the operands are built): out of line, this rarer path leaves the fp16 path's
// code and registers as they are (inlined it cost workload 2 6 %).
template <typename E>
__device__ __noinline__ void tf32_operands(uint8_t *tq, uint8_t *tk, uint8_t *opbuf, const float *ref,
                                           uint32_t taddr, int row, int ch0) {
    uint32_t ar[32];
    tmem_ld_16x32bx2_x16(taddr + 0, *reinterpret_cast<uint32_t(*)[16]>(&ar[0]));
    tmem_ld_16x32bx2_x16(taddr + 16, *reinterpret_cast<uint32_t(*)[16]>(&ar[16]));
    tmem_ld_wait();
    uint8_t *qh = opbuf, *kh = opbuf + kTile32;
#pragma unroll
    for (int g8 = 0; g8 < 4; ++g8) {
        const int cl = ch0 + 8 * g8;
        const uint32_t o16 = sw128(row, cl * 2);
        const uint4 qw = *reinterpret_cast<const uint4 *>(tq + o16);
        const uint4 kw = *reinterpret_cast<const uint4 *>(tk + o16);
        const uint32_t qa[4] = {qw.x, qw.y, qw.z, qw.w}, ka[4] = {kw.x, kw.y, kw.z, kw.w};
        // A_mid log2, c1 and c2 of the 8 channels (16-byte aligned rows of the references)
        float am[8], c1v[8], c2v[8];
        *reinterpret_cast<float4 *>(&am[0]) = *reinterpret_cast<const float4 *>(ref + cl);
        *reinterpret_cast<float4 *>(&am[4]) = *reinterpret_cast<const float4 *>(ref + cl + 4);
#pragma unroll
        for (int e = 0; e < 8; ++e) am[e] *= kLog2e;
        *reinterpret_cast<float4 *>(&c1v[0]) = *reinterpret_cast<const float4 *>(ref + 2 * kD + cl);
        *reinterpret_cast<float4 *>(&c1v[4]) = *reinterpret_cast<const float4 *>(ref + 2 * kD + cl + 4);
        *reinterpret_cast<float4 *>(&c2v[0]) = *reinterpret_cast<const float4 *>(ref + 3 * kD + cl);
        *reinterpret_cast<float4 *>(&c2v[4]) = *reinterpret_cast<const float4 *>(ref + 3 * kD + cl + 4);
        float qs[8], ks[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 q2 = Elem<E>::unpack(qa[e]), k2 = Elem<E>::unpack(ka[e]);
            const float e0 = fmaf(__uint_as_float(ar[8 * g8 + 2 * e]), kLog2e, -am[2 * e]);
            const float e1 = fmaf(__uint_as_float(ar[8 * g8 + 2 * e + 1]), kLog2e, -am[2 * e + 1]);
            qs[2 * e] = q2.x * ex2(e0);
            qs[2 * e + 1] = q2.y * ex2(e1);
            ks[2 * e] = k2.x * ex2(-e0);
            ks[2 * e + 1] = k2.y * ex2(-e1);
        }
        *reinterpret_cast<float4 *>(qh + off32(row, cl)) =
            make_float4(to_tf32(qs[0]), to_tf32(qs[1]), to_tf32(qs[2]), to_tf32(qs[3]));
        *reinterpret_cast<float4 *>(qh + off32(row, cl + 4)) =
            make_float4(to_tf32(qs[4]), to_tf32(qs[5]), to_tf32(qs[6]), to_tf32(qs[7]));
        *reinterpret_cast<float4 *>(kh + off32(row, cl)) =
            make_float4(to_tf32(ks[0]), to_tf32(ks[1]), to_tf32(ks[2]), to_tf32(ks[3]));
        *reinterpret_cast<float4 *>(kh + off32(row, cl + 4)) =
            make_float4(to_tf32(ks[4]), to_tf32(ks[5]), to_tf32(ks[6]), to_tf32(ks[7]));
        uint32_t qo[4], ko[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            qo[e] = h2bits(qs[2 * e] * c1v[2 * e], qs[2 * e + 1] * c1v[2 * e + 1]);
            ko[e] = h2bits(ks[2 * e] * c2v[2 * e], ks[2 * e + 1] * c2v[2 * e + 1]);
        }
        *reinterpret_cast<uint4 *>(tq + o16) = make_uint4(qo[0], qo[1], qo[2], qo[3]);
        *reinterpret_cast<uint4 *>(tk + o16) = make_uint4(ko[0], ko[1], ko[2], ko[3]);
    }
}

// GP (gate producer, one key half, whole sequences): the gates are not read but computed
// from the rank-16 projection, g = logsigmoid(a W2 + b) / tau (Sec. 3.1, retention gate):
// Z = a W2 by one MMA into the chunk's TMEM A buffer, g by the gen warpgroup that owns the
// chunk, written as fp16 over the chunk's gate tile, then A = L G as usual (fp16).
// GATED (outputs stored by the gen warpgroups, one key half, one value slice): the stores
// apply the output gate u = SiLU(r) * RMSNorm(o) * w of Sec. 3.1 to the row's fp32 outputs
// (the deployed kernel's fused epilogue, App. C.3), so o is rounded once, as u.
template <typename E, int NH, int NV, int MODE, bool GENOUT, bool GP = false, bool GATED = false>
__global__ void __launch_bounds__(kThreads, 1) gla_tc_kernel(const __grid_constant__ TcParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
    volatile uint32_t *tmem_base_s = reinterpret_cast<volatile uint32_t *>(smem + kOffMisc);
    volatile uint32_t *abort_flag = reinterpret_cast<volatile uint32_t *>(smem + kOffMisc + 4);
    float *decay_s = reinterpret_cast<float *>(smem + kOffDecay);
    volatile uint32_t *mode_s = reinterpret_cast<volatile uint32_t *>(smem + kOffMode);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // the output pass after a summary pass may start now: its CTAs set up (barriers, TMEM) on
    // the free SMs and wait for this grid only before they read the summaries
    if constexpr (MODE == kSummary) pdl_launch_dependents();
    // MODE kFull / kSplitFull: outputs (a split sequence's later segments start from
    // the state folded from the segment summaries).  MODE kSummary: per segment only
    // the end state from zero and the total decay (k, v and gates; no scores or outputs).
    constexpr bool kSum = MODE == kSummary;
    constexpr bool kSplit = MODE == kSplitFull || MODE == kSummary;
    constexpr bool kBal = MODE == kBalanced;
    static_assert(!kBal || NH == 1, "balanced ranges hand over one key half's state");
    static_assert(!GP || (NH == 1 && MODE == kFull), "the gate producer runs whole sequences, one key half");
    static_assert(!GATED || (GENOUT && NH == 1 && NV == 1 && MODE != kSummary), "the fused gate normalises whole rows");
    // element type of the gate tile: the loaded gates, or the fp16 gates the gate producer writes
    using GE = typename std::conditional<GP, __half, E>::type;
    // GENOUT (one key half, outputs): the gen warpgroup that built a chunk also reads its
    // outputs back from TMEM and stores them, while it waits for the P of its next chunk,
    // which takes that work off the epi's serial per-chunk chain.  The host selects it where
    // that was measured faster (fp16 launches of at most one wave); elsewhere the epi stores.
    constexpr bool kGenOut = GENOUT && NH == 1 && !kSum;
    const int N = p.n_chunks;   // chunks per sequence
    const int L = p.seg_len;    // chunks per unit
    constexpr int nh = NH;   // 64-channel key halves per chunk (Dk / 64)
    constexpr int lognv = NV - 1;  // 64-column value slices per sequence (Dv / 64): 1 or 2
    constexpr int kDk = 64 * NH, kDv = 64 * NV;
    // this CTA's stream of virtual chunks: every barrier phase, stage slot and TMEM
    // buffer below follows the stream index (O: the real chunk's index), so
    // consecutive units flow through one pipeline
    BalRange br{};
    if constexpr (kBal) br = bal_range(N, p.n_units, static_cast<int>(blockIdx.x), static_cast<int>(gridDim.x));
    const int b_head = br.base_head, b_full = br.base_full, b_tail = br.base_tail, b_chi = br.c_hi, b_t0 = br.t0;
    const int G = kBal ? br.G
                       : L * nh *
                             ((p.n_units - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                              static_cast<int>(gridDim.x));
    auto pos = [&](int v) -> StreamPos {
        if constexpr (kBal) return stream_pos_bal(v, N, lognv, b_head, b_full, b_tail, b_chi, b_t0, p.bal_n);
        else return stream_pos(v, L, nh, lognv, p.fd_per, kSplit, p.fd_nsu);
    };
    const int rev = p.order & 1;

    if (threadIdx.x == 0) {
        *abort_flag = 0u;
        for (int i = 0; i < kSlots; ++i) {
            mbar_init(&bars[BAR_FULL + i], 1);
            mbar_init(&bars[BAR_EMPTY + i], MODE == kSummary ? 1 : 2);  // after U(c) and after O(c)
            mbar_init(&bars[BAR_REFS + i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars[BAR_AFULL + i], 1);
            mbar_init(&bars[BAR_PURDY + i], 8);
            mbar_init(&bars[BAR_PFULL + i], 1);
            mbar_init(&bars[BAR_UFULL + i], 1);
            mbar_init(&bars[BAR_ORDY + i], 8);
            mbar_init(&bars[BAR_OFULL + i], 1);
            mbar_init(&bars[BAR_ZFULL + i], 1);
            mbar_init(&bars[BAR_GRDY + i], 4);
        }
        mbar_init(&bars[BAR_DONE], 3);  // one commit per issuer warp
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(const_cast<uint32_t *>(tmem_base_s), kTmemCols);
        tmem_relinquish();
    }
    if (warp >= 2 && warp < 6) {
        // triangle of ones in scan order: L[rho][sigma] = 1 when sigma is at or before rho
        const int tg = threadIdx.x - 64;
        const int rho = tg >> 1, half = tg & 1;
        uint8_t *L = smem + kOffL;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int s0 = half * 32 + u * 8 + 2 * e;
                const bool k0 = rev ? (s0 >= rho) : (s0 <= rho);
                const bool k1 = rev ? (s0 + 1 >= rho) : (s0 + 1 <= rho);
                w[e] = (k0 ? (uint32_t)Elem<GE>::one : 0u) | ((k1 ? (uint32_t)Elem<GE>::one : 0u) << 16);
            }
            *reinterpret_cast<uint4 *>(L + sw128(rho, (half * 32 + u * 8) * 2)) = make_uint4(w[0], w[1], w[2], w[3]);
        }
        fence_proxy_async_smem();
    }
    // kSplitFull: the start state of the CTA's segment (a split launch gives every CTA one
    // segment), folded from the summaries of the segments before it by all 512 threads, each
    // taking 8 of a key half's 64 x 64 values and walking the summaries from the latest back
    // (S_start = sum_s' (prod_{s' < s'' < seg} Diag(D_s'')) S_end(s'), Eq. chunk_boundary_main
    // across segments) with several summaries' loads in flight.  A serial fold by the epi alone
    // waited one L2 round trip per summary, about 8 us for the 13th segment.  The result lands in
    // gen warpgroup 0's tf32 operand buffer, which the epi reads on entry; the group writes the
    // buffer only after the epi's arrival on named barrier kBarSin.
    if constexpr (MODE == kSplitFull) {
        pdl_wait();  // the summaries are the previous grid's: this launch may start before it ends
        const StreamPos p0 = pos(0);
        if (G > 0 && p0.seg > 0) {
            float *sin = reinterpret_cast<float *>(smem + kOffOp);  // [NH][64 rows][64 columns] fp32
            const size_t stride = (size_t)kDk * kDv + kDk;
            const float *base = p.summary + (size_t)p0.bh * (p.nseg - 1) * stride;
            const int r = threadIdx.x >> 3, col = (threadIdx.x & 7) * 8;
#pragma unroll
            for (int a = 0; a < NH; ++a) {
                float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                float coef = 1.f;
#pragma unroll 4
                for (int s2 = p0.seg - 1; s2 >= 0; --s2) {
                    const float *bs = base + (size_t)s2 * stride;
                    const float4 *x = reinterpret_cast<const float4 *>(bs + (size_t)(64 * a + r) * kDv + 64 * p0.vb + col);
                    const float4 x0 = x[0], x1 = x[1];
                    const float d = bs[(size_t)kDk * kDv + 64 * a + r];
                    acc[0] = fmaf(coef, x0.x, acc[0]);
                    acc[1] = fmaf(coef, x0.y, acc[1]);
                    acc[2] = fmaf(coef, x0.z, acc[2]);
                    acc[3] = fmaf(coef, x0.w, acc[3]);
                    acc[4] = fmaf(coef, x1.x, acc[4]);
                    acc[5] = fmaf(coef, x1.y, acc[5]);
                    acc[6] = fmaf(coef, x1.z, acc[6]);
                    acc[7] = fmaf(coef, x1.w, acc[7]);
                    coef *= d;
                }
                float4 *dst = reinterpret_cast<float4 *>(sin + (64 * a + r) * 64 + col);
                dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
                dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_base_s;

    if (warp == 0) {
        // ======================================================= TMA producer
        if (lane == 0) {
            int issued = 0;
            for (int g = 0; g < G; ++g) {
                const int sl = g % kSlots;
                const StreamPos ps = pos(g);
                const int b = fdiv(ps.bh, p.fd_H), h = ps.bh - b * p.H, c = ps.c;
                const int xk = 64 * ps.a, xv = 64 * ps.vb;  // channel offsets of the key half, value slice
                if (!mbar_wait(&bars[BAR_EMPTY + sl], ((g / kSlots) & 1) ^ 1, abort_flag, kWaitLimitNs)) {
                    record_timeout(abort_flag);
                    break;
                }
                uint8_t *st = smem + kOffSlot + sl * kSlotBytes;
                uint64_t *fb = &bars[BAR_FULL + sl];
                if (!(p.drop_load && blockIdx.x == 0 && g == 0)) {
                    // gate producer: a unit's first chunk also brings the head's W2 block, into the
                    // buffer of the unit's parity (the unit before last, whose Z products used it,
                    // ended at least four chunks earlier: its last Z completed before this slot freed)
                    const bool w2 = GP && ps.cl == 0;
                    mbar_arrive_expect_tx(fb, (kSum ? kSlotBytes - kTile16 : kSlotBytes) + (w2 ? kW2Bytes : 0));
                    if (w2) tma_load_5d(smem + kOffW2 + (fdiv(g, p.fd_L) & 1) * kW2Bytes, &p.w2map, fb, 0, 0, h, 0, 0);
                    int x0, y0;
                    if (chunk_walk_start(p.order, p.T, p.fd_gh, c, &x0, &y0)) {
                        // column orders, chunk inside the sequence: one im2col walk per tensor
                        // (boxes per column segment cost the TMA unit one request each and ran
                        // up to 1.9x slower)
                        if (!kSum) tma_load_im2col_5d(st + kQ, &p.cmaps[T_Q], fb, xk, y0, x0, h, b);
                        tma_load_im2col_5d(st + kK, &p.cmaps[T_K], fb, xk, y0, x0, h, b);
                        tma_load_im2col_5d(st + kV, &p.cmaps[T_V], fb, xv, y0, x0, h, b);
                        tma_load_im2col_5d(st + kG, &p.cmaps[T_G], fb, GP ? 0 : xk, y0, x0, GP ? 0 : h, b);
                    } else chunk_load_boxes(p.order, p.T, p.fd_gh, p.grid_w, c, [&](int hi, int row, int c2, int c3) {
                        if (!kSum) tma_load_5d(st + kQ + row * 128, &p.maps[T_Q][hi], fb, xk, h, c2, c3, b);
                        tma_load_5d(st + kK + row * 128, &p.maps[T_K][hi], fb, xk, h, c2, c3, b);
                        tma_load_5d(st + kV + row * 128, &p.maps[T_V][hi], fb, xv, h, c2, c3, b);
                        // the gate tile, or (gate producer) the 16 projection values of each token,
                        // zero-filled to a 128-byte row
                        tma_load_5d(st + kG + row * 128, &p.maps[T_G][hi], fb, GP ? 0 : xk, GP ? 0 : h, c2, c3, b);
                    });
                }
                ++issued;
            }
            if (*abort_flag) {  // never leave while copies are still landing in shared memory
                for (int g = (issued > kSlots ? issued - kSlots : 0); g < issued; ++g)
                    if (!(p.drop_load && blockIdx.x == 0 && g == 0))
                        mbar_wait(&bars[BAR_FULL + g % kSlots], (g / kSlots) & 1, nullptr, kWaitLimitNs);
            }
        }
    } else if (warp == 1 || warp >= 14) {
        // ======================================================= MMA issuers
        // Three warps issue the products, each in program order and waiting only for
        // its own inputs, so that the issue overhead of one product never delays
        // another.  A whole warp runs each loop (operands warp-uniform) and one
        // elected lane issues each MMA.
        //   warp 1   A(c) = L G          once chunk c landed and gen(c-2) built its
        //                                operands (so TMEM A of the parity was read)
        //   warp 14  P(c) = Q^ K^^T,     once PURDY(c): gen(c) operands in smem and epi
        //            U(c) = Kbar^T V     drained U(c-2)
        //   warp 15  O(c) = Q S'_[c] + P V   once ORDY(c)
        // A tcgen05.commit tracks only its own thread's MMAs: the slot of chunk c is
        // released by two commits, after U(c) (warp 14) and after O(c) (warp 15); P(c)
        // and A(c) completed before ORDY(c).  No waiter can be overtaken by two phases
        // of its barrier: PURDY(c + 2) needs A(c + 2) and U(c), FULL of the next chunk
        // of a slot needs that slot's EMPTY, ORDY(c + 2) needs O(c) read.
        const uint32_t slot0 = smem_u32(smem + kOffSlot);
        bool ok = true;
        if (warp == 1) {
            const uint32_t idesc_a = instr_desc(Elem<GE>::fmt, 64, 64, 0, 1);
            const uint32_t idesc_z = instr_desc(Elem<E>::fmt, 64, 64, 0, 1);  // a K-major, W2 MN-major
            const uint64_t dL = kdesc(smem_u32(smem + kOffL));

            // GP: Z runs one chunk ahead of A = L G, so that the two gen groups compute their
            // chunks' gates concurrently: iteration c issues Z(c), then A(c - 1) once the gen group
            // of c - 1 wrote its gates.  Z(c) reuses the A buffer of chunk c - 2 (PURDY(c - 2): its
            // A was read), A(c - 1) overwrites Z(c - 1) (GRDY(c - 1): Z was read).
            for (int c = 0; c < G + (GP ? 1 : 0); ++c) {
                if (c < G) {
                    if (c >= 2) {
                        ok = !__any_sync(0xffffffffu, !mbar_wait(&bars[BAR_PURDY + (c & 1)], ((c - 2) >> 1) & 1, abort_flag, kWaitLimitNs));
                        if (!ok) break;
                    }
                    ok = !__any_sync(0xffffffffu, !mbar_wait(&bars[BAR_FULL + c % kSlots], (c / kSlots) & 1, abort_flag, kWaitLimitNs));
                    if (!ok) break;
                    tc_fence_after();
                    if constexpr (GP) {
                        // Z = a W2 (M = 64 tokens, N = 64 channels, K = r = 16: one MMA) into the
                        // chunk's A buffer; a tile K-major with 128-byte rows, W2 MN-major
                        const uint64_t da = kdesc(slot0 + (c % kSlots) * kSlotBytes + kG);
                        const uint64_t dw = mndesc(smem_u32(smem + kOffW2) + (fdiv(c, p.fd_L) & 1) * kW2Bytes);
                        mma_f16_ss_warp(tmem + kColA + (c & 1) * 64, da, dw, idesc_z, 0);
                        mma_commit_warp(&bars[BAR_ZFULL + (c & 1)]);
                    }
                }
                const int ca = GP ? c - 1 : c;  // the chunk whose A = L G goes now
                if (ca < 0) continue;
                if constexpr (GP) {
                    ok = !__any_sync(0xffffffffu, !mbar_wait(&bars[BAR_GRDY + (ca & 1)], (ca >> 1) & 1, abort_flag, kWaitLimitNs));
                    if (!ok) break;
                    tc_fence_after();
                }
                const uint64_t dg = mndesc(slot0 + (ca % kSlots) * kSlotBytes + kG);
                const uint32_t d = tmem + kColA + (ca & 1) * 64;
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) mma_f16_ss_warp(d, dL + 2 * ks, dg + 128 * ks, idesc_a, ks > 0);
                mma_commit_warp(&bars[BAR_AFULL + (ca & 1)]);
            }
        } else if (warp == 14) {
            const uint32_t idesc_p16 = instr_desc(kFmtF16, 64, 64, 0, 0);
            const uint32_t idesc_p32 = instr_desc(kFmtTF32, 64, 64, 0, 0);
            const uint32_t idesc_u = instr_desc(kFmtF16, 64, 64, 1, 1);
            const uint64_t dqh0 = kdesc(smem_u32(smem + kOffOp)), dkh0 = kdesc(smem_u32(smem + kOffOp + kTile32));
            int su = 0;
            for (int c = 0; c < G; ++c) {
                ok = !__any_sync(0xffffffffu, !mbar_wait(&bars[BAR_PURDY + (c & 1)], (c >> 1) & 1, abort_flag, kWaitLimitNs));
                if (!ok) break;
                tc_fence_after();
                const uint32_t st = slot0 + su * kSlotBytes;
                const uint32_t mode = __shfl_sync(0xffffffffu, mode_s[su], 0);
                const uint32_t dp = tmem + kColP + (c & 1) * 64;
                if (kSum) {
                    // summaries need no scores
                } else if (mode == kModeF16) {
                    const uint64_t dq = kdesc(st + kQ), dk = kdesc(st + kK);
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks) mma_f16_ss_warp(dp, dq + 2 * ks, dk + 2 * ks, idesc_p16, ks > 0);
                    mma_commit_warp(&bars[BAR_PFULL + (c & 1)]);
                } else if (mode == kModeTF32) {
                    const uint64_t dqh = dqh0 + (c & 1) * (2 * kTile32 >> 4), dkh = dkh0 + (c & 1) * (2 * kTile32 >> 4);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks) {
                        const uint32_t off = (ks >> 2) * 512 + (ks & 3) * 2;  // (8192 B, 32 B) >> 4
                        mma_tf32_ss_warp(dp, dqh + off, dkh + off, idesc_p32, ks > 0);
                    }
                    mma_commit_warp(&bars[BAR_PFULL + (c & 1)]);
                } else if (lane == 0) {
                    mbar_arrive(&bars[BAR_PFULL + (c & 1)]);  // exact scores are already in smem
                }
                __syncwarp();
                // U(c) = Kbar^T V (fp16 mode: K^^T V): the k tile read as the MN-major A
                const uint64_t dk = mndesc(st + kK), dv = mndesc(st + kV);
                const uint32_t du = tmem + kColU + (c & 1) * 64;
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) mma_f16_ss_warp(du, dk + 128 * ks, dv + 128 * ks, idesc_u, ks > 0);
                mma_commit_warp(&bars[BAR_UFULL + (c & 1)]);
                mma_commit_warp(&bars[BAR_EMPTY + su]);  // U is the slot's last reader among this warp's MMAs
                su = (su == kSlots - 1) ? 0 : su + 1;
            }
        } else if (!kSum) {
            const uint32_t idesc_o = instr_desc(kFmtF16, 64, 64, 0, 1);
            const uint32_t sbuf = smem_u32(smem + kOffS);
            int so = 0;
            for (int c = 0; c < G; ++c) {
                ok = !__any_sync(0xffffffffu, !mbar_wait(&bars[BAR_ORDY + (c & 1)], (c >> 1) & 1, abort_flag, kWaitLimitNs));
                if (!ok) break;
                tc_fence_after();
                // O(c) = Qtil S_[c] + P V  (fp16 mode: Q^ (Diag(c1) S_[c]) + P V); the key
                // halves of one real chunk accumulate into the same TMEM buffer
                const uint32_t st = slot0 + so * kSlotBytes;
                const uint64_t dq = kdesc(st + kQ), ds = mndesc(sbuf + (c & 1) * kTile16);
                const uint64_t dpm = kdesc(st + kG), dv = mndesc(st + kV);
                const uint32_t d = tmem + kColO + ((c / nh) & 1) * 64;
                const uint32_t acc0 = (c % nh) != 0;
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) mma_f16_ss_warp(d, dq + 2 * ks, ds + 128 * ks, idesc_o, acc0 | (ks > 0));
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) mma_f16_ss_warp(d, dpm + 2 * ks, dv + 128 * ks, idesc_o, 1);
                mma_commit_warp(&bars[BAR_OFULL + (c & 1)]);
                mma_commit_warp(&bars[BAR_EMPTY + so]);  // every product of the slot's chunk is done
                so = (so == kSlots - 1) ? 0 : so + 1;
            }
        }
        if (!ok && lane == 0) record_timeout(abort_flag);
        mma_commit_warp(&bars[BAR_DONE]);  // TMEM is released only after every MMA completed
        mbar_wait(&bars[BAR_DONE], 0, nullptr, kWaitLimitNs);
    } else if (warp < 10) {
        // ======================================================= gen warpgroups (chunks c = gw mod 2)
        const int gw = (warp - 2) >> 2;          // 0: even chunks, 1: odd chunks
        const int bar_id = 1 + gw;
        if constexpr (MODE == kSplitFull) {
            if (gw == 0) named_barrier_sync(kBarSin, 256);  // the epi took the folded start state
        }
        const int q4 = warp & 3, hc = lane >> 4;
        const int row = 16 * q4 + (lane & 15);   // smem row rho of this thread's accumulator row
        const int ch0 = 32 * hc;                 // its 32 key channels (A) / score columns (P)
        const uint32_t lane_base = static_cast<uint32_t>(32 * q4) << 16;
        const int tg = threadIdx.x - 64 - 128 * gw;
        const int rho_mid = rev ? 32 : 31, rho_last = rev ? 0 : 63;
        // causal mask of this thread's 32 score columns as packed fp16-pair masks (scan order)
        uint32_t vbits = 0u;  // bit s: score column ch0 + s is kept
        for (int s = 0; s < 32; ++s)
            if (rev ? (ch0 + s >= row) : (ch0 + s <= row)) vbits |= 1u << s;
        // outputs of chunk co (this group's) once O(co) completed: TMEM -> this thread's row at its
        // token's spatial position; false when the wait gave up
        auto gen_out = [&](int co) -> bool {
            if (!mbar_wait(&bars[BAR_OFULL + (co & 1)], (co >> 1) & 1, abort_flag, kWaitLimitNs)) return false;
            tc_fence_after();
            uint32_t r[32];
            tmem_ld_16x32bx2_x16(tmem + lane_base + kColO + (co & 1) * 64 + 0, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
            tmem_ld_16x32bx2_x16(tmem + lane_base + kColO + (co & 1) * 64 + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
            tmem_ld_wait();
            uint32_t ow[16];
            const StreamPos po = pos(co);
            const int b = fdiv(po.bh, p.fd_H), h = po.bh - b * p.H;
            const int t = walk_token(p.order, p.T, p.fd_gh, p.grid_w, chunk_w0(p.order, p.T, po.c) + row);
            if constexpr (GATED) {
                // u = SiLU(r) * o / sqrt(mean_j o_j^2 + eps) * w over the head's Dv outputs: this
                // thread holds 32 of the row's columns, the lane 16 apart the other 32 (padded
                // columns are 0 and count for nothing)
                uint4 rq[4] = {};
                const E *rrow = static_cast<const E *>(p.gate_r) + (((size_t)b * p.T + (t < 0 ? 0 : t)) * p.H + h) * p.Dv;
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (t >= 0 && ch0 + 8 * q < p.Dv) rq[q] = *reinterpret_cast<const uint4 *>(rrow + ch0 + 8 * q);
                float ss = 0.f;
#pragma unroll
                for (int j = 0; j < 32; ++j) ss = fmaf(__uint_as_float(r[j]), __uint_as_float(r[j]), ss);
                ss += __shfl_xor_sync(0xffffffffu, ss, 16);
                const float inv = rsqrtf(ss / static_cast<float>(p.Dv) + p.gate_eps);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float wq[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                    if (ch0 + 8 * q < p.Dv) {
                        *reinterpret_cast<float4 *>(&wq[0]) = __ldg(reinterpret_cast<const float4 *>(p.gate_w + ch0 + 8 * q));
                        *reinterpret_cast<float4 *>(&wq[4]) = __ldg(reinterpret_cast<const float4 *>(p.gate_w + ch0 + 8 * q + 4));
                    }
                    const uint32_t rw[4] = {rq[q].x, rq[q].y, rq[q].z, rq[q].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 z = Elem<E>::unpack(rw[e]);
                        const float s0 = __fdividef(z.x, 1.f + __expf(-z.x)), s1 = __fdividef(z.y, 1.f + __expf(-z.y));
                        const float o0 = __uint_as_float(r[8 * q + 2 * e]), o1 = __uint_as_float(r[8 * q + 2 * e + 1]);
                        ow[4 * q + e] = Elem<E>::pack(s0 * o0 * inv * wq[2 * e], s1 * o1 * inv * wq[2 * e + 1]);
                    }
                }
            } else {
#pragma unroll
                for (int j = 0; j < 16; ++j) ow[j] = Elem<E>::pack(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1]));
            }
            if (t >= 0) {  // the row's columns inside Dv (padded columns stay behind)
                const int col0 = 64 * po.vb + ch0;
                uint4 *dst = reinterpret_cast<uint4 *>(static_cast<E *>(p.out) + (((size_t)b * p.T + t) * p.H + h) * p.Dv + col0);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (col0 + 8 * q < p.Dv) dst[q] = make_uint4(ow[4 * q], ow[4 * q + 1], ow[4 * q + 2], ow[4 * q + 3]);
            }
            return true;
        };
        int last_c = -1;  // the group's last chunk completed (its outputs are stored after the loop)
        for (int c = gw; c < G; c += 2) {
            const int sl = c % kSlots, bb = c & 1;
            const uint32_t ph = (c >> 1) & 1;
            uint8_t *st = smem + kOffSlot + sl * kSlotBytes;
            bool zfail = false;
            if constexpr (GP) {
                // the chunk's gates from Z = a W2 (Sec. 3.1): g = logsigmoid(z + b) / tau in fp32,
                // written as fp16 over the a tile, whose Z product has completed; rows outside
                // the sequence keep g = 0 (no decay), as zero-filled gate rows do
                zfail = !mbar_wait(&bars[BAR_ZFULL + bb], ph, abort_flag, kWaitLimitNs);
                tc_fence_after();
                uint32_t zr[32];
                tmem_ld_16x32bx2_x16(tmem + lane_base + kColA + bb * 64 + 0, *reinterpret_cast<uint32_t(*)[16]>(&zr[0]));
                tmem_ld_16x32bx2_x16(tmem + lane_base + kColA + bb * 64 + 16, *reinterpret_cast<uint32_t(*)[16]>(&zr[16]));
                tmem_ld_wait();
                const StreamPos pz = pos(c);
                const int wz = chunk_w0(p.order, p.T, pz.c) + row;
                const bool live = wz >= 0 && wz < p.T;
                const float *bz = p.gbias + (size_t)(pz.bh - fdiv(pz.bh, p.fd_H) * p.H) * p.Dk;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    // 8 channels of the bias (Dk is a multiple of 8: all inside it or all past it)
                    float bq[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                    if (ch0 + 8 * q < p.Dk) {
                        *reinterpret_cast<float4 *>(&bq[0]) = __ldg(reinterpret_cast<const float4 *>(bz + ch0 + 8 * q));
                        *reinterpret_cast<float4 *>(&bq[4]) = __ldg(reinterpret_cast<const float4 *>(bz + ch0 + 8 * q + 4));
                    }
                    uint32_t gq[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float g0 = live ? log_sigmoid(__uint_as_float(zr[8 * q + 2 * e]) + bq[2 * e]) * p.tau_inv : 0.f;
                        const float g1 = live ? log_sigmoid(__uint_as_float(zr[8 * q + 2 * e + 1]) + bq[2 * e + 1]) * p.tau_inv : 0.f;
                        gq[e] = h2bits(g0, g1);
                    }
                    *reinterpret_cast<uint4 *>(st + kG + sw128(row, (ch0 + 8 * q) * 2)) = make_uint4(gq[0], gq[1], gq[2], gq[3]);
                }
                fence_proxy_async_smem();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&bars[BAR_GRDY + bb]);  // this warp's rows of G are in smem
            }
            const bool fail = zfail || !mbar_wait(&bars[BAR_AFULL + bb], ph, abort_flag, kWaitLimitNs);
            // bf16 values become fp16 MMA operands in place (exact for |v| in the fp16
            // normal range); the loads go first so that their latency hides behind the
            // operand build, the converted words are stored with the operands
            tc_fence_after();
            uint32_t ar[32];
            tmem_ld_16x32bx2_x16(tmem + lane_base + kColA + bb * 64 + 0, *reinterpret_cast<uint32_t(*)[16]>(&ar[0]));
            tmem_ld_16x32bx2_x16(tmem + lane_base + kColA + bb * 64 + 16, *reinterpret_cast<uint32_t(*)[16]>(&ar[16]));
            tmem_ld_wait();
            // references of chunk c: [0,64) raw A_mid, [64,128) raw A_last, [128,192) c1 = 2^{A_mid},
            // [192,256) c2 = 2^{A_last - A_mid}
            float *ref = reinterpret_cast<float *>(smem + kOffRef) + sl * kRefFloats;
            if (!fail && (row == rho_mid || row == rho_last)) {
                float *dst = ref + (row == rho_mid ? 0 : kD) + ch0;
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    reinterpret_cast<float4 *>(dst)[q] = make_float4(__uint_as_float(ar[4 * q]), __uint_as_float(ar[4 * q + 1]),
                                                                     __uint_as_float(ar[4 * q + 2]), __uint_as_float(ar[4 * q + 3]));
            }
            tc_fence_before();
            if (named_barrier_or(bar_id, 128, fail || *abort_flag != 0u)) {  // the group gives up together
                record_timeout(abort_flag);
                break;
            }
            // every warp reduces the split range M over the 64 channels itself (no second
            // barrier); warp 0 of the group writes the constants the readout and epi use
            uint32_t mode;
            {
                const float am0 = ref[lane] * kLog2e, al0 = ref[kD + lane] * kLog2e;
                const float am1 = ref[lane + 32] * kLog2e, al1 = ref[kD + lane + 32] * kLog2e;
                float m = fmaxf(fmaxf(-am0, am0 - al0), fmaxf(-am1, am1 - al1));
                if (!(m <= 3.0e38f)) m = 3.0e38f;  // NaN / inf gates: exact path
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 16));
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 8));
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 4));
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 2));
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 1));
                mode = m <= kMaxRefF16 ? kModeF16 : (m <= kMaxRefTF32 ? kModeTF32 : kModeExact);
                if (tg < 32) {
                    ref[2 * kD + lane] = ex2(am0);
                    ref[2 * kD + lane + 32] = ex2(am1);
                    ref[3 * kD + lane] = ex2(al0 - am0);
                    ref[3 * kD + lane + 32] = ex2(al1 - am1);
                    decay_s[sl * kD + lane] = ex2(al0);
                    decay_s[sl * kD + lane + 32] = ex2(al1);
                    if (tg == 0) mode_s[sl] = mode;
                }
            }
            uint8_t *tq = st + kQ, *tk = st + kK, *tgt = st + kG;
            bool opfail = false;
            if (mode != kModeF16) {
                // the constants written by warp 0 above are read by every warp of the group; the
                // group's own operand buffer was last read by P(c - 2), complete before mask(c - 2)
                opfail = named_barrier_or(bar_id, 128, false);
            }
            if (mode == kModeF16) {
#pragma unroll
                for (int g8 = 0; g8 < 4; ++g8) {
                    const int cl = ch0 + 8 * g8;
                    const float4 am0 = *reinterpret_cast<const float4 *>(ref + cl);  // raw A_mid
                    const float4 am1 = *reinterpret_cast<const float4 *>(ref + cl + 4);
                    const float amv[8] = {am0.x * kLog2e, am0.y * kLog2e, am0.z * kLog2e, am0.w * kLog2e,
                                          am1.x * kLog2e, am1.y * kLog2e, am1.z * kLog2e, am1.w * kLog2e};
                    const uint32_t o16 = sw128(row, cl * 2);
                    const uint4 qw = kSum ? make_uint4(0u, 0u, 0u, 0u) : *reinterpret_cast<const uint4 *>(tq + o16);
                    const uint4 kw = *reinterpret_cast<const uint4 *>(tk + o16);
                    const uint32_t qa[4] = {qw.x, qw.y, qw.z, qw.w}, ka[4] = {kw.x, kw.y, kw.z, kw.w};
                    uint32_t qo[4], ko[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 q2 = Elem<E>::unpack(qa[e]), k2 = Elem<E>::unpack(ka[e]);
                        const float e0 = fmaf(__uint_as_float(ar[8 * g8 + 2 * e]), kLog2e, -amv[2 * e]);
                        const float e1 = fmaf(__uint_as_float(ar[8 * g8 + 2 * e + 1]), kLog2e, -amv[2 * e + 1]);
                        qo[e] = h2bits(q2.x * ex2(e0), q2.y * ex2(e1));
                        ko[e] = h2bits(k2.x * ex2(-e0), k2.y * ex2(-e1));
                    }
                    // Q^ over q, K^ over k (each thread rewrites exactly what it read)
                    if (!kSum) *reinterpret_cast<uint4 *>(tq + o16) = make_uint4(qo[0], qo[1], qo[2], qo[3]);
                    *reinterpret_cast<uint4 *>(tk + o16) = make_uint4(ko[0], ko[1], ko[2], ko[3]);
                }
            } else if (!opfail) {
                if (mode == kModeTF32)
                    tf32_operands<E>(tq, tk, smem + kOffOp + gw * 2 * kTile32, ref, tmem + lane_base + kColA + bb * 64, row, ch0);
                else
                    exact_chunk<E, GE>(tq, tk, tgt, reinterpret_cast<float *>(smem + kOffOp + gw * 2 * kTile32), decay_s + sl * kD, rev, tg,
                                   bar_id);
            }
            if constexpr (std::is_same<E, __nv_bfloat16>::value) {
                uint4 vw[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) vw[q] = *reinterpret_cast<const uint4 *>(st + kV + sw128(row, (ch0 + 8 * q) * 2));
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t *wp = reinterpret_cast<uint32_t *>(&vw[q]);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 fv = Elem<E>::unpack(wp[e]);
                        wp[e] = h2bits(fv.x, fv.y);
                    }
                    *reinterpret_cast<uint4 *>(st + kV + sw128(row, (ch0 + 8 * q) * 2)) = vw[q];
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            if (named_barrier_or(bar_id, 128, opfail)) {
                record_timeout(abort_flag);
                break;
            }
            if (tg == 0) mbar_arrive(&bars[BAR_REFS + sl]);  // constants and mode of chunk c -> epi
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_PURDY + bb]);  // operands in smem, A(c) read
            if (kSum) continue;  // no scores
            // ---- outputs of the group's previous chunk c-2 (O(c) reuses its TMEM buffer only
            // after ORDY(c), which this group signals below)
            bool ofail = false;
            if constexpr (kGenOut) {
                if (c >= 2) ofail = !gen_out(c - 2);
            }
            // ---- masked scores of chunk c over its gate tile (consumed by A(c) long ago)
            const bool pfail = ofail || !mbar_wait(&bars[BAR_PFULL + bb], ph, abort_flag, kWaitLimitNs);
            if (named_barrier_or(bar_id, 128, pfail)) {
                record_timeout(abort_flag);
                break;
            }
            if (mode != kModeExact) {
                tc_fence_after();
                uint32_t r[32];
                tmem_ld_16x32bx2_x16(tmem + lane_base + kColP + bb * 64 + 0, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
                tmem_ld_16x32bx2_x16(tmem + lane_base + kColP + bb * 64 + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
                tmem_ld_wait();
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    *reinterpret_cast<uint4 *>(tgt + sw128(row, (ch0 + 8 * q) * 2)) = make_uint4(
                        h2bits(__uint_as_float(r[8 * q + 0]), __uint_as_float(r[8 * q + 1])) & pmask(vbits, 4 * q + 0),
                        h2bits(__uint_as_float(r[8 * q + 2]), __uint_as_float(r[8 * q + 3])) & pmask(vbits, 4 * q + 1),
                        h2bits(__uint_as_float(r[8 * q + 4]), __uint_as_float(r[8 * q + 5])) & pmask(vbits, 4 * q + 2),
                        h2bits(__uint_as_float(r[8 * q + 6]), __uint_as_float(r[8 * q + 7])) & pmask(vbits, 4 * q + 3));
            }
            tc_fence_before();
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars[BAR_ORDY + bb]);  // this warp's rows of P are in smem
            last_c = c;
        }
        if constexpr (kGenOut) {
            if (last_c >= 0 && last_c + 2 >= G && !gen_out(last_c)) record_timeout(abort_flag);
        }
    } else {
        // ======================================================= epi warpgroup (warps 10-13)
        // Carries the fp32 state of the current key half in registers (thread: channel
        // row, 32 value columns; with two key halves the other half's state waits in So
        // and the two swap after every virtual chunk), writes Diag(c1) S for the readout
        // product, folds U into the state, and stores each real chunk's outputs at its
        // tokens' spatial positions once the O product of its last key half completed.
        const int q4 = warp & 3, hc = lane >> 4;
        const int row = 16 * q4 + (lane & 15);   // channel i for U / S, token rho for O
        const int ch0 = 32 * hc;
        const uint32_t lane_base = static_cast<uint32_t>(32 * q4) << 16;
        E *out = static_cast<E *>(p.out);
        float S[32], So[NH == 2 ? 32 : 1];
#pragma unroll
        for (int j = 0; j < 32; ++j) S[j] = 0.f;
        if constexpr (NH == 2) {
#pragma unroll
            for (int j = 0; j < 32; ++j) So[j] = 0.f;
        }
        if constexpr (MODE == kSplitFull) {  // the start state the whole CTA folded (segments past the first)
            if (G > 0 && pos(0).seg > 0) {
                const float *sin = reinterpret_cast<const float *>(smem + kOffOp) + row * 64 + ch0;
#pragma unroll
                for (int j = 0; j < 32; ++j) S[j] = sin[j];
                if constexpr (NH == 2) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) So[j] = sin[64 * 64 + j];
                }
            }
            named_barrier_arrive(kBarSin, 256);  // gen warpgroup 0 may now use its operand buffer
        }
        float dp = 1.f, dpo = 1.f;  // summaries: the segment's decay product per key half
        // Start state of a split sequence's segment seg > 0 (key half `half`): fold the
        // end states from zero of segments 0 .. seg-1 with their total decays,
        // S_start(s + 1) = Diag(D_s) S_start(s) + S_end(s).
        const size_t sum_stride = (size_t)kDk * kDv + kDk;
        auto start_state = [&](float(&st)[32], int half, const StreamPos &q) {
#pragma unroll
            for (int j = 0; j < 32; ++j) st[j] = 0.f;
            const float *base = p.summary + (size_t)q.bh * (p.nseg - 1) * sum_stride;
            for (int s2 = 0; s2 < q.seg; ++s2, base += sum_stride) {
                const float d = base[(size_t)kDk * kDv + 64 * half + row];
                const float4 *x = reinterpret_cast<const float4 *>(base + (size_t)(64 * half + row) * kDv + 64 * q.vb + ch0);
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float4 w = x[j];
                    st[4 * j] = fmaf(d, st[4 * j], w.x);
                    st[4 * j + 1] = fmaf(d, st[4 * j + 1], w.y);
                    st[4 * j + 2] = fmaf(d, st[4 * j + 2], w.z);
                    st[4 * j + 3] = fmaf(d, st[4 * j + 3], w.w);
                }
            }
        };
        bool ok = true;
        if (lane == 0) {  // TMEM U buffers start out free: the drains of chunks -2 and -1
            mbar_arrive(&bars[BAR_PURDY + 0]);
            mbar_arrive(&bars[BAR_PURDY + 1]);
        }
        // kBalanced: the loop runs in three pieces (head run, whole units, tail run) with the
        // hand-offs between them, so that the per-chunk loop itself carries no hand-off code
        // (in the loop it slowed every chunk: the SM's instruction cache is shared by all roles)
        const int cut0 = kBal ? b_chi : G + 1, cut1 = kBal ? b_t0 : G + 1;
        int c = 0;
        // Every epi warp passes the pieces' boundaries, also one that gave up (its warps decide on
        // their own inside the loop): the hand-offs' named barriers then always see all four.
#pragma unroll 1
        for (int piece = 0; piece < (kBal ? 3 : 1); ++piece) {
            if (kBal && piece == 2 && b_t0 < G) {
                // the tail run starts from the previous CTA's hand-off: one thread waits for its
                // flag (bounded) and clears it for the next launch; the barrier orders the other
                // threads' reads after its acquire
                unsigned long long *f = p.flags + blockIdx.x - 1;
                bool got = true;
                if (ok && threadIdx.x == 10 * 32) {
                    got = handoff_wait(f, p.epoch, abort_flag);
                    if (got) *reinterpret_cast<volatile unsigned long long *>(f) = 0ull;
                }
                if (named_barrier_or(3, 128, !ok || !got)) ok = false;  // the epi gives up together
            }
            if (kBal && piece == 2 && b_t0 < G && ok) {
                const float4 *x = reinterpret_cast<const float4 *>(p.summary + (size_t)(blockIdx.x - 1) * kD * kD +
                                                                   (size_t)row * kD + ch0);
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float4 w = __ldcg(x + j);  // from L2: another SM wrote it
                    S[4 * j] = w.x;
                    S[4 * j + 1] = w.y;
                    S[4 * j + 2] = w.z;
                    S[4 * j + 3] = w.w;
                }
            }
            const int c_end = piece == 0 ? cut0 : (piece == 1 ? cut1 : G + 1);
            for (; ok && c < c_end; ++c) {
                if (c < G) {
                    const int sl = c % kSlots, bb = c & 1;
                    const uint32_t ph = (c >> 1) & 1;
                    const StreamPos ps = pos(c);
                    if (ps.start) {  // a run of a unit starts: its state (every key half)
                        if (kBal && ps.hin) {
                            // S holds the previous CTA's hand-off (taken before this piece)
                        } else if (!kSplit || kSum || ps.seg == 0) {
#pragma unroll
                            for (int j = 0; j < 32; ++j) S[j] = 0.f;
                            if constexpr (NH == 2) {
#pragma unroll
                                for (int j = 0; j < 32; ++j) So[j] = 0.f;
                            }
                        } else if constexpr (kSplit) {
                            if (MODE != kSplitFull || c != 0) {  // (c == 0: S holds the prologue's fold)
                                start_state(S, 0, ps);
                                if constexpr (NH == 2) start_state(So, 1, ps);
                            }
                        }
                        dp = dpo = 1.f;
                    }
                    bool fail = !mbar_wait(&bars[BAR_REFS + sl], (c / kSlots) & 1, abort_flag, kWaitLimitNs);
                    // buffer bb was last read by O(c-2) (epi outputs with one key half: observed by
                    // the readout of the previous iteration already)
                    if (!kSum && (NH == 2 || kGenOut) && c >= 2)
                        fail = fail || !mbar_wait(&bars[BAR_OFULL + bb], ph ^ 1, abort_flag, kWaitLimitNs);
                    if (__any_sync(0xffffffffu, fail || *abort_flag != 0u)) {  // the warp leaves together
                        ok = false;
                        break;
                    }
                    const float *ref = reinterpret_cast<const float *>(smem + kOffRef) + sl * kRefFloats;
                    const bool fold = (mode_s[sl] == kModeF16);
                    const float c1 = fold ? ref[2 * kD + row] : 1.f;
                    const float c2 = fold ? ref[3 * kD + row] : 1.f;
                    const float dc = decay_s[sl * kD + row];
                    if (!kSum) {
                        // S'_[c] = Diag(c1) S_[c] (fp16, MN-major B of the readout)
                        uint8_t *sb = smem + kOffS + bb * kTile16;
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            *reinterpret_cast<uint4 *>(sb + sw128(row, (ch0 + 8 * q) * 2)) = make_uint4(
                                h2bits(S[8 * q + 0] * c1, S[8 * q + 1] * c1), h2bits(S[8 * q + 2] * c1, S[8 * q + 3] * c1),
                                h2bits(S[8 * q + 4] * c1, S[8 * q + 5] * c1), h2bits(S[8 * q + 6] * c1, S[8 * q + 7] * c1));
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&bars[BAR_ORDY + bb]);  // with the outputs of c-2 read out
                    }
                    // state carry: S_[c+1] = Diag(d_c) S_[c] + Diag(c2) U_c
                    fail = !mbar_wait(&bars[BAR_UFULL + bb], ph, abort_flag, kWaitLimitNs);
                    if (__any_sync(0xffffffffu, fail)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    if constexpr (NH == 2) {  // two states live: read U in halves to save registers
#pragma unroll
                        for (int hf = 0; hf < 2; ++hf) {
                            uint32_t r[16];
                            tmem_ld_16x32bx2_x16(tmem + lane_base + kColU + bb * 64 + 16 * hf, r);
                            tmem_ld_wait();
#pragma unroll
                            for (int j = 0; j < 16; ++j) S[16 * hf + j] = fmaf(dc, S[16 * hf + j], c2 * __uint_as_float(r[j]));
                        }
                    } else {
                        uint32_t r[32];
                        tmem_ld_16x32bx2_x16(tmem + lane_base + kColU + bb * 64 + 0, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
                        tmem_ld_16x32bx2_x16(tmem + lane_base + kColU + bb * 64 + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < 32; ++j) S[j] = fmaf(dc, S[j], c2 * __uint_as_float(r[j]));
                    }
                    tc_fence_before();
                    if (kSum) {
                        dp *= dc;
                        if (ps.cl == L - 1) {  // the segment's summary
                            float *base = p.summary + ((size_t)ps.bh * (p.nseg - 1) + ps.seg) * sum_stride;
                            float4 *dst = reinterpret_cast<float4 *>(base + (size_t)(64 * ps.a + row) * kDv + 64 * ps.vb + ch0);
#pragma unroll
                            for (int j = 0; j < 8; ++j) dst[j] = make_float4(S[4 * j], S[4 * j + 1], S[4 * j + 2], S[4 * j + 3]);
                            if (ps.vb == 0 && hc == 0) base[(size_t)kDk * kDv + 64 * ps.a + row] = dp;
                        }
                    } else if (ps.c == N - 1 && p.final_state != nullptr && 64 * ps.a + row < p.Dk) {
                        // the sequence's final state [Dk][Dv] (padded channels and columns stay behind)
                        const int col0 = 64 * ps.vb + ch0;
                        float4 *dst = reinterpret_cast<float4 *>(p.final_state + ((size_t)ps.bh * p.Dk + 64 * ps.a + row) * p.Dv + col0);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            if (col0 + 4 * j < p.Dv) dst[j] = make_float4(S[4 * j], S[4 * j + 1], S[4 * j + 2], S[4 * j + 3]);
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bars[BAR_PURDY + bb]);  // U(c) drained: counts for chunk c + 2
                    if constexpr (NH == 2) {  // the other key half comes next
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            const float t = S[j];
                            S[j] = So[j];
                            So[j] = t;
                        }
                        const float t = dp;
                        dp = dpo;
                        dpo = t;
                    }
                }
                if (!kSum && !kGenOut && c >= nh && c % nh == 0) {
                    // outputs of the real chunk whose last key half is c-1
                    const int co = c - 1, ob = (co / nh) & 1;
                    const bool fail = !mbar_wait(&bars[BAR_OFULL + (co & 1)], (co >> 1) & 1, abort_flag, kWaitLimitNs);
                    if (__any_sync(0xffffffffu, fail)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    uint32_t ow[16];  // the row's 32 outputs packed in pairs
#pragma unroll
                    for (int hf = 0; hf < 2; ++hf) {
                        uint32_t r[16];
                        tmem_ld_16x32bx2_x16(tmem + lane_base + kColO + ob * 64 + 16 * hf, r);
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < 8; ++j) ow[8 * hf + j] = Elem<E>::pack(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1]));
                    }
                    tc_fence_before();
                    const StreamPos po = pos(co);
                    const int b = fdiv(po.bh, p.fd_H), h = po.bh - b * p.H;
                    const int t = walk_token(p.order, p.T, p.fd_gh, p.grid_w, chunk_w0(p.order, p.T, po.c) + row);
                    if (t >= 0) {  // the row's columns inside Dv (padded columns stay behind)
                        const int col0 = 64 * po.vb + ch0;
                        uint4 *dst = reinterpret_cast<uint4 *>(out + (((size_t)b * p.T + t) * p.H + h) * p.Dv + col0);
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            if (col0 + 8 * q < p.Dv) dst[q] = make_uint4(ow[4 * q], ow[4 * q + 1], ow[4 * q + 2], ow[4 * q + 3]);
                    }
                }
            }
            if (kBal && piece == 0 && b_chi > 0 && named_barrier_or(3, 128, !ok)) ok = false;
            if (kBal && piece == 0 && b_chi > 0 && ok) {
                // the state at the end of the head run -> the next CTA
                float4 *dst = reinterpret_cast<float4 *>(p.summary + (size_t)blockIdx.x * kD * kD + (size_t)row * kD + ch0);
#pragma unroll
                for (int j = 0; j < 8; ++j) dst[j] = make_float4(S[4 * j], S[4 * j + 1], S[4 * j + 2], S[4 * j + 3]);
                // the epi's four warps wrote their rows; one thread fences (for them all, after the
                // barrier) and sets the flag, so only its warp waits for its stores in flight
                named_barrier_sync(3, 128);
                if (threadIdx.x == 10 * 32) {
                    __threadfence();
                    *reinterpret_cast<volatile unsigned long long *>(p.flags + blockIdx.x) = p.epoch;
                }
            }
        }
        if (!ok) record_timeout(abort_flag);
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
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}

// Row orders: dims (D, H, T, 1, B), box (64, 1, rows, 1, 1).
// Column orders: dims (D, H, W, Hg, B), box (64, 1, 1, rows, 1).
// D is the tensor's row width (Dk or Dv); a box covers 64 channels at x = 0 or 64.
// L2 promotion of 128 bytes, the width of a box row: with 256 bytes every row also fetched
// the neighbouring head's piece of the token row, which the balanced schedule reads much
// later, so DRAM reads rose to 1.38x the input bytes (batched 40x40, H = 12, B = 32: 128-byte
// promotion 1.02x faster there, equal on the other workloads).
bool encode_map(CUtensorMap *m, const void *ptr, const Problem &p, int width, int rows) {
    auto enc = get_encode();
    if (!enc) return false;
    const cuuint64_t es = 2, D = static_cast<cuuint64_t>(width);
    const bool col = (p.order >> 1) != 0;
    cuuint64_t dims[5] = {D, (cuuint64_t)p.H, 0, 0, (cuuint64_t)p.B};
    cuuint64_t strides[4] = {D * es, (cuuint64_t)p.H * D * es, 0, (cuuint64_t)p.T * p.H * D * es};
    cuuint32_t box[5] = {64, 1, 1, 1, 1}, estr[5] = {1, 1, 1, 1, 1};
    if (!col) {
        dims[2] = (cuuint64_t)p.T;
        dims[3] = 1;
        strides[2] = (cuuint64_t)p.T * p.H * D * es;
        box[2] = (cuuint32_t)rows;
    } else {
        dims[2] = (cuuint64_t)p.grid_w;
        dims[3] = (cuuint64_t)p.grid_h;
        strides[2] = (cuuint64_t)p.grid_w * p.H * D * es;
        box[3] = (cuuint32_t)rows;
    }
    const CUtensorMapDataType dt = p.dtype == 1 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    return enc(m, dt, 5, const_cast<void *>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

PFN_cuTensorMapEncodeIm2col_v12000 get_encode_im2col() {
    static PFN_cuTensorMapEncodeIm2col_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void *f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeIm2col", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeIm2col_v12000>(f);
    });
    return fn;
}

// Column orders' walk map: the tensor [B][T][H][D] (T = Hg x W tokens, row-major) seen as the
// im2col dims (D, Hg, W, H, B), grid rows fastest: an im2col load of 64 pixels from (y, x, h, b)
// walks down column x and on into the next columns, exactly the column scan.  64 channels per
// pixel at c0 = 0 or 64 (channels past D load as zero); no filter window (all corners 0).
bool encode_col_map(CUtensorMap *m, const void *ptr, const Problem &p, int H, int width) {
    auto enc = get_encode_im2col();
    if (!enc) return false;
    const cuuint64_t es = 2, D = static_cast<cuuint64_t>(width);
    cuuint64_t dims[5] = {D, (cuuint64_t)p.grid_h, (cuuint64_t)p.grid_w, (cuuint64_t)H, (cuuint64_t)p.B};
    cuuint64_t strides[4] = {(cuuint64_t)p.grid_w * H * D * es, (cuuint64_t)H * D * es, D * es,
                             (cuuint64_t)p.T * H * D * es};
    int lower[3] = {0, 0, 0}, upper[3] = {0, 0, 0};
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    const CUtensorMapDataType dt = p.dtype == 1 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    return enc(m, dt, 5, const_cast<void *>(ptr), dims, strides, lower, upper, 64, kC, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Gate producer: W2 [H][r][Dk] as dims (Dk, r, H, 1, 1), box (64 channels, r rows): one head's
// block lands as r rows of 128 bytes (SW128, MN-major B of Z = a W2); channels past Dk load as 0.
bool encode_w2_map(CUtensorMap *m, const void *w2, int H, int Dk, int dtype) {
    auto enc = get_encode();
    if (!enc) return false;
    const cuuint64_t es = 2;
    cuuint64_t dims[5] = {(cuuint64_t)Dk, (cuuint64_t)kRank, (cuuint64_t)H, 1, 1};
    cuuint64_t strides[4] = {(cuuint64_t)Dk * es, (cuuint64_t)kRank * Dk * es, (cuuint64_t)H * kRank * Dk * es,
                             (cuuint64_t)H * kRank * Dk * es};
    cuuint32_t box[5] = {64, (cuuint32_t)kRank, 1, 1, 1}, estr[5] = {1, 1, 1, 1, 1};
    const CUtensorMapDataType dt = dtype == 1 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    return enc(m, dt, 5, const_cast<void *>(w2), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Encoded maps are cached per (pointers, shape, order, dtype): a repeated call
// reuses them instead of encoding the maps again.
struct MapKey {
    const void *ptr[kTensors];
    int B, H, grid_h, grid_w, order, dtype, Dk, Dv;
    bool operator==(const MapKey &o) const { return std::memcmp(this, &o, sizeof(MapKey)) == 0; }
};
struct MapEntry {
    MapKey key;
    CUtensorMap maps[kTensors][kHeights];
    CUtensorMap cmaps[kTensors];  // column orders only
};
std::mutex g_map_mutex;
std::list<MapEntry> g_map_cache;  // most recent first
constexpr size_t kMapCacheSize = 32;

bool get_maps(const Problem &p, CUtensorMap (&out)[kTensors][kHeights], CUtensorMap (&cout)[kTensors]) {
    MapKey key;
    std::memset(&key, 0, sizeof(key));
    key.ptr[T_Q] = p.q;
    key.ptr[T_K] = p.k;
    key.ptr[T_V] = p.v;
    key.ptr[T_G] = p.g;
    key.B = p.B;
    key.H = p.H;
    key.grid_h = p.grid_h;
    key.grid_w = p.grid_w;
    key.order = p.order;
    key.dtype = p.dtype;
    key.Dk = p.Dk;
    key.Dv = p.Dv;
    std::lock_guard<std::mutex> lock(g_map_mutex);
    for (auto it = g_map_cache.begin(); it != g_map_cache.end(); ++it) {
        if (it->key == key) {
            std::memcpy(out, it->maps, sizeof(out));
            std::memcpy(cout, it->cmaps, sizeof(cout));
            g_map_cache.splice(g_map_cache.begin(), g_map_cache, it);
            return true;
        }
    }
    MapEntry e;
    e.key = key;
    for (int t = 0; t < kTensors; ++t)
        for (int hi = 0; hi < kHeights; ++hi)
            if (!encode_map(&e.maps[t][hi], key.ptr[t], p, t == T_V ? p.Dv : p.Dk, box_height(hi))) return false;
    std::memset(e.cmaps, 0, sizeof(e.cmaps));
    if ((p.order >> 1) != 0)
        for (int t = 0; t < kTensors; ++t)
            if (!encode_col_map(&e.cmaps[t], key.ptr[t], p, p.H, t == T_V ? p.Dv : p.Dk)) return false;
    std::memcpy(out, e.maps, sizeof(out));
    std::memcpy(cout, e.cmaps, sizeof(cout));
    g_map_cache.push_front(e);
    if (g_map_cache.size() > kMapCacheSize) g_map_cache.pop_back();
    return true;
}

template <typename E, int NH, int NV, int MODE, bool GENOUT = false, bool GP = false, bool GATED = false>
cudaError_t launch_kernel(dim3 grid, const TcParams &tp, cudaStream_t stream, bool pdl = false) {
    // the shared-memory opt-in, once per process and device (setting it again is harmless)
    static std::atomic<unsigned long long> set_on_devices(0);
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(set_on_devices.load(std::memory_order_relaxed) & bit)) {
        e = cudaFuncSetAttribute(gla_tc_kernel<E, NH, NV, MODE, GENOUT, GP, GATED>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemBytes);
        if (e != cudaSuccess) return e;
        set_on_devices.fetch_or(bit);
    }
    if (MODE == kSplitFull && pdl) {
        // launched right after its summary pass: it may start while that grid runs (programmatic
        // dependent launch) and waits for it before it reads the summaries
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr.val.programmaticStreamSerializationAllowed = 1;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = grid;
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = kSmemBytes;
        cfg.stream = stream;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, gla_tc_kernel<E, NH, NV, MODE, GENOUT, GP, GATED>, tp);
    }
    gla_tc_kernel<E, NH, NV, MODE, GENOUT, GP, GATED><<<grid, kThreads, kSmemBytes, stream>>>(tp);
    return cudaSuccess;
}

// One instantiation per (element type, key halves, value slices, pass).
// gen_out: outputs stored by the gen warpgroups (fp16, one key half, outputs only)
template <typename E, int MODE>
cudaError_t launch_shape(dim3 grid, const TcParams &tp, cudaStream_t stream, bool gen_out = false, bool pdl = false) {
    if constexpr (std::is_same<E, __half>::value && MODE != kSummary) {
        if (gen_out && tp.nh == 1)
            return tp.nv == 1 ? launch_kernel<E, 1, 1, MODE, true>(grid, tp, stream, pdl)
                              : launch_kernel<E, 1, 2, MODE, true>(grid, tp, stream, pdl);
    }
    if (tp.nh == 1)
        return tp.nv == 1 ? launch_kernel<E, 1, 1, MODE>(grid, tp, stream, pdl)
                          : launch_kernel<E, 1, 2, MODE>(grid, tp, stream, pdl);
    return tp.nv == 1 ? launch_kernel<E, 2, 1, MODE>(grid, tp, stream, pdl)
                      : launch_kernel<E, 2, 2, MODE>(grid, tp, stream, pdl);
}

// kBalanced CTAs wait for their neighbour's hand-off: a cooperative launch guarantees
// that every CTA of the grid is resident at once.
template <typename E, int NV>
cudaError_t launch_balanced(dim3 grid, const TcParams &tp, cudaStream_t stream) {
    static std::atomic<unsigned long long> set_on_devices(0);
    auto kernel = gla_tc_kernel<E, 1, NV, kBalanced, false>;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(set_on_devices.load(std::memory_order_relaxed) & bit)) {
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
        if (e != cudaSuccess) return e;
        set_on_devices.fetch_or(bit);
    }
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeCooperative;
    attr.val.cooperative = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = stream;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, tp);
}

// Launch epochs of the balanced schedule: nonzero and never repeated within a process,
// so a flag left by an earlier launch (or garbage in a fresh workspace) is not taken for
// this launch's hand-off; flags are also cleared once read, which keeps graph replays of
// one captured launch correct.
unsigned long long next_epoch() {
    static std::atomic<unsigned long long> ctr(
        (static_cast<unsigned long long>(std::chrono::steady_clock::now().time_since_epoch().count()) << 16) | 1ull);
    return ctr.fetch_add(2ull);  // odd, so never 0
}

cudaError_t sm_count(int *n_sm) {  // cached per device
    static std::atomic<int> cache[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) {
        const int v = cache[dev].load(std::memory_order_relaxed);
        if (v > 0) {
            *n_sm = v;
            return cudaSuccess;
        }
    }
    e = cudaDeviceGetAttribute(n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess && dev >= 0 && dev < 64) cache[dev].store(*n_sm, std::memory_order_relaxed);
    return e;
}

// Key channels and value columns are processed in 64-wide halves and slices; a
// narrower last one is zero-padded by the TMA loads (boxes past the tensor's row).
int pad64(int d) { return (d + 63) / 64 * 64; }

// Segments per sequence.  A launch whose work units fill fewer than half of the
// SMs splits every sequence into segments of `len` chunks, so that the split
// launch still fits one wave (units x ceil(N / len) <= SMs).  The split's critical
// path is the last segment: `len` chunks in each of the two passes, plus the fold
// of the nseg - 1 earlier summaries into its start state, which the output pass's
// CTAs do together with many loads in flight.  A graph-replayed sweep of every
// length on a GB300 (batch-1 and small-batch shapes, 64 <= N <= 256 chunks) fitted
// about 1.95 us per chunk of length against 0.13 us per segment, so the length
// minimises 15 len + ceil(N / len), at least kMinSegChunks.  Sequences of at most
// kMaxUnsplitChunks chunks stay whole (5 chunks: 11.4 us whole, 13.4 us split).
// The last segment may be shorter than the others: its chunks past the sequence
// load as zeros (no key, decay 1), so they leave the state unchanged, and their
// outputs are not stored.
struct Split {
    int nseg;  // segments per sequence (1: no split)
    int len;   // chunks per segment
};

Split choose_split(const Problem &p, int n_sm) {
    const long long N = (p.T + kC - 1) / kC;
    const long long units = (long long)p.B * p.H * (pad64(p.Dv) / 64);
    const Split none{1, static_cast<int>(N)};
    if (units * 2 > n_sm || N <= kMaxUnsplitChunks) return none;
    Split best = none;
    long long best_cost = -1;
    for (long long L = kMinSegChunks; L < N; ++L) {
        const long long d = (N + L - 1) / L;
        if (units * d > n_sm) continue;
        const long long cost = 15 * L + d;
        if (best_cost < 0 || cost < best_cost) {
            best = Split{static_cast<int>(d), static_cast<int>(L)};
            best_cost = cost;
        }
    }
    return best;
}

// Balanced ranges (one key half, unsplit): when the units are more than the SMs and a
// round-robin deal would take at least 1.1 times the chunks per CTA of an even split,
// every CTA takes an equal contiguous range of chunks instead.  Measured on a GB300
// (graph-replayed, interleaved, against whole units): B = 32, H = 12, 40 x 40 (384 units,
// ratio 1.19) 1.10x in bf16 and 1.05x in fp16; B = 16, H = 12, 80 x 80 (192 units, ratio
// 1.58) 1.52x; B = 24 (288 units, ratio 1.06) 0.98x and B = 38 (456 units, ratio 1.00)
// 0.96x, hence the threshold.  The balanced kernel costs about 6 % a chunk more than the
// round-robin one (the hand-offs and the longer decode).
bool choose_balanced(const Problem &p, int n_sm) {
    if (pad64(p.Dk) != 64 || n_sm < 1) return false;
    const long long units = (long long)p.B * p.H * (pad64(p.Dv) / 64);
    if (units <= n_sm) return false;
    if (units * ((p.T + kC - 1) / kC) > 0x7fffffffLL) return false;  // the decode's flattened chunk index is an int
    const long long waves = (units + n_sm - 1) / n_sm;
    return waves * n_sm * 10 >= units * 11;  // ceil(U / SMs) >= 1.1 U / SMs
}

// hand-off states ([64][64] fp32 per CTA) and flags (one 64-bit word per CTA)
size_t handoff_bytes(int n_sm) {
    return (size_t)n_sm * 64 * 64 * sizeof(float) + (size_t)n_sm * sizeof(unsigned long long);
}

size_t summary_bytes(const Problem &p, int nseg) {
    if (nseg <= 1) return 0;
    return (size_t)p.B * p.H * (nseg - 1) * ((size_t)pad64(p.Dk) * pad64(p.Dv) + pad64(p.Dk)) * sizeof(float);
}

}  // namespace

int tc_chunk_boxes(int order, int T, int grid_h, int grid_w, int c, int *boxes, int cap) {
    int n = 0;
    chunk_load_boxes(order, T, make_fastdiv(grid_h), grid_w, c, [&](int hi, int row, int c2, int c3) {
        if (n < cap) {
            boxes[4 * n + 0] = box_height(hi);
            boxes[4 * n + 1] = row;
            boxes[4 * n + 2] = c2;
            boxes[4 * n + 3] = c3;
        }
        ++n;
    });
    return n;
}

int tc_balanced_walk(int n_units, int N, int grid, int cta, int *entries, int cap, int *head) {
    const BalRange r = bal_range(N, n_units, cta, grid);
    const FastDiv fn = make_fastdiv(N);
    for (int v = 0; v < r.G && v < cap; ++v) {
        const StreamPos ps = stream_pos_bal(v, N, 0, r.base_head, r.base_full, r.base_tail, r.c_hi, r.t0, fn);
        entries[4 * v + 0] = ps.bh;  // with one value slice per unit, the unit itself
        entries[4 * v + 1] = ps.c;
        entries[4 * v + 2] = ps.start ? 1 : 0;
        entries[4 * v + 3] = ps.hin ? 1 : 0;
    }
    *head = r.c_hi;
    return r.G;
}

int tc_chunk_walk(int order, int T, int grid_h, int c, int *x0, int *y0) {
    return chunk_walk_start(order, T, make_fastdiv(grid_h), c, x0, y0) ? 1 : 0;
}

void tc_split_plan(const Problem &p, int n_sm, int *nseg, int *seg_len) {
    const Split sp = choose_split(p, n_sm);
    *nseg = sp.nseg;
    *seg_len = sp.len;
}

size_t tc_workspace_bytes(const Problem &p) {
    int n_sm = 0;
    if (sm_count(&n_sm) != cudaSuccess) return 0;
    const int nseg = choose_split(p, n_sm).nseg;
    if (nseg > 1) return summary_bytes(p, nseg);
    return choose_balanced(p, n_sm) ? handoff_bytes(n_sm) : 0;
}

int tc_balanced_plan(const Problem &p, int n_sm) { return choose_split(p, n_sm).nseg == 1 && choose_balanced(p, n_sm); }

bool tc_supported(const Problem &p) {
    if (p.dtype != 1 && p.dtype != 2) return false;       // fp16 / bf16 operands only
    // rows of 16-byte multiples (TMA strides); up to two 64-wide halves / slices
    if (p.Dk % 8 != 0 || p.Dv % 8 != 0 || p.Dk > 128 || p.Dv > 128) return false;
    if (p.T > (1 << 30)) return false;
    return get_encode() != nullptr;
}

cudaError_t launch_tc(const Problem &p, cudaStream_t stream, void *workspace, size_t workspace_bytes, Ran *ran,
                      const Gate *gate, bool *gate_fused) {
    if (gate_fused) *gate_fused = false;
    TcParams tp;
    if (!get_maps(p, tp.maps, tp.cmaps)) return cudaErrorInvalidValue;
    int n_sm = 0;
    cudaError_t e = sm_count(&n_sm);
    if (e != cudaSuccess) return e;
    tp.out = p.out;
    tp.final_state = p.final_state;
    tp.H = p.H;
    tp.grid_h = p.grid_h;
    tp.fd_H = make_fastdiv(p.H);
    tp.fd_gh = make_fastdiv(p.grid_h);
    tp.grid_w = p.grid_w;
    tp.order = p.order;
    tp.T = static_cast<int>(p.T);
    tp.n_chunks = static_cast<int>((p.T + kC - 1) / kC);
    tp.Dk = p.Dk;
    tp.Dv = p.Dv;
    tp.nh = pad64(p.Dk) / 64;
    tp.nv = pad64(p.Dv) / 64;
    Split sp = choose_split(p, n_sm);
    Ran r;
    const bool bal = choose_balanced(p, n_sm);
    r.planned = sp.nseg > 1 ? kRanTcSplit : (bal ? kRanTcBalanced : kRanTc);
    r.ran = kRanTc;
    if (sp.nseg > 1 && (workspace == nullptr || workspace_bytes < summary_bytes(p, sp.nseg)))
        sp = Split{1, tp.n_chunks};
    if (sp.nseg > 1) r.ran = kRanTcSplit;
    const int nseg = sp.nseg;
    tp.nseg = nseg;
    tp.seg_len = sp.len;
    tp.fd_L = make_fastdiv(sp.len);
    tp.fd_per = make_fastdiv(sp.len * tp.nh);
    tp.summary = static_cast<float *>(workspace);
    tp.flags = nullptr;
    tp.epoch = 0;
    // test hook for the timeout path (no fault: the data of one chunk simply never arrives)
    const char *drop = std::getenv("GTR_GLA_TEST_DROP_LOAD");
    tp.drop_load = (drop != nullptr && drop[0] == '1') ? 1 : 0;
    const int seqs = static_cast<int>(p.B * p.H) * tp.nv;  // (sequence, value slice) pairs
    const bool half = p.dtype == 1;
    // persistent: one CTA per SM, each walking its share of the work units
    unsigned sum_ctas = 0;
    if (nseg > 1) {  // pass 1: end state from zero and total decay of segments 0 .. nseg-2
        tp.nsu = nseg - 1;
        tp.fd_nsu = make_fastdiv(tp.nsu);
        tp.n_units = seqs * tp.nsu;
        const dim3 grid(static_cast<unsigned>(tp.n_units < n_sm ? tp.n_units : n_sm));
        sum_ctas = grid.x;
        e = half ? launch_shape<__half, kSummary>(grid, tp, stream) : launch_shape<__nv_bfloat16, kSummary>(grid, tp, stream);
        if (e != cudaSuccess) return e;
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    tp.nsu = nseg;
    tp.fd_nsu = make_fastdiv(nseg);
    tp.n_units = seqs * nseg;
    if (nseg == 1 && bal && workspace != nullptr && workspace_bytes >= handoff_bytes(n_sm)) {
        // equal contiguous chunk ranges, one CTA per SM
        r.ran = kRanTcBalanced;
        if (ran) *ran = r;
        tp.flags = reinterpret_cast<unsigned long long *>(static_cast<char *>(workspace) + (size_t)n_sm * 64 * 64 * sizeof(float));
        tp.epoch = next_epoch();
        tp.bal_n = make_fastdiv(tp.n_chunks);
        const dim3 bgrid(static_cast<unsigned>(n_sm));
        if (half)
            e = tp.nv == 1 ? launch_balanced<__half, 1>(bgrid, tp, stream) : launch_balanced<__half, 2>(bgrid, tp, stream);
        else
            e = tp.nv == 1 ? launch_balanced<__nv_bfloat16, 1>(bgrid, tp, stream)
                           : launch_balanced<__nv_bfloat16, 2>(bgrid, tp, stream);
        if (e != cudaSuccess) return e;
        return cudaGetLastError();
    }
    if (ran) *ran = r;
    // output gate fused into the stores: one key half and one value slice (a row's Dv outputs in
    // one thread pair), outputs stored by the gen warpgroups, for launches of few sequences (at
    // most half as many units as SMs), where it saves a launch: measured on a GB300 (graph
    // replays, interleaved) 3.5 % faster at B = 1, H = 6, 40 x 40, but 1.14-1.26x slower than
    // the separate gate kernel at B = 32, H = 12, 40 x 40 and B = 8, H = 16, 80 x 80, where the
    // gate's work lands on the gen warpgroups' share of the critical chain
    const bool fuse = gate != nullptr && tp.nh == 1 && tp.nv == 1 && 2 * seqs <= n_sm;
    if (fuse) {
        tp.gate_r = gate->r;
        tp.gate_w = gate->w;
        tp.gate_eps = gate->eps;
        if (gate_fused) *gate_fused = true;
    }
    // the fewest CTAs that keep the busiest one's unit count: equal shares, and no SM works
    // on a short share while the others finish (measured on a GB300: B = 32, H = 12, 40 x 40,
    // bf16, 384 units on 128 CTAs instead of 152 ran 3 % faster, the same at fp16)
    const int per_cta = (tp.n_units + n_sm - 1) / n_sm;
    const dim3 grid(static_cast<unsigned>((tp.n_units + per_cta - 1) / per_cta));
    // outputs from the gen warpgroups: fp16 launches of at most one wave (measured on a GB300:
    // +3 to +6 % there; with several units per CTA, or bf16, the epi storing them was faster)
    const bool gen_out = half && tp.n_units <= n_sm;
    // the output pass of a split starts while its summary pass runs when both fit on the SMs at
    // once (measured on a GB300: 1.04-1.06x at B = 1, H = 6, 40 x 40, 72 + 78 CTAs; with
    // 96 + 128 CTAs at B = 2, H = 8, 128 x 128, Dk = Dv = 128, 0.95x)
    const bool pdl = nseg > 1 && sum_ctas + grid.x <= static_cast<unsigned>(n_sm);
    if (fuse) {
        if (nseg > 1)
            e = half ? launch_kernel<__half, 1, 1, kSplitFull, true, false, true>(grid, tp, stream, pdl)
                     : launch_kernel<__nv_bfloat16, 1, 1, kSplitFull, true, false, true>(grid, tp, stream, pdl);
        else
            e = half ? launch_kernel<__half, 1, 1, kFull, true, false, true>(grid, tp, stream)
                     : launch_kernel<__nv_bfloat16, 1, 1, kFull, true, false, true>(grid, tp, stream);
        if (e != cudaSuccess) return e;
        return cudaGetLastError();
    }
    if (nseg > 1)
        e = half ? launch_shape<__half, kSplitFull>(grid, tp, stream, gen_out, pdl)
                 : launch_shape<__nv_bfloat16, kSplitFull>(grid, tp, stream, false, pdl);
    else
        e = half ? launch_shape<__half, kFull>(grid, tp, stream, gen_out)
                 : launch_shape<__nv_bfloat16, kFull>(grid, tp, stream);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

bool tc_gate_supported(const Problem &p, int rank) {
    // one 64-channel key half, the paper's rank, and units of at least four chunks (the W2 block
    // of a unit is double-buffered by unit parity, see the producer)
    return tc_supported(p) && p.Dk <= 64 && rank == kRank && p.T > 3 * kC;
}

cudaError_t launch_tc_gate(const Problem &p, const GateSource &gs, cudaStream_t stream, Ran *ran) {
    if (!tc_gate_supported(p, kRank) || !(gs.tau > 0.f)) return cudaErrorInvalidValue;
    TcParams tp;
    std::memset(&tp, 0, sizeof(tp));
    // q, k and v as in the plain schedule; the gate tiles' maps then load the projection a
    // ([B, T, r] as a one-head tensor of width r, boxes 64 elements wide: the row's other 48
    // elements are zero-filled, so the a tile has 128-byte rows like the other tiles)
    Problem pq = p;
    pq.g = p.q;
    if (!get_maps(pq, tp.maps, tp.cmaps)) return cudaErrorInvalidValue;
    Problem pa = p;
    pa.H = 1;
    for (int hi = 0; hi < kHeights; ++hi)
        if (!encode_map(&tp.maps[T_G][hi], gs.a_low, pa, kRank, box_height(hi))) return cudaErrorInvalidValue;
    if ((p.order >> 1) != 0 && !encode_col_map(&tp.cmaps[T_G], gs.a_low, p, 1, kRank)) return cudaErrorInvalidValue;
    if (!encode_w2_map(&tp.w2map, gs.w2, p.H, p.Dk, p.dtype)) return cudaErrorInvalidValue;
    tp.gbias = gs.bias;
    tp.tau_inv = 1.f / gs.tau;
    int n_sm = 0;
    cudaError_t e = sm_count(&n_sm);
    if (e != cudaSuccess) return e;
    tp.out = p.out;
    tp.final_state = p.final_state;
    tp.H = p.H;
    tp.grid_h = p.grid_h;
    tp.fd_H = make_fastdiv(p.H);
    tp.fd_gh = make_fastdiv(p.grid_h);
    tp.grid_w = p.grid_w;
    tp.order = p.order;
    tp.T = static_cast<int>(p.T);
    tp.n_chunks = static_cast<int>((p.T + kC - 1) / kC);
    tp.Dk = p.Dk;
    tp.Dv = p.Dv;
    tp.nh = 1;
    tp.nv = pad64(p.Dv) / 64;
    tp.nseg = 1;
    tp.nsu = 1;
    tp.seg_len = tp.n_chunks;
    tp.fd_nsu = make_fastdiv(1);
    tp.fd_L = make_fastdiv(tp.n_chunks);
    tp.fd_per = make_fastdiv(tp.n_chunks);
    const char *drop = std::getenv("GTR_GLA_TEST_DROP_LOAD");
    tp.drop_load = (drop != nullptr && drop[0] == '1') ? 1 : 0;
    tp.n_units = static_cast<int>(p.B * p.H) * tp.nv;
    if (ran) *ran = Ran{kRanTc, kRanTc};
    const int per_cta = (tp.n_units + n_sm - 1) / n_sm;
    const dim3 grid(static_cast<unsigned>((tp.n_units + per_cta - 1) / per_cta));
    const bool gen_out = p.dtype == 1 && tp.n_units <= n_sm;  // as the plain schedule
    if (p.dtype == 1) {
        if (gen_out)
            e = tp.nv == 1 ? launch_kernel<__half, 1, 1, kFull, true, true>(grid, tp, stream)
                           : launch_kernel<__half, 1, 2, kFull, true, true>(grid, tp, stream);
        else
            e = tp.nv == 1 ? launch_kernel<__half, 1, 1, kFull, false, true>(grid, tp, stream)
                           : launch_kernel<__half, 1, 2, kFull, false, true>(grid, tp, stream);
    } else {
        e = tp.nv == 1 ? launch_kernel<__nv_bfloat16, 1, 1, kFull, false, true>(grid, tp, stream)
                       : launch_kernel<__nv_bfloat16, 1, 2, kFull, false, true>(grid, tp, stream);
    }
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

void *tensor_map_encoder() { return reinterpret_cast<void *>(get_encode()); }

cudaError_t read_and_clear_device_status(unsigned int *status) {
    cudaError_t e = cudaMemcpyFromSymbol(status, g_device_status, sizeof(unsigned int));
    if (e != cudaSuccess) return e;
    const unsigned int zero = 0;
    return cudaMemcpyToSymbol(g_device_status, &zero, sizeof(unsigned int));
}

}  // namespace gtr
