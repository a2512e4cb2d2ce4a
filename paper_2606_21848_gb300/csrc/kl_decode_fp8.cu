// Keyless decode over an FP8 value cache (E4M3 codes, one fp32 scale per cached row), on the
// tensor cores for sm_103a.
//
// Same method and split plan as the bf16 decode (routing q_r = q W^R, Section 2.2; one softmax
// over the cached value rows, each row used for the score and for the output, Section 3). The
// tensor cores read the codes as TMA lands them: both products are kind::f8f6f4 MMAs (E4M3 x
// E4M3, fp32 accumulation), so a 128-token tile moves 16 KiB of codes plus 512 B of row scales
// and is never widened:
//
//   scores   S^T = C_t . Q^T     M = 128 tokens, N = 32, K = 128 dims    (C_t K-major)
//   output   O^T = C_t^T . W     M = 128 dims,   N = 32, K = 128 tokens  (C_t MN-major)
//
// The other operands keep more precision than one E4M3 value by being sums of E4M3 terms in
// separate columns: each term is the rounding residual of the previous one times 16, so each
// adds four significant bits. Q holds the routed query (times scale * log2 e) of the 8 heads as
// 4 terms, W the softmax weights times the row scales as 3 terms; head h = 4 hh + k, term j sits
// in score column 16 hh + 4 j + k and output column 16 hh + 4 j + k (output columns 12..15 of
// each half zero). Before the split a power of two brings the operand's largest value below
// 256 (E4M3 reaches 448); it is divided out again after the terms are summed.
//
// The softmax keeps a lazy reference maximum per head: a tile's weights are 2^(s - m) with the
// current reference m, and m moves (rescaling the running sums) only when a score passes it by
// more than 2, so the weights stay at most 4. Most tiles thus need one vote among the compute
// warps instead of an exchange of maxima. The weights' power of two, 2^(6 - e) with every row
// scale so far below 2^e, is lazy the same way, so the output MMAs of all tiles accumulate into
// one O in TMEM; the rare tile that moves a reference or e rescales O there first.
// A row's scale multiplies its score column (s_t = scale_t <q_r, c_t>) and its weight
// (p_t scale_t), so the codes are used as stored.
//
// One CTA per (split, value head g, sequence b); 352 threads, two CTAs per SM:
//   warps 0-7  compute. Warp w reads TMEM lane quarter w % 4 and takes heads 4 (w / 4) .. + 3:
//              routing result and query split (thread = dim); per tile the online softmax in
//              base 2 and the weight split (thread = token), O accumulation (thread = output
//              dim); epilogue (output row or split state). Two warps per lane quarter halve
//              the per-thread work of a tile, which bounds the tile rate.
//   warp 8     producer: W^R[g] (ring stages 0-1) and the group's query rows, then per tile the
//              TMA loads of code pages and bulk copies of their scale rows; for the decode step
//              (kl_decode_step_fp8) it first quantizes the current token's row into the cache
//              when that row falls in the CTA's split, before the loads of the row's tile
//   warp 9     routing and score MMA issuer, TMEM owner
//   warp 10    output MMA issuer; completion of a tile's output MMAs frees its ring stage
// Every wait is bounded (about one second); a wait that runs out raises KL_FLAG_TIMEOUT and
// every role leaves its loop, drains its copies and MMAs, and TMEM is freed.
#include <cuda_fp16.h>
#include <cudaTypedefs.h>
#include <math.h>

#include "kl_fp8_quant.cuh"
#include "kl_internal.cuh"
#include "kl_tc_ptx.cuh"

namespace kl {
namespace {

constexpr int kD = 128;
constexpr int kTile = 128;
constexpr int kJq = 4;                      // E4M3 terms of the routed query
constexpr int kJp = 3;                      // E4M3 terms of the weights
constexpr int kNR = 16;                     // routing MMA N (query rows, padded)
constexpr int kQuarters = 4;                // TMEM lane quarters (warps per head half)
constexpr int kComputeWarps = 8;
constexpr int kComputeThreads = kComputeWarps * 32;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kPvWarp = 10;
constexpr int kThreads = 11 * 32;
constexpr int kStages = 5;
constexpr uint32_t kCodeBytes = kTile * kD;          // 16 KiB of codes per tile
constexpr uint32_t kHalfBytes = 16384;               // one 64-column half of W^R (bf16)
constexpr uint32_t kPBytes = 4096;                   // weight operand buffer (largest shape)
constexpr int kPBuf = 4;                             // weight operands in flight
constexpr uint32_t kTmemCols = 128;
constexpr uint32_t kColS = 0;                        // S[b]: columns 32 b .. 32 b + 31
constexpr uint32_t kColO = 64;                       // O: columns 64 .. 95, summed over tiles
constexpr uint32_t kColR = 96;                       // routing result: 96 .. 111
constexpr float kLazyW = 4.f;                        // reference slack: weights 2^(s - m) <= 4
constexpr uint64_t kTimeoutNs = kDefaultWaitNs;   // bound of the drains
constexpr uint32_t kSleepHintNs = 20000u;         // suspend hint of a wait that did not finish at once
constexpr uint32_t kBarCompute = 1;
constexpr uint32_t kBarComputeAnd = 2;

// Operand shapes for KHH query heads per compute warp (4 when the group has 5..8 heads, 2 when
// it has at most 4, so that no compute warp carries only padded heads). Head h = KHH hh + k
// (hh = warp / 4) and term j sit in score column HS hh + KHH j + k and output column
// HP hh + KHH j + k.
template <int KHH>
struct Fp8Shape {
    static constexpr int NS = 8 * KHH;        // score MMA N: 4 query terms x 2 KHH heads
    static constexpr int NP = 8 * KHH;        // output MMA N: 3 weight terms x 2 KHH heads, padded
    static constexpr int HS = NS / 2;         // score columns of one warp
    static constexpr int HP = NP / 2;         // output columns of one warp
    static constexpr int GS = 8 * NP;         // weight operand: bytes per group of 8 tokens
};

struct __align__(1024) Smem8 {
    // Ring of code tiles as TMA lands them: [128 token rows][128 B], 128B-swizzled. Stages 0
    // and 1 first hold the two 64-column halves of W^R[g] (bf16) for the routing MMA.
    uint8_t codes[kStages][kCodeBytes];
    // Query terms, B operand of the score MMAs: [NS rows n][128 dims], K-major, 128B-swizzled.
    uint8_t qt[32 * 128];
    // Weight terms, B operand of the output MMAs: [16 groups of 8 tokens][NP / 16 blocks of 16
    // columns][8 tokens][16 B], MN-major, no swizzle. During the routing prologue the first one
    // holds the query rows: [64-dim half][16 rows][128 B], K-major, 128B-swizzled.
    uint8_t p[kPBuf][kPBytes];
    float scl[kStages][kTile];         // row scales of each stage's tile, token order
    float red[2][kComputeWarps][8];    // per warp: 4 head maxima (or row sums), the scale max
    uint64_t full[kStages], empty[kStages];
    uint64_t s_full[2], s_empty[2], p_full[kPBuf], o_full[kPBuf];
    uint64_t r_full, qt_full, drain, drain2;
    uint32_t tmem_base;
    int abort;
};

// Warp-collective bounded wait (as in the bf16 decode): false when the CTA is aborting or the
// wait ran out (`limit` ns, about 1 s unless the library's limit was lowered).
// A thread whose phase is not complete sleeps in the try_wait (it wakes when the phase
// completes or the hint runs out) instead of spinning and taking issue slots from the warps
// that share its scheduler.
// The first poll is the plain try_wait (a hinted first poll wakes later when the phase
// completes: 4 % on the 70B batch); kExact (limits below kExactWaitNs) polls with the
// non-blocking test_wait, so that short limits hold exactly.
template <bool kExact>
struct Waiter {
    volatile int *abort;
    int32_t *err;
    uint64_t limit;
    __device__ bool operator()(uint64_t *bar, uint32_t parity) const {
        bool ok = kExact ? ptx::mbar_test_wait(bar, parity) : ptx::mbar_try_wait(bar, parity);
        if (!ok) {
            const uint64_t t0 = ptx::globaltimer();
            while (true) {
                if (kExact ? ptx::mbar_test_wait(bar, parity)
                           : ptx::mbar_try_wait_hint(bar, parity, kSleepHintNs)) {
                    ok = true;
                    break;
                }
                if (*abort) break;
                if (ptx::globaltimer() - t0 > limit) {
                    *abort = 1;
                    raise_flag(err, KL_FLAG_TIMEOUT);
                    break;
                }
            }
        }
        return __all_sync(0xffffffffu, ok);
    }
};

// Warp maximum of a float through the integer reduction unit: the key of a float orders as the
// float does (non-negative floats keep their bits, negative ones flip all but the sign).
__device__ __forceinline__ int order_key(float f) {
    const int i = __float_as_int(f);
    return i >= 0 ? i : i ^ 0x7FFFFFFF;
}
__device__ __forceinline__ float warp_max(float f) {
    const int k = __reduce_max_sync(0xffffffffu, order_key(f));
    return __int_as_float(k >= 0 ? k : k ^ 0x7FFFFFFF);
}

// Two E4M3 codes (low byte first) to two halves (low half first), exact: every E4M3 value is a
// half-precision value.
__device__ __forceinline__ float2 e4m3x2_to_float2(uint32_t two_codes) {
    uint32_t r;
    const uint16_t v = (uint16_t)two_codes;
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(r) : "h"(v));
    return __half22float2(*reinterpret_cast<const __half2 *>(&r));
}

// A power of two 2^(8 - e) with amax < 2^e (so amax * 2^(8 - e) < 256) and its inverse; 1 and 1
// for amax = 0. e is clamped so that both stay normal floats.
__device__ __forceinline__ void pow2_scale(float amax, float &sc, float &inv) {
    int e = (int)((__float_as_uint(amax) >> 23) & 0xFFu) - 126;
    e = max(-100, min(100, e));
    if (!(amax > 0.f)) e = 8;
    sc = __uint_as_float((uint32_t)(127 + 8 - e) << 23);
    inv = __uint_as_float((uint32_t)(127 - 8 + e) << 23);
}

// 2^(8 - e) and 2^(e - 8), e clamped so that both stay normal floats.
__device__ __forceinline__ void pow2_from_exp(int e, float &sc, float &inv) {
    e = max(-100, min(100, e));
    sc = __uint_as_float((uint32_t)(127 + 8 - e) << 23);
    inv = __uint_as_float((uint32_t)(127 - 8 + e) << 23);
}

// An E4M3 value next to x (0 <= x < 448), on the FMA pipe: x rounded to 4 significant bits by
// a Veltkamp split (c = x (2^20 + 1), hv = c - (c - x)), then hv rounded to the multiples of 2^-9
// by adding and subtracting 1.5 * 2^14 (whose spacing is 2^-9). Above 2^-6 hv is an E4M3 value
// and already a multiple of 2^-9, so the second rounding keeps it; below, it lands on the E4M3
// subnormals. The result is exactly representable, so its code conversion is exact, and x minus
// it is exact and at most x / 16 + 2^-10. (The small values matter: the weight scale follows the
// largest row scale seen so far, so many weights sit far below it.)
__device__ __forceinline__ float e4m3_round(float x) {
    // explicit roundings: the compiler must not fuse these into FMAs
    const float c = __fmul_rn(x, 1048577.f);
    const float hv = __fsub_rn(c, __fsub_rn(c, x));
    return __fsub_rn(__fadd_rn(hv, 24576.f), 24576.f);
}

// Packed fp32 pairs: one instruction applies the same IEEE round-to-nearest operation to both
// lanes, so each lane's result is bit for bit that of the scalar operation.
struct F2 {
    float x, y;
};
__device__ __forceinline__ F2 f2(float a, float b) { return F2{a, b}; }
#define KL_F2_OP(name, op)                                                                      \
    __device__ __forceinline__ F2 name(F2 a, F2 b) {                                           \
        F2 d;                                                                                  \
        asm("{\n\t.reg .b64 x, y, z;\n\tmov.b64 x, {%2, %3};\n\tmov.b64 y, {%4, %5};\n\t" op \
            " z, x, y;\n\tmov.b64 {%0, %1}, z;\n\t}"                                            \
            : "=f"(d.x), "=f"(d.y)                                                             \
            : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));                                         \
        return d;                                                                              \
    }
KL_F2_OP(add2, "add.rn.f32x2")
KL_F2_OP(sub2, "sub.rn.f32x2")
KL_F2_OP(mul2, "mul.rn.f32x2")
#undef KL_F2_OP
__device__ __forceinline__ F2 fma2(F2 a, F2 b, F2 c) {
    F2 d;
    asm("{\n\t.reg .b64 x, y, z, w;\n\tmov.b64 x, {%2, %3};\n\tmov.b64 y, {%4, %5};\n\t"
        "mov.b64 z, {%6, %7};\n\tfma.rn.f32x2 w, x, y, z;\n\tmov.b64 {%0, %1}, w;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}

// Byte offset of element (row n, column k) of the query-term operand: [NS rows][128 B],
// K-major, 128B-swizzled (8-row atoms of 1 KiB, 16-byte chunk index XOR row % 8).
__device__ __forceinline__ uint32_t qt_offset(int n, int k) {
    return (n >> 3) * 1024 + (n & 7) * 128 + ((((k >> 4) ^ (n & 7))) << 4) + (k & 15);
}

// D[tmem] (+)= A[smem desc] x B[smem desc], kind::f8f6f4 with E4M3 A and B, fp32 accumulation.
__device__ __forceinline__ void mma_f8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                       uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Instruction descriptor of kind::f8f6f4: fp32 accumulator, E4M3 A and B (format 0), operand
// majorness (0 = K-major, 1 = MN-major), N and M.
__host__ __device__ constexpr uint32_t idesc_f8(uint32_t M, uint32_t N, bool a_mn, bool b_mn) {
    return (1u << 4) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) | ((N >> 3) << 17) |
           ((M >> 4) << 24);
}

// Store 16 consecutive 32-bit columns of the thread's TMEM lane (complete with tmem_wait_st()).
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&u)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(u[0]), "r"(u[1]), "r"(u[2]), "r"(u[3]), "r"(u[4]), "r"(u[5]), "r"(u[6]), "r"(u[7]),
        "r"(u[8]), "r"(u[9]), "r"(u[10]), "r"(u[11]), "r"(u[12]), "r"(u[13]), "r"(u[14]),
        "r"(u[15])
        : "memory");
}

// 8 consecutive 32-bit columns of the thread's TMEM lane (load and wait in one statement).
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, float (&r)[8]) {
    uint32_t u[8];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]),
          "=r"(u[7])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 8; ++i) r[i] = __uint_as_float(u[i]);
}

__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&u)[8]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"r"(
                     taddr),
                 "r"(u[0]), "r"(u[1]), "r"(u[2]), "r"(u[3]), "r"(u[4]), "r"(u[5]), "r"(u[6]),
                 "r"(u[7])
                 : "memory");
}

// N (8 or 16) consecutive columns of the thread's TMEM lane.
template <int N>
__device__ __forceinline__ void tmem_ldn(uint32_t taddr, float (&r)[N]) {
    if constexpr (N == 16) ptx::tmem_ld16(taddr, r);
    else tmem_ld8(taddr, r);
}
template <int N>
__device__ __forceinline__ void tmem_stn(uint32_t taddr, const uint32_t (&u)[N]) {
    if constexpr (N == 16) tmem_st16(taddr, u);
    else tmem_st8(taddr, u);
}

// Barrier `id` over `count` threads that also returns how many of them passed v = true.
__device__ __forceinline__ uint32_t bar_popc(uint32_t id, uint32_t count, bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.popc.u32 %0, %2, %3, p;\n\t}\n"
        : "=r"(r)
        : "r"((uint32_t)v), "r"(id), "r"(count)
        : "memory");
    return r;
}

template <int KHH, bool kAllLive, bool kExact>
__global__ void __launch_bounds__(kThreads, 2)
    decode_fp8_kernel(const __grid_constant__ CUtensorMap cmap,
                      const __grid_constant__ CUtensorMap wmap,
                      const __grid_constant__ CUtensorMap qmap, const DecodeArgs a,
                      const float *__restrict__ v_scales) {
    using Sh = Fp8Shape<KHH>;
    extern __shared__ uint8_t smem_raw[];
    // kAllLive: the group has 2 KHH heads, so no compute warp holds a padded head
    Smem8 &sm = *reinterpret_cast<Smem8 *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                           ~uintptr_t(1023));
    const Geometry &geo = a.geo;
    // A group of more than 8 query heads is served by geo.nhb sibling CTAs, adjacent in
    // blockIdx.x, each for up to 8 of its heads (the second and later reads of a page come
    // from L2).
    const int hb = blockIdx.x % geo.nhb, split = blockIdx.x / geo.nhb;
    const int g = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = min(8, geo.G - 8 * hb);       // query heads of this CTA
    const int qh0 = g * geo.G + 8 * hb;          // its first query head within the sequence
    const bool route = a.w_r != nullptr;      // W^R given; else q is the composed query
    // Ring uses: with routing, uses 0 and 1 are the W^R halves and tile i is use i + 2.
    const int base = route ? 2 : 0;

    const int L_raw = a.seq_lens[b];
    const int pos_raw = a.v_new ? a.positions[b] : -1;
    const int t_begin = split * geo.chunk;
    const int32_t *bt = a.block_table + (size_t)b * geo.max_pages;

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&sm.full[s], 1);
            ptx::mbar_init(&sm.empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&sm.s_full[i], 1);
            ptx::mbar_init(&sm.s_empty[i], kComputeWarps);
        }
        for (int i = 0; i < kPBuf; ++i) {
            ptx::mbar_init(&sm.p_full[i], kComputeWarps);
            ptx::mbar_init(&sm.o_full[i], 1);
        }
        ptx::mbar_init(&sm.r_full, 1);
        ptx::mbar_init(&sm.qt_full, kComputeWarps);
        ptx::mbar_init(&sm.drain, 1);
        ptx::mbar_init(&sm.drain2, 1);
        sm.abort = 0;
        ptx::fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        ptx::tmem_alloc(&sm.tmem_base, kTmemCols);
        ptx::tmem_relinquish();
    }
    if (warp == kProducerWarp && lane == 0) {
        ptx::prefetch_tensormap(&cmap);
        if (route) {
            ptx::prefetch_tensormap(&wmap);
            ptx::prefetch_tensormap(&qmap);
        }
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    // the combine of the split states, launched behind as a programmatic dependent, may start
    // setting up once every CTA is here
    grid_dep_launch();

    int L = L_raw;
    if (L < 0 || L > geo.max_pages * geo.P) {
        if (tid == 0 && split == 0 && g == 0) raise_flag(a.err, KL_FLAG_BAD_LENGTH);
        L = 0;
    }
    const int t_end = min(t_begin + geo.chunk, L);
    const int n_tiles = t_end > t_begin ? (t_end - t_begin + kTile - 1) / kTile : 0;

    // Fused append (kl_decode_step_fp8): the CTA whose split holds row positions[b] quantizes
    // v_new[b][g] into it before the loads of that row's tile (first, when the row lies past the
    // sequence's end), with the arithmetic of kl_append_v_fp8.
    const bool pos_ok = pos_raw >= 0 && pos_raw < geo.max_pages * geo.P;
    if (a.v_new && !pos_ok && tid == 0 && split == 0 && g == 0)
        raise_flag(a.err, KL_FLAG_BAD_POSITION);
    const bool app_owner = a.v_new && pos_ok && pos_raw / geo.chunk == split;
    // the row (page-checked), its codes for this lane and its scale; warp-uniform
    auto quantize_new_row = [&](size_t &row, uint32_t &codes, float &scale) -> bool {
        const int page = bt[pos_raw / geo.P];
        if (page < 0 || page >= geo.num_pages) {
            if (lane == 0) raise_flag(a.err, KL_FLAG_BAD_PAGE);
            return false;
        }
        row = ((size_t)page * geo.Hkv + g) * geo.P + pos_raw % geo.P;
        codes = quantize_row4(
            reinterpret_cast<const uint2 *>(a.v_new + ((size_t)b * geo.Hkv + g) * kD)[lane], scale);
        return true;
    };

    if (n_tiles == 0) {
        if (app_owner && warp == 0) {
            size_t row;
            uint32_t codes;
            float scale;
            if (quantize_new_row(row, codes, scale)) {
                reinterpret_cast<uint32_t *>(a.codes_rw + row * kD)[lane] = codes;
                if (lane == 0) a.scales_rw[row] = scale;
            }
        }
        // an empty split: zero output (direct) or an empty state
        if (tid < kD) {
            for (int h = 0; h < G; ++h) {
                const size_t bh = (size_t)b * geo.Hq + qh0 + h;
                if (a.direct_out) {
                    if (a.out_dtype == KL_FP32) static_cast<float *>(a.out)[bh * kD + tid] = 0.f;
                    else static_cast<__nv_bfloat16 *>(a.out)[bh * kD + tid] = __float2bfloat16_rn(0.f);
                } else {
                    const size_t slot = bh * geo.S + split;
                    a.part_o[slot * kD + tid] = 0.f;
                    if (tid == 0) {
                        a.part_ml[slot * 2] = -INFINITY;
                        a.part_ml[slot * 2 + 1] = 0.f;
                    }
                }
            }
        }
        if (warp == kMmaWarp) ptx::tmem_dealloc(sm.tmem_base, kTmemCols);
        return;
    }

    const uint32_t tmem = sm.tmem_base;
    int issued = 0;                 // ring uses whose copies the producer issued
    const Waiter<kExact> wait{&sm.abort, a.err, a.wait_ns};

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------------ producer ----
        const int P = geo.P;
        const int ppt = kTile / P;                           // pages per tile (<= 8)
        const int first_page = t_begin / P;
        const int end_page = (t_end + P - 1) / P;
        const uint32_t page_bytes = (uint32_t)P * 128u + (uint32_t)P * 4u;
        bool bad = false;
        issued = 0;
        int app_tile = -1;
        size_t app_row = 0;
        uint32_t app_codes = 0;
        float app_scale = 0.f;
        if (app_owner && quantize_new_row(app_row, app_codes, app_scale))
            app_tile = pos_raw < t_end ? (pos_raw - t_begin) / kTile : 0;
        if (route) {
            if (lane == 0) {
                // W^R[g] halves into stages 0 and 1 (MN-major A of the routing MMA); the
                // group's query rows into the first weight buffer (K-major B)
                ptx::mbar_arrive_expect_tx(&sm.full[0], kHalfBytes + 2u * (uint32_t)geo.qbox * 128u);
                ptx::tma_load_2d(sm.codes[0], &wmap, &sm.full[0], 0, g * kD);
                ptx::tma_load_2d(sm.p[0], &qmap, &sm.full[0], 0, b * geo.Hq + qh0);
                ptx::tma_load_2d(sm.p[0] + kNR * 128, &qmap, &sm.full[0], 64, b * geo.Hq + qh0);
                ptx::mbar_arrive_expect_tx(&sm.full[1], kHalfBytes);
                ptx::tma_load_2d(sm.codes[1], &wmap, &sm.full[1], 64, g * kD);
            }
            issued = 2;
            __syncwarp();
        }
        for (int i = 0; i < n_tiles; ++i) {
            const int u = i + base, s = u % kStages, round = u / kStages;
            const int p0 = first_page + i * ppt;
            const bool exists = lane < ppt && p0 + lane < end_page;
            const int page = exists ? bt[p0 + lane] : -1;
            if (round >= 1 && !wait(&sm.empty[s], (round - 1) & 1)) break;
            if (i == app_tile) {
                reinterpret_cast<uint32_t *>(a.codes_rw + app_row * kD)[lane] = app_codes;
                if (lane == 0) a.scales_rw[app_row] = app_scale;
                ptx::fence_proxy_async_global();
                __syncwarp();
            }
            const bool in_range = exists && page >= 0 && page < geo.num_pages;
            if (exists && !in_range) bad = true;
            const unsigned mask = __ballot_sync(0xffffffffu, in_range);
            if (lane == 0) ptx::mbar_arrive_expect_tx(&sm.full[s], __popc(mask) * page_bytes);
            __syncwarp();
            if (in_range) {
                const int row = (page * geo.Hkv + g) * P;
                ptx::tma_load_2d(sm.codes[s] + lane * P * 128, &cmap, &sm.full[s], 0, row);
                ptx::bulk_load(&sm.scl[s][lane * P], v_scales + (size_t)row, (uint32_t)P * 4u,
                               &sm.full[s]);
            }
            issued = u + 1;
        }
        if (__any_sync(0xffffffffu, bad) && lane == 0) raise_flag(a.err, KL_FLAG_BAD_PAGE);

    } else if (warp == kMmaWarp) {
        // ------------------------------------------------- routing and score MMA issuer ----
        bool ok = true;
        if (route) {
            // q_r^T[128 j x 16] = W^R^T (MN-major, bf16) . q^T (K-major rows of the query buffer)
            constexpr uint32_t idesc_r = ptx::idesc_bf16(128, kNR, true, false);
            ok = wait(&sm.full[0], 0);
            ok = ok && wait(&sm.full[1], 0);
            if (ok) {
                ptx::tc_fence_after();
                if (lane == 0) {
                    const uint64_t w_desc = ptx::smem_desc(ptx::smem_addr(sm.codes[0]), kHalfBytes,
                                                           1024, ptx::kSwizzle128B);
                    const uint64_t q_desc =
                        ptx::smem_desc(ptx::smem_addr(sm.p[0]), 16, 1024, ptx::kSwizzle128B);
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        const uint32_t qoff = (kk >> 2) * (kNR * 128) + (kk & 3) * 32;
                        ptx::mma_bf16(tmem + kColR, w_desc + ((kk * 2048) >> 4),
                                      q_desc + (qoff >> 4), idesc_r, kk > 0);
                    }
                    ptx::mma_commit(&sm.r_full);
                    ptx::mma_commit(&sm.empty[0]);      // stages 0 and 1 are free again
                    ptx::mma_commit(&sm.empty[1]);
                }
                __syncwarp();
            }
        }
        ok = ok && wait(&sm.qt_full, 0);
        if (ok) ptx::tc_fence_after();
        constexpr uint32_t idesc_s = idesc_f8(128, Sh::NS, false, false);
        const uint64_t c_desc =
            ptx::smem_desc(ptx::smem_addr(sm.codes[0]), 16, 1024, ptx::kSwizzle128B);
        const uint64_t q_desc = ptx::smem_desc(ptx::smem_addr(sm.qt), 16, 1024, ptx::kSwizzle128B);
        for (int i = 0; ok && i < n_tiles; ++i) {
            const int u = i + base, s = u % kStages, sb = i & 1;
            if (!wait(&sm.full[s], (u / kStages) & 1)) break;
            if (i >= 2 && !wait(&sm.s_empty[sb], ((i >> 1) - 1) & 1)) break;
            ptx::tc_fence_after();
            if (lane == 0) {
                const uint64_t a0 = c_desc + ((s * kCodeBytes) >> 4);
#pragma unroll
                for (int kk = 0; kk < kD / 32; ++kk)
                    mma_f8(tmem + kColS + sb * 32, a0 + ((kk * 32) >> 4), q_desc + ((kk * 32) >> 4),
                           idesc_s, kk > 0);
                ptx::mma_commit(&sm.s_full[sb]);
            }
            __syncwarp();
        }
        if (lane == 0) ptx::mma_commit(&sm.drain);
        __syncwarp();
        const uint64_t t0 = ptx::globaltimer();
        while (!ptx::mbar_try_wait(&sm.drain, 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
        }
    } else if (warp == kPvWarp) {
        // ------------------------------------------------------ output MMA issuer -------
        // A = C^T: the code tile read MN-major (8-token row groups 1 KiB apart); B = W:
        // MN-major, no swizzle (16-column blocks 128 B apart, 8-token groups GS bytes apart)
        constexpr uint32_t idesc_o = idesc_f8(128, Sh::NP, true, true);
        const uint64_t c_desc =
            ptx::smem_desc(ptx::smem_addr(sm.codes[0]), 8192, 1024, ptx::kSwizzle128B);
        const uint64_t p_desc =
            ptx::smem_desc(ptx::smem_addr(sm.p[0]), Sh::GS, 128, ptx::kSwizzleNone);
        for (int j = 0; j < n_tiles; ++j) {
            const int u = j + base, s = u % kStages, pb = j % kPBuf;
            if (!wait(&sm.p_full[pb], (j / kPBuf) & 1)) break;
            ptx::tc_fence_after();
            const int nvalid = min(kTile, t_end - (t_begin + j * kTile));
            const int ksteps = (nvalid + 31) >> 5;
            if (lane == 0) {
                const uint64_t a0 = c_desc + ((s * kCodeBytes) >> 4);
                const uint64_t b0 = p_desc + ((pb * kPBytes) >> 4);
                for (int kk = 0; kk < ksteps; ++kk)
                    mma_f8(tmem + kColO, a0 + ((kk * 4096) >> 4), b0 + ((kk * 4 * Sh::GS) >> 4),
                           idesc_o, (j > 0 || kk > 0) ? 1u : 0u);
                ptx::mma_commit(&sm.o_full[pb]);   // tile j: phase j / kPBuf of o_full[j % kPBuf]
                ptx::mma_commit(&sm.empty[s]);     // the tile's last reader is done
            }
            __syncwarp();
        }
        if (lane == 0) ptx::mma_commit(&sm.drain2);
        __syncwarp();
        const uint64_t t0 = ptx::globaltimer();
        while (!ptx::mbar_try_wait(&sm.drain2, 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
        }
    } else {
        // ------------------------------------------------------------------ compute -----
        // Warp w: TMEM lane quarter q4 = w % 4 (dims / tokens 32 q4 .. 32 q4 + 31) and heads
        // h = 4 hh + k (k = 0..3) with hh = w / 4.
        const int q4 = warp & 3, hh = warp >> 2;
        const int t = q4 * 32 + lane;                       // dim / token / output dim
        const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
        const float sl2 = geo.scale * kLog2e;
        bool ok = true;

        // Routed query: from the routing MMA (TMEM), or the composed query itself.
        float acc[KHH];
#pragma unroll
        for (int k = 0; k < KHH; ++k) acc[k] = 0.f;
        if (route) {
            ok = ptx::bar_and(kBarComputeAnd, kComputeThreads, wait(&sm.r_full, 0));
            if (ok) {
                ptx::tc_fence_after();
                float rv[16];
                ptx::tmem_ld16(tmem + kColR + lane_base, rv);
#pragma unroll
                for (int k = 0; k < KHH; ++k)
                    acc[k] = (kAllLive || KHH * hh + k < G) ? (hh ? rv[KHH + k] : rv[k]) : 0.f;
                ptx::tc_fence_before();
            }
        } else {
#pragma unroll
            for (int k = 0; k < KHH; ++k) {
                const int h = KHH * hh + k;
                acc[k] = h < G ? __uint_as_float((uint32_t)a.q[((size_t)b * geo.Hq + qh0 + h) * kD + t] << 16)
                               : 0.f;
            }
        }
        // Query terms: per head, 2^(8 - e) over its largest |value|, then 6 E4M3 terms.
        float invq[KHH];
        if (ok) {
            float v[KHH], av[KHH];
#pragma unroll
            for (int k = 0; k < KHH; ++k) {
                v[k] = acc[k] * sl2;
                av[k] = fabsf(v[k]);
            }
            float wm[KHH];
#pragma unroll
            for (int k = 0; k < KHH; ++k) wm[k] = warp_max(av[k]);
            if (lane == 0) {
#pragma unroll
                for (int k = 0; k < KHH; ++k) sm.red[1][warp][k] = wm[k];
            }
            ptx::bar_sync(kBarCompute, kComputeThreads);
#pragma unroll
            for (int k = 0; k < KHH; ++k) {
                float amax = sm.red[1][kQuarters * hh][k];
#pragma unroll
                for (int w = 1; w < 4; ++w) amax = fmaxf(amax, sm.red[1][kQuarters * hh + w][k]);
                float sc;
                pow2_scale(amax, sc, invq[k]);
                float x = v[k] * sc;
#pragma unroll
                for (int j = 0; j < kJq; ++j) {
                    const __nv_fp8_storage_t c = __nv_cvt_float_to_fp8(x, __NV_SATFINITE, __NV_E4M3);
                    sm.qt[qt_offset(Sh::HS * hh + KHH * j + k, t)] = c;
                    x = (x - e4m3x2_to_float2((uint32_t)c).x) * 16.f;
                }
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.qt_full);
        }

        // m: the reference maximum of each head (0 for padded heads, whose scores are -inf);
        // a weight 2^(s - m) past kLazyW moves it
        float m[KHH], lsum[KHH];
#pragma unroll
        for (int k = 0; k < KHH; ++k) {
            const bool live = kAllLive || KHH * hh + k < G;
            m[k] = live ? -INFINITY : 0.f;
            lsum[k] = 0.f;
        }
        // Lazy weight scale: every row scale so far is below lim = 2^es; weights are taken
        // times sc = 2^(6 - es) and O times inv = 2^(es - 6) at the end.
        int es = -1000;
        float lim = 0.f, sc = 1.f, inv = 1.f;
        // Completions of the output MMAs: tile j is phase j / kPBuf of o_full[j % kPBuf]. The
        // tiles are observed in order, and a warp observes tile i - kPBuf (the last reader of
        // the weight buffer it is about to fill) before it releases tile i, so no barrier runs
        // more than one phase ahead of its observer and no phase is mistaken for a later one of
        // the same parity.
        int o_seen = 0;                                // tiles 0 .. o_seen - 1 observed
        auto observe = [&](int j) -> bool {            // the output MMAs up to tile j are done
            while (o_seen <= j) {
                if (!wait(&sm.o_full[o_seen % kPBuf], (o_seen / kPBuf) & 1)) return false;
                ++o_seen;
            }
            return true;
        };

        // One barrier per tile for all compute warps: it counts the warps with a score past its
        // reference, a row scale past lim, or a failed wait since the last barrier. Only then a
        // second one exchanges the tile maxima (or lets all of them leave the loop together
        // after a failed wait).
        bool carried = true;
        for (int i = 0; ok && i < n_tiles; ++i) {
            const int u = i + base, s = u % kStages, sb = i & 1;
            // the stage's loads have landed (its scale row is read below), S is ready, and the
            // output MMAs of tile i - kPBuf (the last reader of this weight buffer) are done
            const int pb = i % kPBuf;
            bool ready = wait(&sm.full[s], (u / kStages) & 1);
            ready = ready && wait(&sm.s_full[sb], (i >> 1) & 1);
            ready = ready && observe(i - kPBuf);
            float sv[Sh::HS];
            if (ready) {
                ptx::tc_fence_after();
                tmem_ldn<Sh::HS>(tmem + kColS + sb * 32 + Sh::HS * hh + lane_base, sv);
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&sm.s_empty[sb]);
            } else {
#pragma unroll
                for (int c = 0; c < Sh::HS; ++c) sv[c] = 0.f;
            }

            const int nvalid = min(kTile, t_end - (t_begin + i * kTile));
            const bool valid = t < nvalid;
            float st = sm.scl[s][t];                      // the row scale of token t
            if (nvalid < kTile && !valid) st = 0.f;       // (stale bytes past the end)
            float s_k[KHH];
#pragma unroll
            for (int k = 0; k < KHH; k += 2) {
                // sum of the term columns, 16^-j D_j, from the last term (two heads at once)
                const F2 s16 = f2(1.f / 16.f, 1.f / 16.f);
                const F2 d = fma2(fma2(fma2(f2(sv[3 * KHH + k], sv[3 * KHH + k + 1]), s16,
                                            f2(sv[2 * KHH + k], sv[2 * KHH + k + 1])),
                                       s16, f2(sv[KHH + k], sv[KHH + k + 1])),
                                  s16, f2(sv[k], sv[k + 1]));
                const F2 sk = mul2(d, mul2(f2(invq[k], invq[k + 1]), f2(st, st)));
                s_k[k] = (kAllLive || KHH * hh + k < G) ? sk.x : -INFINITY;
                s_k[k + 1] = (kAllLive || KHH * hh + k + 1 < G) ? sk.y : -INFINITY;
            }
            if (nvalid < kTile && !valid) {
#pragma unroll
                for (int k = 0; k < KHH; ++k) s_k[k] = -INFINITY;
            }
            // the weights against the current references; a weight past kLazyW moves them
            float p_k[KHH];
#pragma unroll
            for (int k = 0; k < KHH; k += 2) {   // 0 for padded heads
                const F2 e = sub2(f2(s_k[k], s_k[k + 1]), f2(m[k], m[k + 1]));
                p_k[k] = ptx::ex2(e.x);
                p_k[k + 1] = ptx::ex2(e.y);
            }
            float pmax = p_k[0];
#pragma unroll
            for (int k = 1; k < KHH; ++k) pmax = fmaxf(pmax, p_k[k]);
            bool grow = pmax > kLazyW;
            // row scales are non-negative: their bits order as the values do
            const float smx = __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(st)));
            grow = grow || smx >= lim;
            if (lane == 0) sm.red[sb][warp][KHH] = smx;
            const bool fine = ready && carried;
            float alpha[KHH];
#pragma unroll
            for (int k = 0; k < KHH; ++k) alpha[k] = 1.f;
            if (bar_popc(kBarComputeAnd, kComputeThreads, grow || !fine) != 0) {
                // move the references to the heads' running maxima and lim past the row scales
                float wm[KHH];
#pragma unroll
                for (int k = 0; k < KHH; ++k) wm[k] = warp_max(s_k[k]);
                if (lane == 0) {
#pragma unroll
                    for (int k = 0; k < KHH; ++k) sm.red[sb][warp][k] = wm[k];
                }
                if (!ptx::bar_and(kBarComputeAnd, kComputeThreads, fine)) {
                    ok = false;
                    break;
                }
                float tmax[KHH];
#pragma unroll
                for (int k = 0; k < KHH; ++k) {
                    tmax[k] = sm.red[sb][kQuarters * hh][k];
#pragma unroll
                    for (int w = 1; w < kQuarters; ++w)
                        tmax[k] = fmaxf(tmax[k], sm.red[sb][kQuarters * hh + w][k]);
                }
                float smax = sm.red[sb][0][KHH];
#pragma unroll
                for (int w = 1; w < 4; ++w) smax = fmaxf(smax, sm.red[sb][w][KHH]);
                const int es_new =
                    smax > 0.f ? max(es, (int)((__float_as_uint(smax) >> 23) & 0xFFu) - 126) : es;
                // O so far was taken with 2^(6 - es): bring it to 2^(6 - es_new)
                const float shift = es_new > es && es > -1000 ? __uint_as_float((uint32_t)max(1, 127 + es - es_new) << 23)
                                                               : 1.f;
                bool rescale = shift != 1.f;
#pragma unroll
                for (int k = 0; k < KHH; ++k) {
                    const bool live = kAllLive || KHH * hh + k < G;
                    const float mn = fmaxf(m[k], tmax[k]);
                    alpha[k] = live ? ptx::ex2(m[k] - mn) : 1.f;
                    m[k] = live ? mn : m[k];
                    p_k[k] = ptx::ex2(s_k[k] - m[k]);
                    lsum[k] *= alpha[k];
                    rescale = rescale || alpha[k] != 1.f;
                }
                if (es_new != es) {
                    es = es_new;
                    pow2_from_exp(es + 2, sc, inv);
                    lim = __uint_as_float((uint32_t)max(1, min(254, es + 127)) << 23);
                }
                if (i >= 1 && rescale) {
                    // every output MMA so far is done (tile i's waits for this warp's weights)
                    if (observe(i - 1)) {
                        ptx::tc_fence_after();
                        float ov[Sh::HP];
                        tmem_ldn<Sh::HP>(tmem + kColO + Sh::HP * hh + lane_base, ov);
                        uint32_t ou[Sh::HP];
#pragma unroll
                        for (int c = 0; c < Sh::HP; ++c)
                            ou[c] = __float_as_uint(ov[c] * (alpha[c % KHH] * shift));
                        tmem_stn<Sh::HP>(tmem + kColO + Sh::HP * hh + lane_base, ou);
                        ptx::tmem_wait_st();
                        ptx::tc_fence_before();
                    } else {
                        carried = false;
                    }
                }
            }
            const float sts = st * sc;
            F2 x[KHH / 2];
#pragma unroll
            for (int e = 0; e < KHH / 2; ++e) {
                const F2 p = f2(p_k[2 * e], p_k[2 * e + 1]);
                const F2 l = add2(f2(lsum[2 * e], lsum[2 * e + 1]), p);
                lsum[2 * e] = l.x;
                lsum[2 * e + 1] = l.y;
                x[e] = mul2(p, f2(sts, sts));
            }
            // W row of token t: 3 E4M3 terms of this warp's KHH heads (4 KHH bytes, zero
            // padded). Each term but the last is the value rounded to E4M3; the exact residual
            // times 16 goes on.
            uint32_t w[kJp];
#pragma unroll
            for (int j = 0; j < kJp; ++j) {
                uint32_t c2[KHH / 2];
#pragma unroll
                for (int e = 0; e < KHH / 2; ++e) {
                    F2 v = x[e];
                    if (j + 1 < kJp) {
                        // (scalar: the compiler may simplify c - (c - x) and (h + k) - k when
                        // they are written with packed operations, which breaks the rounding)
                        v = f2(e4m3_round(v.x), e4m3_round(v.y));
                        x[e] = mul2(sub2(x[e], v), f2(16.f, 16.f));   // exact
                    }
                    c2[e] = (uint32_t)__nv_cvt_float2_to_fp8x2(make_float2(v.x, v.y), __NV_SATFINITE,
                                                                __NV_E4M3);
                }
                if constexpr (KHH == 4) w[j] = c2[0] | (c2[1] << 16);
                else w[j] = c2[0];
            }
            {
                // the warp's first output column HP hh: 16-column block and byte within it
                uint8_t *row = sm.p[pb] + (t >> 3) * Sh::GS + ((Sh::HP * hh) >> 4) * 128 +
                               (t & 7) * 16 + ((Sh::HP * hh) & 15);
                if constexpr (KHH == 4)
                    *reinterpret_cast<uint4 *>(row) = make_uint4(w[0], w[1], w[2], 0u);
                else
                    *reinterpret_cast<uint2 *>(row) = make_uint2(w[0] | (w[1] << 16), w[2]);
            }
            // The output MMAs read whole 32-token steps of the tile: rows past the end of the
            // sequence hold stale bytes (possibly NaN codes), so zero them.
            if (hh == 0 && !valid && t < ((nvalid + 31) & ~31)) {
                uint4 *cr = reinterpret_cast<uint4 *>(sm.codes[s] + t * 128);
#pragma unroll
                for (int c = 0; c < 8; ++c) cr[c] = make_uint4(0u, 0u, 0u, 0u);
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.p_full[pb]);
        }
        // O = (O_0 + O_1 / 16 + O_2 / 256) * inv once every output MMA is done
        float o[KHH];
#pragma unroll
        for (int k = 0; k < KHH; ++k) o[k] = 0.f;
        if (ok && carried) {
            if (observe(n_tiles - 1)) {
                ptx::tc_fence_after();
                float ov[Sh::HP];
                tmem_ldn<Sh::HP>(tmem + kColO + Sh::HP * hh + lane_base, ov);
                ptx::tc_fence_before();
#pragma unroll
                for (int k = 0; k < KHH; ++k)
                    o[k] = fmaf(ov[2 * KHH + k], 1.f / 256.f, fmaf(ov[KHH + k], 1.f / 16.f, ov[k])) * inv;
            } else {
                carried = false;
            }
        }

        // the epilogue's barrier (the row sums) settles the last waits
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
#pragma unroll
            for (int k = 0; k < KHH; ++k) lsum[k] += __shfl_xor_sync(0xffffffffu, lsum[k], off);
        const int rb = n_tiles & 1;
        if (lane == 0) {
#pragma unroll
            for (int k = 0; k < KHH; ++k) sm.red[rb][warp][k] = lsum[k];
        }
        if (ptx::bar_and(kBarComputeAnd, kComputeThreads, ok && carried)) {
#pragma unroll
            for (int k = 0; k < KHH; ++k) {
                const int h = KHH * hh + k;
                if (h >= G) continue;
                float lt = 0.f;
#pragma unroll
                for (int w = 0; w < 4; ++w) lt += sm.red[rb][kQuarters * hh + w][k];
                const float val = o[k] / lt;
                const size_t bh = (size_t)b * geo.Hq + qh0 + h;
                if (a.direct_out) {
                    if (a.out_dtype == KL_FP32) static_cast<float *>(a.out)[bh * kD + t] = val;
                    else static_cast<__nv_bfloat16 *>(a.out)[bh * kD + t] = __float2bfloat16_rn(val);
                } else {
                    const size_t slot = bh * geo.S + split;
                    a.part_o[slot * kD + t] = val;
                    if (t == 0) {
                        a.part_ml[slot * 2] = m[k] * kLn2;
                        a.part_ml[slot * 2 + 1] = lt;
                    }
                }
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, kTmemCols);
    }
    // A CTA that gave up (every role has left its loop by now, so the flag is final): the most
    // recent use of every stage may still have copies in flight; they land before its shared
    // memory goes away.
    if (warp == kProducerWarp && sm.abort) {
        for (int v = max(0, issued - kStages); v < issued; ++v) {
            const uint64_t t0 = ptx::globaltimer();
            while (!ptx::mbar_try_wait(&sm.full[v % kStages], (v / kStages) & 1) &&
                   ptx::globaltimer() - t0 < kTimeoutNs) {
            }
        }
    }
}

// ------------------------------------------------------------------------ host side ------

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

bool encode2d(CUtensorMap *map, CUtensorMapDataType type, const void *base, uint64_t inner,
              uint64_t rows, uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows,
              CUtensorMapSwizzle swizzle) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {inner, rows};
    const cuuint64_t strides[1] = {row_bytes};
    const cuuint32_t box[2] = {box_inner, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, type, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The decode for one head count per compute warp (2 for groups of up to 4 query heads, else 4)
// and whether every compute warp's heads are real (groups of exactly 4 or 8).
template <int KHH, bool kAllLive, bool kExact>
cudaError_t launch_shape(const DecodeArgs &a, const CUtensorMap &cmap, const CUtensorMap &wmap,
                         const CUtensorMap &qmap, const float *v_scales) {
    const Geometry &g = a.geo;
    const size_t smem = sizeof(Smem8) + 1024;
    static PerDeviceOnce once;
    const cudaError_t e = once.run([&] {
        return cudaFuncSetAttribute(decode_fp8_kernel<KHH, kAllLive, kExact>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.S * g.nhb, g.Hkv, g.B);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = a.stream;
    return cudaLaunchKernelEx(&cfg, decode_fp8_kernel<KHH, kAllLive, kExact>, cmap, wmap, qmap, a,
                              v_scales);
}

template <bool kExact>
cudaError_t launch_waits(const DecodeArgs &a, const CUtensorMap &cmap, const CUtensorMap &wmap,
                         const CUtensorMap &qmap, const float *v_scales) {
    const Geometry &g = a.geo;
    // groups of more than 8 heads: blocks of 8 (and a last, smaller one)
    if (g.G % 8 == 0) return launch_shape<4, true, kExact>(a, cmap, wmap, qmap, v_scales);
    if (g.G > 8) return launch_shape<4, false, kExact>(a, cmap, wmap, qmap, v_scales);
    if (g.G == 4) return launch_shape<2, true, kExact>(a, cmap, wmap, qmap, v_scales);
    return g.G < 4 ? launch_shape<2, false, kExact>(a, cmap, wmap, qmap, v_scales)
                   : launch_shape<4, false, kExact>(a, cmap, wmap, qmap, v_scales);
}

}  // namespace

cudaError_t launch_decode_fp8(const DecodeArgs &a, const float *v_scales) {
    const Geometry &g = a.geo;
    if (g.B == 0) return cudaSuccess;
    const uint64_t rows = (uint64_t)g.num_pages * g.Hkv * g.P;
    CUtensorMap cmap, wmap, qmap;
    // codes [rows][128] u8, one box = one page of one head (scale rows go by bulk copy)
    if (!encode2d(&cmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, a.v_cache, kD, rows, kD, kD, (uint32_t)g.P,
                  CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    wmap = qmap = cmap;
    if (a.w_r) {
        if (!encode2d(&wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.w_r, kD, (uint64_t)g.Hkv * kD,
                      kD * 2, 64, kD, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
        if (!encode2d(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.q, kD, (uint64_t)g.B * g.Hq, kD * 2,
                      64, (uint32_t)g.qbox, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
    }
    // exact short waits only when the limit asks for them
    return a.wait_ns < kExactWaitNs ? launch_waits<true>(a, cmap, wmap, qmap, v_scales)
                                      : launch_waits<false>(a, cmap, wmap, qmap, v_scales);
}

}  // namespace kl
