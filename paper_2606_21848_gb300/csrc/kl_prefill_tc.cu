// Tensor-core chunked prefill for sm_103a: the full attention of Eq. 3 for the query rows of a
// chunk of new tokens, over the paged Value-Only Cache, under the causal mask.
//
// One CTA per (query head h, sequence b, block of 128 query rows); head_dim 128. The rows of the
// block sit at consecutive positions p0 .. p0 + 127 of the sequence (the chunk is the tail of the
// cached rows), so the CTA walks the cache tiles 0 .. p_last / 128 and masks only the last ones.
//
//   routing  Q_r = Q . W^R[w(h)]                      M = 128 rows, N = 128, K = 128 (Section 2.2)
//   scores   S   = Q_hi . V_t^T + Q_lo . V_t^T        M = 128 rows, N = 128 tokens, K = 2 x 128
//   output   O  += P . V_t                             M = 128 rows, N = 128 dims,  K = 128
//
// Each cached tile V_t [128 tokens x 128 dims] arrives once by TMA (one box per page) and feeds
// both products from the same shared-memory copy: as the K-major B operand of the score MMAs
// (bf16, as it landed) and, once the softmax warps have converted it to fp16 in place, as the
// MN-major B operand of the output MMAs. Everything else lives in TMEM (512 columns, 128 each):
// two S buffers, O, and the routed query Q_hi | Q_lo. Q and P enter the MMAs as A operands
// straight from TMEM, so the only operand the tensor cores read from shared memory is the cache
// tile. Tile t's scores go to buffer t % 2 as soon as the output MMAs of tile t - 2 have read
// that buffer, so the score MMAs of tile t + 1 run during the softmax of tile t and the softmax
// of tile t + 1 finds its scores ready; the softmax writes tile t's weights P over the first 64
// columns of tile t's own buffer, and the output MMAs of tile t run during the softmax of tile
// t + 1.
//
// Precision: the routed query (times scale * log2 e) is carried as a pair of bf16 operands,
// x = hi + lo, about 16 significant bits where one bf16 operand keeps 8; the softmax weights
// are one fp16 operand (11 bits) against the tile in fp16. A CPU replay of these roundings on
// the parity cases (peaked rows at the start of a prompt, scores of tens of units, 1 % outlier
// values x20) puts the worst error at 0.40 of |err| <= 2e-3 + 1e-2 |ref|; with one bf16 operand
// for the weights it is 1.0-2.5 times the bound, with one fp16 operand for the query 2-5 times.
// So each tile costs three 128 x 128 x 128 MMAs instead of the four of a pair on both sides.
// bf16 values convert to fp16 exactly from 2^-14 to 65280 (smaller ones round to fp16's
// subnormal grid, an absolute error below 2^-25); a cached value of magnitude 65536 or more has
// no finite fp16 form and makes the outputs of the rows whose tiles hold it non-finite. The
// epilogue raises KL_FLAG_RANGE for any non-finite output.
//
// Softmax (thread = query row = TMEM lane): scores arrive already scaled by scale * log2 e (the
// routed query is scaled before its bf16 rounding), so p = 2^(s - m). The reference maximum m of
// a row only moves when the tile maximum exceeds it by more than 8 (a factor 256): then the row's
// O in TMEM and its running sum l are rescaled; otherwise p may reach 2^8, well inside fp16 and
// fp32 range, and the final O / l is unchanged because O and l share the same reference.
//
// Roles (352 threads, one CTA per SM):
//   warps 0-7  softmax and epilogue: warps w and w + 4 share TMEM lane quarter w % 4 (its 32
//              query rows) and split the 128 columns of S, P and O between them
//   warp 8     producer: TMA of W^R and the query block (ring position 0), then cache tiles
//   warp 9     routing and score MMA issuer (one elected lane) and TMEM owner
//   warp 10    output MMA issuer. One thread issuing tcgen05.mma back to back reaches about
//              88 cycles per 128 x 128 x 16 MMA; two issuing threads together reach the
//              tensor cores' 64.
// Every wait is bounded (about one second); a wait that runs out raises KL_FLAG_TIMEOUT, makes
// every role leave its loop, drains outstanding copies and MMAs and frees TMEM.
#include <cudaTypedefs.h>
#include <math.h>

#include "kl_internal.cuh"
#include "kl_tc_ptx.cuh"

namespace kl {
namespace {

constexpr int kD = 128;
constexpr int kBM = 128;                          // query rows per CTA
constexpr int kBN = 128;                          // cache rows per tile
constexpr int kStages = 4;
constexpr int kComputeWarps = 8;                  // two per TMEM lane quarter
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;                       // routing and score MMAs; TMEM owner
constexpr int kPvWarp = 10;                       // output MMAs
constexpr int kThreads = 11 * 32;
constexpr uint32_t kTileBytes = kBN * kD * 2;     // 32 KiB
constexpr uint32_t kHalfBytes = kTileBytes / 2;   // one 64-column half: 128 rows x 128 B
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;                     // S of tile t: 128 t % 2 .. + 127 (then P of
                                                  // tile t, fp16 pairs, in its first 64); the
                                                  // routed query first lands in buffer 0
constexpr uint32_t kColO = 256;                   // O: columns 256 .. 383
constexpr uint32_t kColQ = 384;                   // Q_hi: 384 .. 447, Q_lo: 448 .. 511
constexpr uint32_t kLoCols = 64;                  // hi -> lo of a packed bf16 operand
constexpr float kRescaleLog2 = 8.f;
constexpr uint64_t kTimeoutNs = 1000000000ull;

struct __align__(1024) PrefillSmem {
    // The query block (A operand of the routing MMA); K-major, 128B-swizzled:
    // [64-dim half][128 rows][128 B].
    uint8_t q[kBM * kD * 2];
    // Ring of 32 KiB slots: W^R[w(h)] at position 0 ([64-column half][128 k rows][128 B]), then
    // the cache tiles ([64-dim half][128 tokens][128 B]); all 128B-swizzled.
    uint8_t tiles[kStages][kTileBytes];
    uint64_t full[kStages], empty[kStages];
    uint64_t s_full[2], s_free[2], p_full, pv_done;
    uint64_t r_full, qr_ready, drain, drain2;
    float red[2][2][kBM];      // per-tile half-row maxima of the two warps of a pair (2 tiles)
    float lsum[2][kBM];        // the two warps' shares of the row sums, for the epilogue
    uint32_t tmem_base;
    int abort;
};

// Warp-collective bounded wait (every lane calls it in uniform control flow and gets the same
// answer). False when the CTA is aborting or the wait ran out (about 1 s).
struct Waiter {
    volatile int *abort;
    int32_t *err;
    __device__ bool operator()(uint64_t *bar, uint32_t parity) const {
        bool ok = ptx::mbar_try_wait(bar, parity);
        if (!ok) {
            const uint64_t t0 = ptx::globaltimer();
            while (true) {
                if (ptx::mbar_try_wait(bar, parity)) { ok = true; break; }
                if (*abort) break;
                if (ptx::globaltimer() - t0 > kTimeoutNs) {
                    *abort = 1;
                    raise_flag(err, KL_FLAG_TIMEOUT);
                    break;
                }
            }
        }
        return __all_sync(0xffffffffu, ok);
    }
};

__device__ __forceinline__ uint32_t pack2(float a, float b) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&v);
}

// x = hi + lo with hi = bf16(x), lo = bf16(x - hi), for two values packed as bf16 pairs.
__device__ __forceinline__ void split2(float x0, float x1, uint32_t &hi, uint32_t &lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
    const float2 hf = __bfloat1622float2(h);
    const __nv_bfloat162 l = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

// Instruction descriptor of kind::f16 with fp16 A and B (A and B formats 0), fp32 accumulator,
// operand majorness (0 = K-major, 1 = MN-major), N and M.
__host__ __device__ constexpr uint32_t idesc_f16(uint32_t M, uint32_t N, bool a_mn, bool b_mn) {
    return (1u << 4) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) | ((N >> 3) << 17) |
           ((M >> 4) << 24);
}

// max(a, b, c): the three-operand PTX max.
__device__ __forceinline__ float max3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// Packed fp32 pair arithmetic (one instruction for two lanes of data).
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 x, y, z;\n\t"
        "mov.b64 x, {%2, %3};\n\tmov.b64 y, {%4, %5};\n\t"
        "add.rn.f32x2 z, x, y;\n\tmov.b64 {%0, %1}, z;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 x, y, z;\n\t"
        "mov.b64 x, {%2, %3};\n\tmov.b64 y, {%4, %5};\n\t"
        "sub.rn.f32x2 z, x, y;\n\tmov.b64 {%0, %1}, z;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 mul2(float2 a, float f) {
    return make_float2(a.x * f, a.y * f);
}

// Two values as an fp16 pair (a in the low half), round to nearest even.
__device__ __forceinline__ uint32_t pack_f16(float a, float b) {
    uint32_t d;
    asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(b), "f"(a));
    return d;
}

__device__ __forceinline__ void ld_shared_v4(uint32_t addr, uint32_t (&v)[4]) {
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3])
                 : "r"(addr)
                 : "memory");
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
                 "r"(d)
                 : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap vmap,
                      const __grid_constant__ CUtensorMap wmap,
                      const __grid_constant__ CUtensorMap qmap, const PrefillArgs a) {
    extern __shared__ uint8_t smem_raw[];
    PrefillSmem &sm = *reinterpret_cast<PrefillSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const Geometry &geo = a.geo;
    const int h = blockIdx.x, b = blockIdx.y;
    const int mblk = (int)gridDim.z - 1 - (int)blockIdx.z;   // the longest blocks start first
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    const int q0 = a.cu_q[b], q1 = a.cu_q[b + 1];
    const int L = a.seq_lens[b];
    const int n = q1 - q0;
    if (q0 < 0 || n < 0 || q1 > a.total_q || L < n || L > geo.max_pages * geo.P) {
        if (tid == 0 && h == 0 && mblk == 0) raise_flag(a.err, KL_FLAG_BAD_LENGTH);
        return;
    }
    const int m0 = mblk * kBM;
    if (m0 >= n) return;
    const int rows = min(kBM, n - m0);           // query rows of this block
    const int pos0 = L - n + m0;                 // position of row 0
    const int pos_last = pos0 + rows - 1;        // <= L - 1
    const int n_tiles = pos_last / kBN + 1;      // cache tiles 0 .. n_tiles - 1
    const int g = h / geo.G;
    const int wsel = geo.wr_per_qh ? h : g;

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&sm.full[s], 1);
            ptx::mbar_init(&sm.empty[s], 1);
        }
        // One completion per tile on p_full and pv_done, one per tile of its buffer on
        // s_full[b] (scores of tile t in buffer b = t % 2) and s_free[b] (the output MMAs of
        // tile t have read buffer t % 2). Every wait names the completion it needs: MMAs that
        // write different TMEM ranges are not assumed to complete in issue order.
        for (int b2 = 0; b2 < 2; ++b2) {
            ptx::mbar_init(&sm.s_full[b2], 1);
            ptx::mbar_init(&sm.s_free[b2], 1);
        }
        ptx::mbar_init(&sm.p_full, kComputeWarps);
        ptx::mbar_init(&sm.pv_done, 1);
        ptx::mbar_init(&sm.r_full, 1);
        ptx::mbar_init(&sm.qr_ready, kComputeWarps);
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
        ptx::prefetch_tensormap(&vmap);
        ptx::prefetch_tensormap(&wmap);
        ptx::prefetch_tensormap(&qmap);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();

    const uint32_t tmem = sm.tmem_base;
    const Waiter wait{&sm.abort, a.err};

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------------ producer ----
        const int P = geo.P;
        const int ppt = kBN / P;                          // pages per tile (<= 8)
        const int seq_pages = (L + P - 1) / P;
        const uint32_t page_bytes = (uint32_t)P * 128u;  // one half of one page
        const int32_t *bt = a.block_table + (size_t)b * geo.max_pages;
        int issued = 0;
        bool bad = false;
        // position 0: W^R[w(h)] (B operand of the routing MMA) and the query block
        if (lane == 0) {
            ptx::mbar_arrive_expect_tx(&sm.full[0], kTileBytes + kBM * kD * 2);
            ptx::tma_load_2d(sm.tiles[0], &wmap, &sm.full[0], 0, wsel * kD);
            ptx::tma_load_2d(sm.tiles[0] + kHalfBytes, &wmap, &sm.full[0], 64, wsel * kD);
            ptx::tma_load_3d(sm.q, &qmap, &sm.full[0], 0, h, q0 + m0);
            ptx::tma_load_3d(sm.q + kHalfBytes, &qmap, &sm.full[0], 64, h, q0 + m0);
        }
        __syncwarp();
        issued = 1;
        for (int i = 0; i < n_tiles; ++i) {
            const int r = i + 1, s = r % kStages;
            const int pg = i * ppt + lane;                // page index within the sequence
            const bool exists = lane < ppt && pg < seq_pages;
            const int page = exists ? bt[pg] : -1;
            if (r >= kStages && !wait(&sm.empty[s], ((r / kStages) & 1) ^ 1)) break;
            const bool in_range = exists && page >= 0 && page < geo.num_pages;
            if (exists && !in_range) bad = true;
            const unsigned mask = __ballot_sync(0xffffffffu, in_range);
            if (lane == 0) ptx::mbar_arrive_expect_tx(&sm.full[s], __popc(mask) * page_bytes * 2u);
            __syncwarp();
            if (in_range) {
                const int row = (page * geo.Hkv + g) * P;
                uint8_t *dst = sm.tiles[s] + lane * page_bytes;
                ptx::tma_load_2d(dst, &vmap, &sm.full[s], 0, row);
                ptx::tma_load_2d(dst + kHalfBytes, &vmap, &sm.full[s], 64, row);
            }
            issued = r + 1;
        }
        if (__any_sync(0xffffffffu, bad) && lane == 0) raise_flag(a.err, KL_FLAG_BAD_PAGE);
        if (sm.abort) {
            // copies still in flight land before the CTA's shared memory goes away
            for (int i = max(0, issued - kStages); i < issued; ++i) {
                const uint64_t t0 = ptx::globaltimer();
                while (!ptx::mbar_try_wait(&sm.full[i % kStages], (i / kStages) & 1) &&
                       ptx::globaltimer() - t0 < kTimeoutNs) {
                }
            }
        }
    } else if (warp == kMmaWarp || warp == kPvWarp) {
        // ---------------------------------------------------------------- MMA issuers ----
        // K-major SW128 operands step 32 B per 16 columns inside a 64-column half and jump a
        // half (kHalfBytes) every 4 steps; MN-major SW128 operands step 16 rows = 2 KiB; TMEM
        // A operands step 8 columns (16 packed 16-bit values).
        constexpr uint32_t idesc_qk = ptx::idesc_bf16(128, 128, false, false);
        constexpr uint32_t idesc_route = ptx::idesc_bf16(128, 128, false, true);
        constexpr uint32_t idesc_pv = idesc_f16(128, 128, false, true);   // (mma_bf16_ts issues
        // the kind::f16 MMA; this descriptor makes both of its operands fp16)
        const uint64_t q_desc = ptx::smem_desc(ptx::smem_addr(sm.q), 16, 1024, ptx::kSwizzle128B);
        const uint64_t k_desc = ptx::smem_desc(ptx::smem_addr(sm.tiles[0]), 16, 1024, ptx::kSwizzle128B);
        const uint64_t mn_desc =
            ptx::smem_desc(ptx::smem_addr(sm.tiles[0]), kHalfBytes, 1024, ptx::kSwizzle128B);
        auto kstep = [](int kk) -> uint32_t { return ((kk >> 2) * kHalfBytes + (kk & 3) * 32) >> 4; };
        bool ok = true;
        if (warp == kMmaWarp) {
            // routing, then the score MMAs of every tile
            ok = wait(&sm.full[0], 0);
            if (ok) {
                ptx::tc_fence_after();
                if (lane == 0) {
                    // Q_r = Q . W^R: A = query block (K-major), B = W^R (N = output dim j,
                    // MN-major)
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk)
                        ptx::mma_bf16(tmem + kColS, q_desc + kstep(kk), mn_desc + ((kk * 2048) >> 4),
                                      idesc_route, kk > 0);
                    ptx::mma_commit(&sm.empty[0]);
                    ptx::mma_commit(&sm.r_full);
                }
                __syncwarp();
            }
            ok = ok && wait(&sm.qr_ready, 0);
            for (int i = 0; ok && i < n_tiles; ++i) {
                const int r = i + 1, s = r % kStages, sb = i & 1;
                // the output MMAs of tile i - 2 have read buffer sb (its P); waited on before
                // the tile, so that this is the buffer's next completion (the one after it
                // needs tile i's scores)
                if (i >= 2 && !wait(&sm.s_free[sb], ((i >> 1) - 1) & 1)) { ok = false; break; }
                if (!wait(&sm.full[s], (r / kStages) & 1)) { ok = false; break; }
                ptx::tc_fence_after();
                if (lane == 0) {
                    // S = Q_hi . V_i^T + Q_lo . V_i^T: A = Q_r in TMEM, B = the tile
                    // (N = tokens, K-major)
                    const uint64_t b0 = k_desc + ((s * kTileBytes) >> 4);
#pragma unroll
                    for (int kk = 0; kk < 2 * kD / 16; ++kk)
                        ptx::mma_bf16_ts(tmem + kColS + sb * 128u,
                                         tmem + kColQ + (kk >= 8 ? kLoCols : 0u) + (kk & 7) * 8,
                                         b0 + kstep(kk & 7), idesc_qk, kk > 0);
                    ptx::mma_commit(&sm.s_full[sb]);
                }
                __syncwarp();
            }
        } else {
            // the output MMAs of every tile: O += P . V_j, fp16; A = P in TMEM (the first 64
            // columns of buffer j % 2), B = the tile (N = dims, MN-major), converted to fp16 by
            // the softmax warps before they arrive on p_full
            for (int j = 0; j < n_tiles; ++j) {
                const int s = (j + 1) % kStages;
                if (!wait(&sm.p_full, j & 1)) { ok = false; break; }
                ptx::tc_fence_after();
                if (lane == 0) {
                    const uint64_t b0 = mn_desc + ((s * kTileBytes) >> 4);
                    const uint32_t pa = tmem + kColS + (j & 1) * 128u;
#pragma unroll
                    for (int kk = 0; kk < kBN / 16; ++kk)
                        ptx::mma_bf16_ts(tmem + kColO, pa + kk * 8, b0 + ((kk * 2048) >> 4), idesc_pv,
                                         (j > 0 || kk > 0) ? 1u : 0u);
                    ptx::mma_commit(&sm.empty[s]);
                    ptx::mma_commit(&sm.s_free[j & 1]);
                    ptx::mma_commit(&sm.pv_done);
                }
                __syncwarp();
            }
        }
        (void)ok;
        // every MMA this warp issued completes before TMEM is freed
        uint64_t *drain = warp == kMmaWarp ? &sm.drain : &sm.drain2;
        if (lane == 0) ptx::mma_commit(drain);
        __syncwarp();
        const uint64_t t0 = ptx::globaltimer();
        while (!ptx::mbar_try_wait(drain, 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
        }
    } else {
        // --------------------------------------------------------- softmax, epilogue ----
        // Two warps per TMEM lane quarter: warp w serves rows 32 (w % 4) .. + 31 and columns
        // 64 hf .. + 63 (hf = w / 4) of S, P and O. The pair meets once per tile on a named
        // barrier (id 1 + w % 4) that also ANDs their progress, so both leave a loop together.
        const int qd = warp & 3, hf = warp >> 2;
        const int r = qd * 32 + lane;                        // query row = TMEM lane
        const int c0 = hf * 64;                              // this warp's columns
        const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
        const uint32_t pair_bar = 1 + qd;
        // rows past the block's end take the last valid position: finite, never stored
        const int pos_r = min(pos0 + r, pos_last);
        const float sl2 = geo.scale * kLog2e;
        bool ok = wait(&sm.r_full, 0);

        // Routed query row, this warp's 64 columns: Q_r * scale * log2 e as hi + lo bf16 pairs
        // into the Q columns (32 packed columns each).
        if (ok) {
            ptx::tc_fence_after();
            uint32_t u0[32], u1[32];
            ptx::tmem_ld32(tmem + kColS + c0 + lane_base, u0);
            ptx::tmem_ld32(tmem + kColS + c0 + 32 + lane_base, u1);
            ptx::tmem_wait_ld();
            ptx::reg_fence(u0);
            ptx::reg_fence(u1);
            uint32_t hi[32], lo[32];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                split2(__uint_as_float(u0[2 * e]) * sl2, __uint_as_float(u0[2 * e + 1]) * sl2,
                       hi[e], lo[e]);
                split2(__uint_as_float(u1[2 * e]) * sl2, __uint_as_float(u1[2 * e + 1]) * sl2,
                       hi[16 + e], lo[16 + e]);
            }
            ptx::tmem_st32(tmem + kColQ + c0 / 2 + lane_base, hi);
            ptx::tmem_st32(tmem + kColQ + kLoCols + c0 / 2 + lane_base, lo);
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.qr_ready);
        }

        float m_ref = -INFINITY;   // reference maximum of the row (base 2), shared by the pair
        // this warp's share of sum 2^(s - m_ref), in two packed pairs of partial sums
        float2 la = make_float2(0.f, 0.f), lb = make_float2(0.f, 0.f);
        // Both warps of a pair run the same tiles and meet on exactly one pair barrier per
        // tile and one in the epilogue; a wait that fails only turns this warp's vote false, and
        // the pair leaves together at the next barrier.
        bool okl = ok;
        for (int i = 0; i < n_tiles; ++i) {
            const int t0 = i * kBN, rb = i & 1;
            const uint32_t sbuf = tmem + kColS + (uint32_t)rb * 128u;   // S, then P, of tile i
            if (okl) okl = wait(&sm.s_full[rb], (i >> 1) & 1);
            float sv[64];
            float mp = -INFINITY;
            if (okl) {
                ptx::tc_fence_after();
                uint32_t u0[32], u1[32];
                ptx::tmem_ld32(sbuf + c0 + lane_base, u0);
                ptx::tmem_ld32(sbuf + c0 + 32 + lane_base, u1);
                ptx::tmem_wait_ld();
                ptx::reg_fence(u0);
                ptx::reg_fence(u1);
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    sv[c] = __uint_as_float(u0[c]);
                    sv[32 + c] = __uint_as_float(u1[c]);
                }
                // causal mask: token t0 + c0 + c is visible to the row when it is <= pos_r
                if (t0 + c0 + 63 > pos0) {
                    const int lim = pos_r - t0 - c0;
#pragma unroll
                    for (int c = 0; c < 64; ++c)
                        if (c > lim) sv[c] = -INFINITY;
                }
                float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int c = 0; c < 64; c += 8) {
                    mx[0] = max3(mx[0], sv[c], sv[c + 1]);
                    mx[1] = max3(mx[1], sv[c + 2], sv[c + 3]);
                    mx[2] = max3(mx[2], sv[c + 4], sv[c + 5]);
                    mx[3] = max3(mx[3], sv[c + 6], sv[c + 7]);
                }
                mp = max3(mx[0], mx[1], fmaxf(mx[2], mx[3]));
                sm.red[rb][hf][r] = mp;
            }
            // the pair exchanges its half maxima (and leaves together on any failed wait); past
            // this barrier both warps hold their S in registers, so P may overwrite the buffer
            if (!ptx::bar_and(pair_bar, 64, okl)) {
                okl = false;
                break;
            }
            const float m_tile = fmaxf(mp, sm.red[rb][hf ^ 1][r]);
            const float m_new = fmaxf(m_ref, m_tile);
            // a new reference when the maximum grew by more than 2^8 (or is the first finite);
            // both warps of the pair take the same decision from the same numbers
            const bool grow = m_new > m_ref + kRescaleLog2;
            if (__any_sync(0xffffffffu, grow)) {
                const float f = (m_new == -INFINITY || m_ref == -INFINITY) ? 0.f : ptx::ex2(m_ref - m_new);
                if (i > 0) {
                    // O holds tiles 0 .. i - 1 once the output MMAs of tile i - 1 are done
                    okl = okl && wait(&sm.pv_done, (i - 1) & 1);
                    if (okl) {
                        ptx::tc_fence_after();
#pragma unroll
                        for (int c = 0; c < 64; c += 32) {
                            uint32_t u[32];
                            ptx::tmem_ld32(tmem + kColO + c0 + c + lane_base, u);
                            ptx::tmem_wait_ld();
                            ptx::reg_fence(u);
#pragma unroll
                            for (int e = 0; e < 32; ++e) u[e] = __float_as_uint(__uint_as_float(u[e]) * f);
                            ptx::tmem_st32(tmem + kColO + c0 + c + lane_base, u);
                        }
                        ptx::tmem_wait_st();
                    }
                }
                la = mul2(la, f);
                lb = mul2(lb, f);
                m_ref = m_new;
            }
            const float mr = m_ref == -INFINITY ? 0.f : m_ref;

            // this warp's 64 weights -> 32 packed fp16 columns of P (in pairs: s - m, 2^x, the
            // running sums, the fp16 pack)
            uint32_t ph[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                const float2 d = sub2(make_float2(sv[2 * e], sv[2 * e + 1]), make_float2(mr, mr));
                const float2 pe = make_float2(ptx::ex2(d.x), ptx::ex2(d.y));
                if (e & 1) lb = add2(lb, pe); else la = add2(la, pe);
                ph[e] = pack_f16(pe.x, pe.y);
            }
            // The score MMAs are done with tile i: this thread converts its cache row r,
            // dims 64 hf .. + 63 (128 contiguous bytes whatever the swizzle), to fp16 in place
            // for the output MMAs. Rows at or past the sequence's end (an unwritten page
            // tail, or a page slot no TMA filled) become zeros instead, so that 0-weights
            // never meet a non-finite value. The lanes start at different 16-byte chunks so
            // that a warp's accesses spread over all banks.
            if (okl) {
                const uint32_t v_s = ptx::smem_addr(sm.tiles[(i + 1) % kStages]) +
                                     hf * kHalfBytes + r * 128;
                if (t0 + r < L) {
#pragma unroll 4
                    for (int c = 0; c < 8; ++c) {
                        const uint32_t addr = v_s + ((c + lane) & 7) * 16;
                        uint32_t w[4];
                        ld_shared_v4(addr, w);
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            w[e] = pack_f16(__uint_as_float(w[e] << 16),
                                            __uint_as_float(w[e] & 0xffff0000u));
                        }
                        st_shared_v4(addr, w[0], w[1], w[2], w[3]);
                    }
                } else {
#pragma unroll
                    for (int c = 0; c < 8; ++c) st_shared_v4(v_s + c * 16, 0u, 0u, 0u, 0u);
                }
                // P over the first 64 columns of the buffer (the output MMAs of tile i - 2, the
                // last reader of P there, finished before tile i's scores were written)
                ptx::tmem_st32(sbuf + c0 / 2 + lane_base, ph);
                ptx::tmem_wait_st();
                // the converted tile (generic-proxy stores) is read next by the output MMAs
                ptx::tc_fence_before();
                ptx::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&sm.p_full);
            }
            // a wait that failed above leaves okl false: this warp skips its work and votes
            // false at the next pair barrier (or the epilogue's), where the pair leaves together
        }

        // Epilogue: out = O / l, this warp's 64 output dims; l is the pair's two shares. A
        // non-finite output (a cached value beyond fp16's range, or a non-finite input) raises
        // KL_FLAG_RANGE.
        const float l = (la.x + la.y) + (lb.x + lb.y);
        const bool oke = okl && wait(&sm.pv_done, (n_tiles - 1) & 1);
        sm.lsum[hf][r] = l;
        if (ptx::bar_and(pair_bar, 64, oke)) {
            ptx::tc_fence_after();
            const float lt = l + sm.lsum[hf ^ 1][r];
            const float inv = lt > 0.f ? 1.f / lt : 0.f;
            float nf = 0.f;   // x * 0 is NaN exactly when x is not finite
            const size_t orow = ((size_t)(q0 + m0 + r) * geo.Hq + h) * kD + c0;
#pragma unroll
            for (int c4 = 0; c4 < 2; ++c4) {
                uint32_t u[32];
                ptx::tmem_ld32(tmem + kColO + c0 + c4 * 32 + lane_base, u);
                ptx::tmem_wait_ld();
                ptx::reg_fence(u);
                if (r < rows) {
#pragma unroll
                    for (int e = 0; e < 32; ++e) nf = fmaf(__uint_as_float(u[e]), 0.f, nf);
                    if (a.out_dtype == KL_FP32) {
                        float4 *o = reinterpret_cast<float4 *>(static_cast<float *>(a.out) + orow + c4 * 32);
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            o[c] = make_float4(__uint_as_float(u[4 * c]) * inv, __uint_as_float(u[4 * c + 1]) * inv,
                                               __uint_as_float(u[4 * c + 2]) * inv, __uint_as_float(u[4 * c + 3]) * inv);
                    } else {
                        uint4 *o = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.out) + orow + c4 * 32);
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            uint32_t w[4];
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                w[e] = pack2(__uint_as_float(u[8 * c + 2 * e]) * inv,
                                             __uint_as_float(u[8 * c + 2 * e + 1]) * inv);
                            o[c] = make_uint4(w[0], w[1], w[2], w[3]);
                        }
                    }
                }
            }
            if (__any_sync(0xffffffffu, nf != nf) && lane == 0) raise_flag(a.err, KL_FLAG_RANGE);
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, kTmemCols);
    }
}

// Chunk append: row i of sequence b's chunk goes to position seq_lens[b] - n_b + i. One CTA per
// (16 chunk rows, sequence); 16-byte copies.
constexpr int kAppendRows = 16;

__global__ void __launch_bounds__(128) append_chunk_kernel(int Hkv, int D, int P, int num_pages,
                                                           int max_pages, int total_q,
                                                           const uint4 *__restrict__ v_new,
                                                           const int32_t *__restrict__ block_table,
                                                           const int32_t *__restrict__ seq_lens,
                                                           const int32_t *__restrict__ cu_q,
                                                           uint4 *__restrict__ v_cache, int32_t *err) {
    const int b = blockIdx.y;
    const int q0 = cu_q[b], n = cu_q[b + 1] - q0, L = seq_lens[b];
    if (q0 < 0 || n < 0 || q0 + n > total_q || L < n || L > max_pages * P) {
        if (threadIdx.x == 0 && blockIdx.x == 0) raise_flag(err, KL_FLAG_BAD_LENGTH);
        return;
    }
    const int i0 = blockIdx.x * kAppendRows;
    const int cpr = D / 8;   // 16-byte chunks per row
    const int per_row = Hkv * cpr;
    for (int k = threadIdx.x; k < kAppendRows * per_row; k += blockDim.x) {
        const int i = i0 + k / per_row;
        if (i >= n) break;
        const int gc = k % per_row, g = gc / cpr, c = gc % cpr;
        const int pos = L - n + i;
        const int page = block_table[(size_t)b * max_pages + pos / P];
        if (page < 0 || page >= num_pages) {
            raise_flag(err, KL_FLAG_BAD_PAGE);
            continue;
        }
        v_cache[(((size_t)page * Hkv + g) * P + pos % P) * cpr + c] =
            v_new[((size_t)(q0 + i) * Hkv + g) * cpr + c];
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

// bf16 tensor map of `rank` dimensions, innermost 128 elements (256-byte rows), box 64 x ...,
// 128-byte swizzle.
bool encode(CUtensorMap *map, const void *base, int rank, const cuuint64_t *dims,
            const cuuint64_t *strides, const cuuint32_t *box) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void *>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool prefill_tc_supported(const Geometry &g) {
    if (g.D != kD) return false;
    if (g.P != 16 && g.P != 32 && g.P != 64 && g.P != 128) return false;
    if ((int64_t)g.num_pages * g.Hkv * g.P >= ((int64_t)1 << 31)) return false;
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3;
}

cudaError_t launch_prefill_tc(const PrefillArgs &a) {
    const Geometry &g = a.geo;
    if (g.B == 0 || a.total_q == 0 || a.max_q == 0) return cudaSuccess;
    CUtensorMap vmap, wmap, qmap;
    {
        // cache as [num_pages * Hkv * P rows][128], one box = one page of one head (64 dims)
        const cuuint64_t dims[2] = {kD, (cuuint64_t)g.num_pages * g.Hkv * g.P};
        const cuuint64_t strides[1] = {kD * 2};
        const cuuint32_t box[2] = {64, (cuuint32_t)g.P};
        if (!encode(&vmap, a.v_cache, 2, dims, strides, box)) return cudaErrorInvalidValue;
    }
    {
        // W^R as [Hw * 128 k rows][128 j], one box = a 64-column half of one matrix
        const cuuint64_t hw = g.wr_per_qh ? (cuuint64_t)g.Hq : (cuuint64_t)g.Hkv;
        const cuuint64_t dims[2] = {kD, hw * kD};
        const cuuint64_t strides[1] = {kD * 2};
        const cuuint32_t box[2] = {64, kD};
        if (!encode(&wmap, a.w_r, 2, dims, strides, box)) return cudaErrorInvalidValue;
    }
    {
        // q as [total_q][Hq][128], one box = 128 consecutive rows of one head (64 dims); rows
        // past total_q read as zeros
        const cuuint64_t dims[3] = {kD, (cuuint64_t)g.Hq, (cuuint64_t)a.total_q};
        const cuuint64_t strides[2] = {kD * 2, (cuuint64_t)g.Hq * kD * 2};
        const cuuint32_t box[3] = {64, 1, kBM};
        if (!encode(&qmap, a.q, 3, dims, strides, box)) return cudaErrorInvalidValue;
    }
    const size_t smem = sizeof(PrefillSmem) + 1024;
    static PerDeviceOnce once;
    const cudaError_t e = once.run([&] {
        return cudaFuncSetAttribute(prefill_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)smem);
    });
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.Hq, g.B, (a.max_q + kBM - 1) / kBM);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = a.stream;
    return cudaLaunchKernelEx(&cfg, prefill_tc_kernel, vmap, wmap, qmap, a);
}

cudaError_t launch_append_chunk(const Geometry &g, int total_q, int max_q, const uint16_t *v_new,
                                const int32_t *block_table, const int32_t *seq_lens,
                                const int32_t *cu_q, uint16_t *v_cache, int32_t *err,
                                cudaStream_t stream) {
    if (g.B == 0 || total_q == 0 || max_q == 0) return cudaSuccess;
    const dim3 grid((max_q + kAppendRows - 1) / kAppendRows, g.B);
    append_chunk_kernel<<<grid, 128, 0, stream>>>(g.Hkv, g.D, g.P, g.num_pages, g.max_pages, total_q,
                                                  reinterpret_cast<const uint4 *>(v_new), block_table,
                                                  seq_lens, cu_q, reinterpret_cast<uint4 *>(v_cache), err);
    return cudaGetLastError();
}

}  // namespace kl
