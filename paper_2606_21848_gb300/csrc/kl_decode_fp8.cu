// Keyless decode over an FP8 value cache (E4M3 codes, one fp32 scale per cached row), on the
// tensor cores for sm_103a; and the quantizing append.
//
// Same method and split plan as the bf16 decode (routing q_r = q W^R, Section 2.2; one softmax
// over the cached value rows, each row used for the score and for the output, Section 3), but
// the cache moves half the bytes: a 128-token tile is 16 KiB of codes plus 512 B of scales.
// Every code is an exact half-precision value, so two warps widen each landed tile into a
// half-precision copy in shared memory, and the tensor cores run kind::f16 MMAs on it (the
// routed query and the softmax weights as hi + lo half pairs):
//
//   scores   S^T = C_t . [q_hi | q_lo]^T        (C_t the codes of tile t, as halves)
//   output   O^T = C_t^T . [p_hi | p_lo]
//
// A row's scale multiplies its score column (s_t = scale_t <q_r, c_t>) and its softmax weight
// (p_t scale_t feeds the output MMA), so the codes never need rescaling.
//
// One CTA per (split, value head g, sequence b); 288 threads, two CTAs per SM:
//   warps 0-3  softmax (thread = token), O accumulation (thread = output dim), epilogue
//              (output row, or split state for the combine kernel)
//   warp 4     producer: W^R[g] and the group's query rows (routing operands), then TMA loads
//              of code pages and scale rows into a 2-stage ring
//   warp 5     routing and score MMA issuer, TMEM owner
//   warp 6     output MMA issuer
//   warps 7-8  widen each landed code tile into the half tile that the output MMAs two tiles
//              back have released, so the softmax warps never wait on the widening
// Every wait is bounded (about one second); a wait that runs out raises KL_FLAG_TIMEOUT and
// every role leaves its loop, drains its copies and MMAs, and TMEM is freed.
#include <cuda_fp16.h>
#include <cuda_fp8.h>
#include <cudaTypedefs.h>
#include <math.h>

#include "kl_internal.cuh"
#include "kl_tc_ptx.cuh"

namespace kl {
namespace {

constexpr int kD = 128;
constexpr int kTile = 128;
constexpr int kNG = 8;                      // query heads per value group (padded)
constexpr int kN = 2 * kNG;                 // MMA N: hi and lo halves
constexpr int kComputeWarps = 4;
constexpr int kProducerWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kPvWarp = 6;
constexpr int kConvWarp0 = 7;               // warps 7-8 widen code tiles
constexpr int kConvWarps = 2;
constexpr int kThreads = 9 * 32;
constexpr int kStages = 2;                  // code tiles in flight
constexpr uint32_t kCodeBytes = kTile * kD;          // 16 KiB of codes per tile
constexpr uint32_t kTileBytes = kTile * kD * 2;      // 32 KiB half tile (MMA operand)
constexpr uint32_t kHalfBytes = kTileBytes / 2;      // one 64-dim half: 128 rows x 128 B
constexpr uint32_t kTmemCols = 64;                   // S: 2 x 16 columns, O: 2 x 16 columns
constexpr int kScaleFloats = 256;                    // (128 / P) slots of max(32, P) floats
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr uint32_t kBarCompute = 1;
constexpr uint32_t kBarComputeAnd = 2;

struct __align__(1024) Smem8 {
    // Half-precision tiles, the MMA operands: [64-dim half][128 rows][128 B], 128B-swizzled.
    // cvt[1] first holds W^R[g] (bf16) for the routing MMA.
    uint8_t cvt[2][kTileBytes];
    // Code tiles as TMA writes them: [128 rows][128 B], 128B-swizzled. Row scales: one slot of
    // max(32, P) floats per page, so that every TMA destination is 128-byte aligned.
    uint8_t codes[kStages][kCodeBytes];
    float scl[kStages][kScaleFloats];
    float cscl[2][kTile];              // row scales of the tile in cvt[b], token order
    uint8_t qr[2 * kN * 128];          // routed query operand [half][16 rows][128 B], K-major
    uint8_t p[2][kTile * kN * 2];      // P^T operands, no swizzle, MN-major
    float red[2][kComputeWarps][kNG];
    uint64_t full[kStages], empty[kStages];
    uint64_t c_full[2];
    uint64_t s_full[2], s_empty[2], p_full[2], o_full[2], o_empty[2];
    uint64_t r_load, r_full, qr_full, drain, drain2;
    uint32_t tmem_base;
    int abort;
};

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

// Per-head maximum over the 32 lanes of a warp by transposed halving (see the bf16 decode).
__device__ __forceinline__ float warp_max8(const float (&x)[8], int lane) {
    const bool b4 = lane & 16, b3 = lane & 8, b2 = lane & 4;
    float a4[4], a2[2];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float send = b4 ? x[j] : x[j + 4];
        const float keep = b4 ? x[j + 4] : x[j];
        a4[j] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 16));
    }
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        const float send = b3 ? a4[j] : a4[j + 2];
        const float keep = b3 ? a4[j + 2] : a4[j];
        a2[j] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 8));
    }
    float a1;
    {
        const float send = b2 ? a2[0] : a2[1];
        const float keep = b2 ? a2[1] : a2[0];
        a1 = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 4));
    }
    a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 2));
    a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 1));
    return a1;
}

// Two E4M3 codes (low byte first) to two halves (low half first): the PTX conversion
// instruction, exact since every E4M3 value is a half-precision value.
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t two_codes) {
    uint32_t r;
    const uint16_t v = (uint16_t)two_codes;
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(r) : "h"(v));
    return r;
}

// x = hi + lo in half precision for two values.
__device__ __forceinline__ void split_h2(float x0, float x1, uint32_t &hi, uint32_t &lo) {
    const __half2 h = __floats2half2_rn(x0, x1);
    const float2 hf = __half22float2(h);
    const __half2 l = __floats2half2_rn(x0 - hf.x, x1 - hf.y);
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

// Byte offset of element (row n, column k) in the K-major, 128B-swizzled query operand of 16
// rows and 128 columns laid out as [half][16 rows][128 B].
__device__ __forceinline__ uint32_t qr_offset(int n, int k) {
    const int half = k >> 6, kk = k & 63;
    return half * (kN * 128) + (n >> 3) * 1024 + (n & 7) * 128 + (((kk >> 3) ^ (n & 7)) << 4) +
           ((kk & 7) << 1);
}

// Instruction descriptor of kind::f16 with half-precision A and B, fp32 accumulator.
__host__ __device__ constexpr uint32_t idesc_f16(uint32_t M, uint32_t N, bool a_mn, bool b_mn) {
    return (1u << 4) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) | ((N >> 3) << 17) |
           ((M >> 4) << 24);
}

__global__ void __launch_bounds__(kThreads, 2)
    decode_fp8_kernel(const __grid_constant__ CUtensorMap cmap,
                      const __grid_constant__ CUtensorMap smap,
                      const __grid_constant__ CUtensorMap wmap,
                      const __grid_constant__ CUtensorMap qmap, const DecodeArgs a) {
    constexpr int NS = kStages;
    extern __shared__ uint8_t smem_raw[];
    Smem8 &sm = *reinterpret_cast<Smem8 *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                           ~uintptr_t(1023));
    const Geometry &geo = a.geo;
    const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = geo.G;
    const bool route = a.w_r != nullptr;      // W^R given; else q is the composed query

    const int L_raw = a.seq_lens[b];
    const int t_begin = split * geo.chunk;
    const int32_t *bt = a.block_table + (size_t)b * geo.max_pages;

    if (tid == 0) {
        for (int s = 0; s < NS; ++s) {
            ptx::mbar_init(&sm.full[s], 1);
            ptx::mbar_init(&sm.empty[s], kConvWarps);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&sm.c_full[i], kConvWarps);
            ptx::mbar_init(&sm.s_full[i], 1);
            ptx::mbar_init(&sm.s_empty[i], kComputeWarps);
            ptx::mbar_init(&sm.p_full[i], kComputeWarps);
            ptx::mbar_init(&sm.o_full[i], 1);
            ptx::mbar_init(&sm.o_empty[i], kComputeWarps);
        }
        ptx::mbar_init(&sm.r_load, 1);
        ptx::mbar_init(&sm.r_full, 1);
        ptx::mbar_init(&sm.qr_full, kComputeWarps);
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
        ptx::prefetch_tensormap(&smap);
        if (route) {
            ptx::prefetch_tensormap(&wmap);
            ptx::prefetch_tensormap(&qmap);
        }
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();

    int L = L_raw;
    if (L < 0 || L > geo.max_pages * geo.P) {
        if (tid == 0 && split == 0 && g == 0) raise_flag(a.err, KL_FLAG_BAD_LENGTH);
        L = 0;
    }
    const int t_end = min(t_begin + geo.chunk, L);
    const int n_tiles = t_end > t_begin ? (t_end - t_begin + kTile - 1) / kTile : 0;

    if (n_tiles == 0) {
        // an empty split: zero output (direct) or an empty state
        if (tid < kD) {
            for (int h = 0; h < G; ++h) {
                const size_t bh = (size_t)b * geo.Hq + g * G + h;
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
    const Waiter wait{&sm.abort, a.err};

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------------ producer ----
        const int P = geo.P;
        const int ppt = kTile / P;                           // pages per tile (<= 8)
        const int first_page = t_begin / P;
        const int end_page = (t_end + P - 1) / P;
        const uint32_t page_bytes = (uint32_t)P * 128u + (uint32_t)P * 4u;
        const int scale_slot = max(32, P);                   // floats per page slot
        bool bad = false;
        int issued = 0;
        if (route && lane == 0) {
            // routing operands: W^R[g] (MN-major A of the routing MMA) into cvt[1], the group's
            // query rows (K-major B) into the query operand buffer
            ptx::mbar_arrive_expect_tx(&sm.r_load, kTileBytes + 2u * (uint32_t)G * 128u);
            ptx::tma_load_2d(sm.cvt[1], &wmap, &sm.r_load, 0, g * kD);
            ptx::tma_load_2d(sm.cvt[1] + kHalfBytes, &wmap, &sm.r_load, 64, g * kD);
            ptx::tma_load_2d(sm.qr, &qmap, &sm.r_load, 0, b * geo.Hq + g * G);
            ptx::tma_load_2d(sm.qr + kN * 128, &qmap, &sm.r_load, 64, b * geo.Hq + g * G);
        }
        __syncwarp();
        for (int i = 0; i < n_tiles; ++i) {
            const int s = i % NS;
            const int p0 = first_page + i * ppt;
            const bool exists = lane < ppt && p0 + lane < end_page;
            const int page = exists ? bt[p0 + lane] : -1;
            if (i >= NS && !wait(&sm.empty[s], ((i / NS) & 1) ^ 1)) break;
            const bool in_range = exists && page >= 0 && page < geo.num_pages;
            if (exists && !in_range) bad = true;
            const unsigned mask = __ballot_sync(0xffffffffu, in_range);
            if (lane == 0) ptx::mbar_arrive_expect_tx(&sm.full[s], __popc(mask) * page_bytes);
            __syncwarp();
            if (in_range) {
                const int row = (page * geo.Hkv + g) * P;
                ptx::tma_load_2d(sm.codes[s] + lane * P * 128, &cmap, &sm.full[s], 0, row);
                ptx::tma_load_2d(&sm.scl[s][lane * scale_slot], &smap, &sm.full[s], 0,
                                 page * geo.Hkv + g);
            }
            issued = i + 1;
        }
        if (__any_sync(0xffffffffu, bad) && lane == 0) raise_flag(a.err, KL_FLAG_BAD_PAGE);
        if (sm.abort) {
            for (int i = max(0, issued - NS); i < issued; ++i) {
                const uint64_t t0 = ptx::globaltimer();
                while (!ptx::mbar_try_wait(&sm.full[i % NS], (i / NS) & 1) &&
                       ptx::globaltimer() - t0 < kTimeoutNs) {
                }
            }
            if (route) {
                const uint64_t t0 = ptx::globaltimer();
                while (!ptx::mbar_try_wait(&sm.r_load, 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
                }
            }
        }
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------- score MMA issuer -------
        constexpr uint32_t idesc_s = idesc_f16(128, kN, false, false);
        const uint64_t q_desc = ptx::smem_desc(ptx::smem_addr(sm.qr), 16, 1024, ptx::kSwizzle128B);
        const uint64_t c_desc = ptx::smem_desc(ptx::smem_addr(sm.cvt[0]), 16, 1024, ptx::kSwizzle128B);
        bool ok = true;
        if (route) {
            // q_r^T[128 j x 16] = W^R^T (MN-major, bf16) . q^T (K-major rows of the query buffer)
            constexpr uint32_t idesc_r = ptx::idesc_bf16(128, kN, true, false);
            ok = wait(&sm.r_load, 0);
            if (ok) {
                ptx::tc_fence_after();
                if (lane == 0) {
                    const uint64_t w_desc = ptx::smem_desc(ptx::smem_addr(sm.cvt[1]), kHalfBytes,
                                                           1024, ptx::kSwizzle128B);
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        const uint32_t qoff = (kk >> 2) * (kN * 128) + (kk & 3) * 32;
                        ptx::mma_bf16(tmem + 2 * kN, w_desc + ((kk * 2048) >> 4), q_desc + (qoff >> 4),
                                      idesc_r, kk > 0);
                    }
                    ptx::mma_commit(&sm.r_full);
                }
                __syncwarp();
            }
        }
        ok = ok && wait(&sm.qr_full, 0);
        if (ok) ptx::tc_fence_after();
        for (int i = 0; ok && i < n_tiles; ++i) {
            const int cb = i & 1, sb = i & 1;
            if (!wait(&sm.c_full[cb], (i >> 1) & 1)) break;
            if (i >= 2 && !wait(&sm.s_empty[sb], ((i >> 1) - 1) & 1)) break;
            ptx::tc_fence_after();
            if (lane == 0) {
                const uint64_t a0 = c_desc + ((cb * kTileBytes) >> 4);
#pragma unroll
                for (int kk = 0; kk < kD / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
                    const uint32_t qoff = (kk >> 2) * (kN * 128) + (kk & 3) * 32;
                    ptx::mma_bf16(tmem + sb * kN, a0 + (koff >> 4), q_desc + (qoff >> 4), idesc_s, kk > 0);
                }
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
        // A = C^T: MN-major SW128 (64-dim halves kHalfBytes apart, 8-token groups 1 KiB apart);
        // B = P^T: MN-major, no swizzle (hi/lo blocks 128 B apart, 8-token groups 256 B apart)
        constexpr uint32_t idesc_o = idesc_f16(128, kN, true, true);
        const uint64_t c_desc =
            ptx::smem_desc(ptx::smem_addr(sm.cvt[0]), kHalfBytes, 1024, ptx::kSwizzle128B);
        const uint64_t p_desc = ptx::smem_desc(ptx::smem_addr(sm.p[0]), 256, 128, ptx::kSwizzleNone);
        constexpr uint32_t kPBytes = sizeof(sm.p[0]);
        for (int j = 0; j < n_tiles; ++j) {
            const int cb = j & 1, pb = j & 1;
            if (!wait(&sm.p_full[pb], (j >> 1) & 1)) break;
            if (j >= 2 && !wait(&sm.o_empty[pb], ((j >> 1) - 1) & 1)) break;
            ptx::tc_fence_after();
            const int nvalid = min(kTile, t_end - (t_begin + j * kTile));
            const int ksteps = (nvalid + 15) >> 4;
            if (lane == 0) {
                const uint64_t a0 = c_desc + ((cb * kTileBytes) >> 4);
                const uint64_t b0 = p_desc + ((pb * kPBytes) >> 4);
                for (int kk = 0; kk < ksteps; ++kk)
                    ptx::mma_bf16(tmem + 2 * kN + pb * kN, a0 + ((kk * 2048) >> 4), b0 + ((kk * 512) >> 4),
                                  idesc_o, kk > 0);
                ptx::mma_commit(&sm.o_full[pb]);
            }
            __syncwarp();
        }
        if (lane == 0) ptx::mma_commit(&sm.drain2);
        __syncwarp();
        const uint64_t t0 = ptx::globaltimer();
        while (!ptx::mbar_try_wait(&sm.drain2, 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
        }
    } else if (warp >= kConvWarp0) {
        // ------------------------------------------------------------------ widening ----
        // Thread u takes rows u and u + 64 of each tile. Tile j goes into cvt[j & 1] once the
        // output MMAs of tile j - 2 (the last reader of that buffer) are done.
        const int u = tid - kConvWarp0 * 32;
        for (int j = 0; j < n_tiles; ++j) {
            const int s = j % NS, cb = j & 1;
            if (!wait(&sm.full[s], (j / NS) & 1)) break;
            if (j >= 2 && !wait(&sm.o_full[cb], ((j - 2) >> 1) & 1)) break;
            const int nvalid = min(kTile, t_end - (t_begin + j * kTile));
#pragma unroll
            for (int rr = 0; rr < 2; ++rr) {
                const int t = u + 64 * rr;
                const bool valid = t < nvalid;
                sm.cscl[cb][t] = valid ? sm.scl[s][(t / geo.P) * max(32, geo.P) + t % geo.P] : 0.f;
                const uint32_t src = ptx::smem_addr(sm.codes[s]) + t * 128;
                const uint32_t dst = ptx::smem_addr(sm.cvt[cb]) + t * 128;
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    uint4 v = make_uint4(0, 0, 0, 0);
                    if (valid)
                        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                                     : "r"(src + (((c ^ (t & 7))) << 4)));
                    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
                    uint32_t hv[8];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        hv[2 * e] = e4m3x2_to_f16x2(w[e]);
                        hv[2 * e + 1] = e4m3x2_to_f16x2(w[e] >> 16);
                    }
                    // codes 16c .. 16c + 15: dims of half c / 4, chunks 2 (c % 4) and + 1 there
                    const int half = c >> 2, ch = 2 * (c & 3);
                    const uint32_t d0 = dst + half * kHalfBytes + ((ch ^ (t & 7)) << 4);
                    const uint32_t d1 = dst + half * kHalfBytes + (((ch + 1) ^ (t & 7)) << 4);
                    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(d0), "r"(hv[0]),
                                 "r"(hv[1]), "r"(hv[2]), "r"(hv[3])
                                 : "memory");
                    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(d1), "r"(hv[4]),
                                 "r"(hv[5]), "r"(hv[6]), "r"(hv[7])
                                 : "memory");
                }
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(&sm.empty[s]);   // the code stage is free again
                ptx::mbar_arrive(&sm.c_full[cb]);
            }
        }
    } else {
        // ------------------------------------------------------------------ compute -----
        const int t = tid;                                  // 0..127: token / output dim
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        const float sl2 = geo.scale * kLog2e;
        bool ok = true;


        // Routed query: from the routing MMA (TMEM), or the composed query itself.
        float acc[kNG];
#pragma unroll
        for (int h = 0; h < kNG; ++h) acc[h] = 0.f;
        if (ok && route) {
            ok = ptx::bar_and(kBarComputeAnd, kTile, wait(&sm.r_full, 0));
            if (ok) {
                ptx::tc_fence_after();
                float rv[16];
                ptx::tmem_ld16(tmem + 2 * kN + lane_base, rv);
#pragma unroll
                for (int h = 0; h < kNG; ++h) acc[h] = h < G ? rv[h] : 0.f;
                ptx::tc_fence_before();
            }
        } else if (ok) {
#pragma unroll
            for (int h = 0; h < kNG; ++h)
                acc[h] = h < G ? __uint_as_float((uint32_t)a.q[((size_t)b * geo.Hq + g * G + h) * kD + t] << 16)
                               : 0.f;
        }
        ok = ptx::bar_and(kBarComputeAnd, kTile, ok);
        if (ok) {
            // half-precision hi/lo operand rows: n = h (hi), n = 8 + h (lo); column k = t
#pragma unroll
            for (int h = 0; h < kNG; ++h) {
                const float v = acc[h] * sl2;
                const __half hi = __float2half_rn(v);
                const __half lo = __float2half_rn(v - __half2float(hi));
                *reinterpret_cast<__half *>(sm.qr + qr_offset(h, t)) = hi;
                *reinterpret_cast<__half *>(sm.qr + qr_offset(kNG + h, t)) = lo;
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.qr_full);
        }

        float m[kNG], lsum[kNG], o[kNG], alpha_prev[kNG];
#pragma unroll
        for (int h = 0; h < kNG; ++h) {
            m[h] = -INFINITY;
            lsum[h] = 0.f;
            o[h] = 0.f;
            alpha_prev[h] = 0.f;
        }
        // O accumulation of tile j: o = o * alpha_j + O_j (thread = output dim t)
        auto correct = [&](int j, const float (&alpha)[kNG]) -> bool {
            const int ob = j & 1;
            if (!ptx::bar_and(kBarComputeAnd, kTile, wait(&sm.o_full[ob], (j >> 1) & 1))) return false;
            ptx::tc_fence_after();
            float ov[16];
            ptx::tmem_ld16(tmem + 2 * kN + ob * kN + lane_base, ov);
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.o_empty[ob]);
#pragma unroll
            for (int h = 0; h < kNG; ++h) o[h] = fmaf(o[h], alpha[h], ov[h] + ov[kNG + h]);
            return true;
        };

        for (int i = 0; ok && i < n_tiles; ++i) {
            const int sb = i & 1;
            if (!ptx::bar_and(kBarComputeAnd, kTile, wait(&sm.s_full[sb], (i >> 1) & 1))) {
                ok = false;
                break;
            }
            ptx::tc_fence_after();
            float sv[16];
            ptx::tmem_ld16(tmem + sb * kN + lane_base, sv);
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.s_empty[sb]);

            const int nvalid = min(kTile, t_end - (t_begin + i * kTile));
            const bool valid = t < nvalid;
            // the row scale of token t: written by the widening warps before c_full[i & 1],
            // which completed before this tile's score MMAs
            if (!ptx::bar_and(kBarComputeAnd, kTile, wait(&sm.c_full[sb], (i >> 1) & 1))) {
                ok = false;
                break;
            }
            const float scale_cur = sm.cscl[sb][t];
            float s[kNG], mx[kNG];
#pragma unroll
            for (int h = 0; h < kNG; ++h) {
                // the row scale multiplies the score column of token t
                s[h] = (valid && h < G) ? (sv[h] + sv[kNG + h]) * scale_cur : -INFINITY;
                mx[h] = s[h];
            }
            {
                const float wm = warp_max8(mx, lane);
                if ((lane & 3) == 0)
                    sm.red[sb][warp][((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1)] = wm;
            }
            ptx::bar_sync(kBarCompute, kTile);
            float alpha[kNG], p[kNG];
#pragma unroll
            for (int h = 0; h < kNG; ++h) {
                float tmax = sm.red[sb][0][h];
#pragma unroll
                for (int w = 1; w < kComputeWarps; ++w) tmax = fmaxf(tmax, sm.red[sb][w][h]);
                const float mn = fmaxf(m[h], tmax);
                const bool live = h < G;
                alpha[h] = live ? exp2f(m[h] - mn) : 0.f;
                p[h] = live ? exp2f(s[h] - mn) : 0.f;
                lsum[h] = fmaf(lsum[h], alpha[h], p[h]);
                m[h] = live ? mn : m[h];
            }
            // P^T row of token t, weights times the row scale: hi and lo halves
            {
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    split_h2(p[2 * e] * scale_cur, p[2 * e + 1] * scale_cur, hi[e], lo[e]);
                uint8_t *row = sm.p[sb] + (t >> 3) * 256 + (t & 7) * 16;
                *reinterpret_cast<uint4 *>(row) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                *reinterpret_cast<uint4 *>(row + 128) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.p_full[sb]);

            if (i >= 1 && !correct(i - 1, alpha_prev)) { ok = false; break; }
#pragma unroll
            for (int h = 0; h < kNG; ++h) alpha_prev[h] = alpha[h];
        }
        if (ok) ok = correct(n_tiles - 1, alpha_prev);

        if (ok) {
#pragma unroll
            for (int off = 16; off > 0; off >>= 1)
#pragma unroll
                for (int h = 0; h < kNG; ++h) lsum[h] += __shfl_xor_sync(0xffffffffu, lsum[h], off);
            const int rb = n_tiles & 1;
            if (lane == 0) {
#pragma unroll
                for (int h = 0; h < kNG; ++h) sm.red[rb][warp][h] = lsum[h];
            }
            ptx::bar_sync(kBarCompute, kTile);
#pragma unroll
            for (int h = 0; h < kNG; ++h) {
                if (h >= G) continue;
                float lt = 0.f;
#pragma unroll
                for (int w = 0; w < kComputeWarps; ++w) lt += sm.red[rb][w][h];
                const float val = o[h] / lt;
                const size_t bh = (size_t)b * geo.Hq + g * G + h;
                if (a.direct_out) {
                    if (a.out_dtype == KL_FP32) static_cast<float *>(a.out)[bh * kD + t] = val;
                    else static_cast<__nv_bfloat16 *>(a.out)[bh * kD + t] = __float2bfloat16_rn(val);
                } else {
                    const size_t slot = bh * geo.S + split;
                    a.part_o[slot * kD + t] = val;
                    if (t == 0) {
                        a.part_ml[slot * 2] = m[h] * kLn2;
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
}

// Quantizing append: one CTA per sequence, one warp per value head; lane j holds dims
// 4j .. 4j + 3. scale = max |v| / 448 (fp32), code = E4M3(v / scale) rounded to nearest even,
// saturating.
__global__ void __launch_bounds__(256)
    append_fp8_kernel(int Hkv, int P, int num_pages, int max_pages, const uint16_t *__restrict__ v_new,
                      const int32_t *__restrict__ block_table, const int32_t *__restrict__ positions,
                      uint8_t *__restrict__ codes, float *__restrict__ scales, int32_t *err) {
    const int b = blockIdx.x, lane = threadIdx.x & 31;
    const int pos = positions[b];
    if (pos < 0 || pos >= max_pages * P) {
        if (threadIdx.x == 0) raise_flag(err, KL_FLAG_BAD_POSITION);
        return;
    }
    const int page = block_table[(size_t)b * max_pages + pos / P];
    if (page < 0 || page >= num_pages) {
        if (threadIdx.x == 0) raise_flag(err, KL_FLAG_BAD_PAGE);
        return;
    }
    for (int g = threadIdx.x >> 5; g < Hkv; g += blockDim.x >> 5) {
        const uint2 w = reinterpret_cast<const uint2 *>(v_new + ((size_t)b * Hkv + g) * kD)[lane];
        const float v[4] = {bf16lo(w.x), bf16hi(w.x), bf16lo(w.y), bf16hi(w.y)};
        float amax = fmaxf(fmaxf(fabsf(v[0]), fabsf(v[1])), fmaxf(fabsf(v[2]), fabsf(v[3])));
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
        const float s = __fdiv_rn(amax, 448.0f);
        uint32_t packed = 0;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const uint32_t c = s > 0.f
                                   ? (uint32_t)__nv_cvt_float_to_fp8(__fdiv_rn(v[e], s), __NV_SATFINITE, __NV_E4M3)
                                   : 0u;
            packed |= c << (8 * e);
        }
        const size_t row = ((size_t)page * Hkv + g) * P + pos % P;
        reinterpret_cast<uint32_t *>(codes + row * kD)[lane] = packed;
        if (lane == 0) scales[row] = s;
    }
}

// Quantize a whole bf16 cache [rows][128] into codes [rows][128] and row scales [rows]: one warp
// per row, the same arithmetic as the append.
__global__ void __launch_bounds__(256)
    quantize_rows_kernel(size_t rows, const uint16_t *__restrict__ v, uint8_t *__restrict__ codes,
                         float *__restrict__ scales) {
    const int lane = threadIdx.x & 31;
    const size_t warps = (size_t)gridDim.x * (blockDim.x >> 5);
    for (size_t row = (size_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < rows;
         row += warps) {
        const uint2 w = reinterpret_cast<const uint2 *>(v + row * kD)[lane];
        const float x[4] = {bf16lo(w.x), bf16hi(w.x), bf16lo(w.y), bf16hi(w.y)};
        float amax = fmaxf(fmaxf(fabsf(x[0]), fabsf(x[1])), fmaxf(fabsf(x[2]), fabsf(x[3])));
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
        const float s = __fdiv_rn(amax, 448.0f);
        uint32_t packed = 0;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const uint32_t c = s > 0.f
                                   ? (uint32_t)__nv_cvt_float_to_fp8(__fdiv_rn(x[e], s), __NV_SATFINITE, __NV_E4M3)
                                   : 0u;
            packed |= c << (8 * e);
        }
        reinterpret_cast<uint32_t *>(codes + row * kD)[lane] = packed;
        if (lane == 0) scales[row] = s;
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

}  // namespace

cudaError_t launch_decode_fp8(const DecodeArgs &a, const float *v_scales) {
    const Geometry &g = a.geo;
    if (g.B == 0) return cudaSuccess;
    const uint64_t rows = (uint64_t)g.num_pages * g.Hkv * g.P;
    CUtensorMap cmap, smap, wmap, qmap;
    // codes [rows][128] u8, one box = one page of one head; scales [pages * Hkv][P] fp32
    if (!encode2d(&cmap, CU_TENSOR_MAP_DATA_TYPE_UINT8, a.v_cache, kD, rows, kD, kD, (uint32_t)g.P,
                  CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    if (!encode2d(&smap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, v_scales, (uint64_t)g.P,
                  (uint64_t)g.num_pages * g.Hkv, (uint64_t)g.P * 4, (uint32_t)g.P, 1,
                  CU_TENSOR_MAP_SWIZZLE_NONE))
        return cudaErrorInvalidValue;
    wmap = qmap = cmap;
    if (a.w_r) {
        if (!encode2d(&wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.w_r, kD, (uint64_t)g.Hkv * kD,
                      kD * 2, 64, kD, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
        if (!encode2d(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.q, kD, (uint64_t)g.B * g.Hq, kD * 2,
                      64, (uint32_t)g.G, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
    }
    const size_t smem = sizeof(Smem8) + 1024;
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(decode_fp8_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g.S, g.Hkv, g.B);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = a.stream;
    return cudaLaunchKernelEx(&cfg, decode_fp8_kernel, cmap, smap, wmap, qmap, a);
}

cudaError_t launch_append_fp8(const Geometry &g, const uint16_t *v_new, const int32_t *block_table,
                              const int32_t *positions, uint8_t *codes, float *scales, int32_t *err,
                              cudaStream_t stream) {
    if (g.B == 0) return cudaSuccess;
    append_fp8_kernel<<<g.B, 256, 0, stream>>>(g.Hkv, g.P, g.num_pages, g.max_pages, v_new,
                                               block_table, positions, codes, scales, err);
    return cudaGetLastError();
}

cudaError_t launch_quantize_fp8(size_t rows, const uint16_t *v, uint8_t *codes, float *scales,
                                cudaStream_t stream) {
    if (rows == 0) return cudaSuccess;
    const size_t blocks = (rows + 7) / 8;
    const unsigned grid = (unsigned)(blocks < 65535 * 16 ? blocks : 65535 * 16);
    quantize_rows_kernel<<<grid, 256, 0, stream>>>(rows, v, codes, scales);
    return cudaGetLastError();
}

}  // namespace kl
