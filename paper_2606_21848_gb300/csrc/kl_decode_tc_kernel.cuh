// Tensor-core split-sequence decode for sm_103a: TMA page gathers into a shared-memory ring,
// tcgen05 MMAs with TMEM accumulators, warp-specialized roles.
//
// One CTA per (run of splits, value head g, sequence b, block of up to 8 of the group's query
// heads: groups of more than 8 heads run ceil(G / 8) sibling CTAs that read the same pages);
// head_dim 128 or 64. The value-space routing (Section 2.2: q_r = q W^R) runs first, as tensor-core MMAs on
// W^R tiles that stream through the ring, into a split-bf16 operand (q_r * scale * log2 e =
// hi + lo, both bf16) for the G heads of the group.
// Then each 128-token tile of cached value rows V_t [128 x 128] (Section 3) is used twice by
// the tensor cores, straight from one shared-memory copy:
//
//   scores   S^T = V_t . [q_hi | q_lo]^T        M = 128 tokens, N = 16, K = 128 (A K-major)
//   output   O^T = V_t^T . [p_hi | p_lo]        M = 128 dims,   N = 16, K = 128 (A MN-major)
//
// so every cached row is read from HBM exactly once for both roles. The hi/lo split of the
// routed query and of the softmax weights keeps about 16 significant bits where a plain bf16
// operand would keep 8; the tensor cores have ample headroom for the doubled N.
//
// Roles (224 or 352 threads, two CTAs per SM):
//   compute    routing prologue; per tile read S from TMEM (thread = token), online softmax in
//              base 2 against a lazy per-head reference (moved only when a score passes it by
//              more than 2), write P^T to shared memory; read O from TMEM (thread = output dim)
//              and accumulate with rescaling; epilogue writes the output or the split state, or
//              merges the splits. Groups of 5-8 heads: warps 0-3, one per TMEM lane quarter, all
//              8 (padded) heads each (KH 8; the 70B batch is HBM-bound there and ran 2 % slower
//              on eight warps). Sibling CTAs of larger groups, whose tiles are computed once per
//              sibling and so bound by the compute warps: warps 0-7, warps w and w + 4 sharing
//              lane quarter w % 4 with 4 heads each (KH 4), twice the warps to hide each one's
//              latencies. Groups of up to 4: the same eight warps with 2 heads each (KH 2), so
//              the live heads alone are computed (6.7 % faster on the 4-head long context).
//   next warp  producer: block-table lookups and TMA loads of (page, head) tiles.
//   next       score-MMA issuer (one elected lane; also the routing MMA) and TMEM owner.
//   last       output-MMA issuer. Two issuing threads raise the SM's MMA issue rate (each
//              small-N tcgen05.mma costs tens of cycles to issue) and keep the output MMA of
//              one tile from waiting behind the score MMA of the next.
// Every wait is bounded (about one second); a wait that runs out raises KL_FLAG_TIMEOUT,
// makes every role leave its loop, drains outstanding copies and MMAs and frees TMEM.
//
// This header holds the kernel template and its launch for one head dim; kl_decode_tc.cu
// instantiates head dim 128 and the host-side plan, kl_decode_tc64.cu head dim 64 and
// kl_decode_tc_groups.cu the CTAs of groups of more than 8 heads, so that they compile in
// parallel.
#pragma once

#include <cudaTypedefs.h>
#include <math.h>

#include "kl_internal.cuh"
#include "kl_tc_ptx.cuh"

namespace kl {
namespace {

constexpr int kD = 128;
constexpr int kTile = 128;                  // tokens per tile
constexpr int kNG = 8;                      // query heads per CTA (padded)
constexpr int kMaxGroup = 128;              // query heads per value head (16 CTAs of 8)
constexpr int kN = 2 * kNG;                 // MMA N: hi and lo halves
constexpr uint32_t kTileBytes = kTile * kD * 2;   // 32 KiB per cache tile
constexpr uint32_t kHalfBytes = kTileBytes / 2;   // one 64-dim half: 128 rows x 128 B
constexpr uint32_t kTmemCols = 64;                // S: 2 x 16 columns, O: 2 x 16 columns
constexpr uint32_t kTmemColsPq = 256;             // + one 16-column routing result per head
constexpr uint64_t kTimeoutNs = kDefaultWaitNs;   // bound of the drains
constexpr float kLazyW = 4.f;                     // reference slack: weights 2^(s - m) <= 4
// Warp roles for KH heads per compute warp: KH = 8, one compute warp per TMEM lane quarter;
// KH = 4 (the CTAs of groups of more than 8 heads) and KH = 2 (groups of up to 4 heads), two
// per quarter, the second of them taking the upper head block.
template <int KH>
struct Roles {
    static constexpr int kComputeWarps = KH == 8 ? 4 : 8;
    static constexpr int kComputeThreads = kComputeWarps * 32;
    static constexpr int kProducerWarp = kComputeWarps;
    static constexpr int kMmaWarp = kComputeWarps + 1;   // score MMAs (and routing); owns TMEM
    static constexpr int kPvWarp = kComputeWarps + 2;    // output MMAs
    static constexpr int kThreads = (kComputeWarps + 3) * 32;
};
// Named barriers of the compute threads (id 0 is __syncthreads).
constexpr uint32_t kBarCompute = 1;       // plain sync
constexpr uint32_t kBarComputeAnd = 2;    // sync + AND of a flag

// Maximum over the 32 lanes of a warp of each of KH = 2, 4 or 8 values by transposed halving:
// each exchange step sends half of the lane's values and keeps the other half, so lane l ends
// with the maximum of value e(l) = max_head<KH>(l): bit 4 of l (KH 2), 2 bit4 + bit3 (KH 4),
// 4 bit4 + 2 bit3 + bit2 (KH 8: 9 shuffles instead of 40).
template <int KH>
__device__ __forceinline__ float warp_max_k(const float (&x)[KH], int lane) {
    const bool b4 = lane & 16;
    float a1;
    if constexpr (KH == 8) {
        const bool b3 = lane & 8, b2 = lane & 4;
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
        const float send = b2 ? a2[0] : a2[1];
        const float keep = b2 ? a2[1] : a2[0];
        a1 = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 4));
    } else if constexpr (KH == 4) {
        const bool b3 = lane & 8;
        float a2[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const float send = b4 ? x[j] : x[j + 2];
            const float keep = b4 ? x[j + 2] : x[j];
            a2[j] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 16));
        }
        const float send = b3 ? a2[0] : a2[1];
        const float keep = b3 ? a2[1] : a2[0];
        a1 = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 8));
        a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 4));
    } else {
        static_assert(KH == 2, "two, four or eight heads per compute warp");
        const float send = b4 ? x[0] : x[1];
        const float keep = b4 ? x[1] : x[0];
        a1 = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 16));
        a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 8));
        a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 4));
    }
    a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 2));
    a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 1));
    return a1;
}

// The head (of the warp's KH) whose maximum lane l holds after warp_max_k, and whether l is
// the first lane that holds it (the one that publishes it).
template <int KH>
__device__ __forceinline__ int max_head(int lane) {
    if constexpr (KH == 8) return ((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1);
    else if constexpr (KH == 4) return ((lane >> 4) & 1) * 2 + ((lane >> 3) & 1);
    else return (lane >> 4) & 1;
}
template <int KH>
__device__ __forceinline__ bool max_writer(int lane) {
    return (lane & (32 / KH - 1)) == 0;
}

// The hi and lo columns of the warp's KH heads h0 .. h0 + KH - 1 in a 16-column TMEM row
// [hi of heads 0-7 | lo of heads 0-7] at column address `row` (lane base included): one load
// of the whole row for KH 8, two runs of KH columns otherwise.
template <int KH>
__device__ __forceinline__ void tmem_ld_heads(uint32_t row, int h0, float (&hi)[KH], float (&lo)[KH]) {
    if constexpr (KH == 8) {
        float v[16];
        ptx::tmem_ld16(row, v);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            hi[e] = v[e];
            lo[e] = v[8 + e];
        }
    } else {
        ptx::tmem_ld_two<KH>(row + h0, row + kNG + h0, hi, lo);
    }
}

// Column base + h0 + e of a 16-column TMEM row [hi of heads 0-7 | lo of heads 0-7]: the upper
// head block of a KH = 2 or 4 warp is picked with a select, so register arrays keep constant
// indices.
template <int KH>
__device__ __forceinline__ float head_col(const float (&v)[16], int base, bool hh, int e) {
    if constexpr (KH == 8) return v[base + e];
    else return hh ? v[base + KH + e] : v[base + e];
}


template <bool kStandard>
struct Cfg {
    static constexpr int kStages = 3;
    static constexpr int kTilesPerStage = kStandard ? 2 : 1;   // K and V, or V only
};

template <bool kStandard>
struct __align__(1024) Smem {
    // Cache tiles, 128B-swizzled: [half (dims 0-63 | 64-127)][128 rows][128 B]. For the
    // K+V comparison the K tile follows the V tile of the same stage.
    uint8_t tiles[Cfg<kStandard>::kStages][Cfg<kStandard>::kTilesPerStage][kTileBytes];
    // Routed query operand [half][16 rows][128 B], 128B-swizzled, K-major.
    uint8_t qr[2 * kN * 128];
    // P^T operands, no swizzle, MN-major: [16 groups of 8 tokens][hi | lo][8 tokens][16 B].
    // During the routing prologue the first one holds the raw query, fp32 [k][8].
    uint8_t p[2][kTile * kN * 2];
    float red[2][4][kNG];              // per lane quarter and head: tile maxima, row sums
    float lred[4][kNG];                // row sums of a split closed inside a CTA's run
    float mred[4][kNG];                // per lane quarter and head: largest score of a state
    uint64_t full[Cfg<kStandard>::kStages], empty[Cfg<kStandard>::kStages];
    uint64_t s_full[2], s_empty[2], p_full[2], o_full[2], o_empty[2];
    uint64_t qr_full, q_ready, r_full, drain, drain2, merge_full;
    int is_last;
    uint32_t tmem_base;
    int abort;
};

// Warp-collective bounded wait: every lane of the warp calls it in uniform control flow and
// gets the same answer. False when this CTA is aborting or the wait ran out (`limit` ns, about
// 1 s unless the library's limit was lowered), in which case the caller leaves its loop.
// The try_wait may suspend the thread for a hardware-defined time before it returns false;
// kExact (limits below kExactWaitNs) polls with the non-blocking test_wait instead, so that
// short limits hold exactly.
template <bool kExact>
struct Waiter {
    volatile int *abort;
    int32_t *err;
    uint64_t limit;
    __device__ bool poll(uint64_t *bar, uint32_t parity) const {
        if constexpr (kExact) return ptx::mbar_test_wait(bar, parity);
        else return ptx::mbar_try_wait(bar, parity);
    }
    __device__ bool operator()(uint64_t *bar, uint32_t parity) const {
        bool ok = poll(bar, parity);
        if (!ok) {
            const uint64_t t0 = ptx::globaltimer();
            while (true) {
                if (poll(bar, parity)) { ok = true; break; }
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

template <int N>
struct Vec {
    float v[N];
};

// The split-bf16 form of two values a and b: hi = their bf16 roundings, lo = the bf16 roundings
// of the remainders, each pair packed as a | b << 16 (a + b keeps about 16 significant bits).
__device__ __forceinline__ void split_bf16x2(float a, float b, uint32_t &hi, uint32_t &lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    hi = *reinterpret_cast<const uint32_t *>(&h);
    const float ha = __uint_as_float(hi << 16), hb = __uint_as_float(hi & 0xffff0000u);
    const __nv_bfloat162 l = __floats2bfloat162_rn(a - ha, b - hb);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo_half, float hi_half) {
    const uint32_t a = __bfloat16_as_ushort(__float2bfloat16_rn(lo_half));
    const uint32_t b = __bfloat16_as_ushort(__float2bfloat16_rn(hi_half));
    return a | (b << 16);
}

// Byte offset of element (row n, column k) in a K-major, 128B-swizzled operand of 16 rows
// and 128 columns laid out as [half][16 rows][128 B].
__device__ __forceinline__ uint32_t qr_offset(int n, int k) {
    const int half = k >> 6, kk = k & 63;
    return half * (kN * 128) + (n >> 3) * 1024 + (n & 7) * 128 + (((kk >> 3) ^ (n & 7)) << 4) +
           ((kk & 7) << 1);
}

// Arrival of one split of a (b, g) unit on its counter in the workspace: true for the last of
// the unit's n splits. The increment wraps the counter back to zero on that arrival, so the
// workspace is ready for the next call without any reset; one atomic per split, no retry.
// Acquire-release at GPU scope: it publishes the split state that this CTA's threads wrote
// before the CTA barrier that precedes it, and, for the last arrival, makes every other
// split's state visible to the threads that synchronize with this one afterwards.
__device__ __forceinline__ bool arrive_last(unsigned int *counter, int n) {
    unsigned int old;
    asm volatile("atom.acq_rel.gpu.global.inc.u32 %0, [%1], %2;"
                 : "=r"(old)
                 : "l"(counter), "r"((unsigned int)(n - 1))
                 : "memory");
    return old == (unsigned int)(n - 1);
}

// Merge of the n_u split states of (b, g) by the compute warps of the CTA that finished last
// (t = the thread's index among them)
// (kl_combine's formula). Up to eight splits: direct loads. More: the cache ring is idle by
// now; the {m, l} table and the normalized weights go to its front, and TMA bulk copies bring
// the state rows through the rest, folded by thread (head, 4 dims) from shared memory.
template <int KH, int D, typename SmemT, typename WaitT>
__device__ void merge_states(SmemT &sm, const DecodeArgs &a, int b, int qh0, int G, int n_u,
                             int t, int warp, int lane, const WaitT &wait) {
    constexpr int kComputeWarps = Roles<KH>::kComputeWarps;
    constexpr int kComputeThreads = Roles<KH>::kComputeThreads;
    const Geometry &geo = a.geo;
    // a state row holds D floats: lanes below D / 4 fold them
    const bool lane_live = lane < D / 4;
    if (n_u <= 8) {
        // Few splits: thread (head, 4 dims) loads its n_u {m, l} pairs and state rows at once
        // (one round trip) and folds them; no staging.
        const float2 *ml = reinterpret_cast<const float2 *>(a.part_ml);
        for (int h = warp; h < G; h += kComputeWarps) {
            const size_t bh = (size_t)b * geo.Hq + qh0 + h;
            const float4 *po = reinterpret_cast<const float4 *>(a.part_o + bh * geo.S * D) + lane;
            float2 v[8];
            float4 r[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (j < n_u) {
                    v[j] = __ldcg(ml + bh * geo.S + j);
                    r[j] = lane_live ? __ldcg(po + (size_t)j * (D / 4)) : make_float4(0.f, 0.f, 0.f, 0.f);
                }
            }
            float M = -INFINITY;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (j < n_u && v[j].y > 0.f) M = fmaxf(M, v[j].x);
            float z = 0.f;
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (j < n_u && v[j].y > 0.f) {
                    const float w = v[j].y * expf(v[j].x - M);
                    z += w;
                    acc.x = fmaf(w, r[j].x, acc.x);
                    acc.y = fmaf(w, r[j].y, acc.y);
                    acc.z = fmaf(w, r[j].z, acc.z);
                    acc.w = fmaf(w, r[j].w, acc.w);
                }
            }
            const float inv = z > 0.f ? 1.f / z : 0.f;
            acc.x *= inv; acc.y *= inv; acc.z *= inv; acc.w *= inv;
            const size_t oi = bh * D + 4 * lane;
            if (!lane_live) continue;
            if (a.out_dtype == KL_FP32) {
                *reinterpret_cast<float4 *>(static_cast<float *>(a.out) + oi) = acc;
            } else {
                __nv_bfloat16 *o16 = static_cast<__nv_bfloat16 *>(a.out) + oi;
                *reinterpret_cast<uint2 *>(o16) = make_uint2(pack_bf16(acc.x, acc.y), pack_bf16(acc.z, acc.w));
            }
        }
        return;
    }
    // Many splits: the {m, l} table and the weights go to the front of the idle ring, then the
    // state rows stream through the rest of it, `cap` splits per head per bulk-copy round.
    uint8_t *ring = &sm.tiles[0][0][0];
    constexpr uint32_t kRingBytes = sizeof(sm.tiles);
    float2 *tab = reinterpret_cast<float2 *>(ring);                        // [G][n_u] {m, l}
    float *wt = reinterpret_cast<float *>(tab + G * n_u);                  // [G][n_u] weights
    const uint32_t table_bytes = ((uint32_t)G * n_u * 12u + 1023u) & ~1023u;
    float *rows = reinterpret_cast<float *>(ring + table_bytes);           // [G][cap][128]
    const int cap = (int)((kRingBytes - table_bytes) / ((uint32_t)G * D * sizeof(float)));
    const float2 *ml = reinterpret_cast<const float2 *>(a.part_ml);
    // The first round's state rows go out at once, so that their copy overlaps the {m, l}
    // loads and the weights (the ring is idle: every tile has been consumed).
    auto issue_rows = [&](int c0, int nrow) {
        if (t == 0) {
            ptx::fence_proxy_async_global();
            ptx::mbar_arrive_expect_tx(&sm.merge_full, (uint32_t)(G * nrow * D * sizeof(float)));
            for (int h = 0; h < G; ++h)
                ptx::bulk_load(rows + (size_t)h * cap * D,
                               a.part_o + (((size_t)b * geo.Hq + qh0 + h) * geo.S + c0) * D,
                               (uint32_t)(nrow * D * sizeof(float)), &sm.merge_full);
        }
    };
    issue_rows(0, min(cap, n_u));
    for (int i = t; i < G * n_u; i += kComputeThreads) {
        const int h = i / n_u, j = i - h * n_u;
        tab[i] = __ldcg(ml + ((size_t)b * geo.Hq + qh0 + h) * geo.S + j);
    }
    ptx::bar_sync(kBarCompute, kComputeThreads);
    for (int h = warp; h < G; h += kComputeWarps) {
        float M = -INFINITY;
        for (int j = lane; j < n_u; j += 32) {
            const float2 v = tab[h * n_u + j];
            if (v.y > 0.f) M = fmaxf(M, v.x);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
        float z = 0.f;
        for (int j = lane; j < n_u; j += 32) {
            const float2 v = tab[h * n_u + j];
            const float w = (v.y > 0.f && M != -INFINITY) ? v.y * expf(v.x - M) : 0.f;
            wt[h * n_u + j] = w;
            z += w;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(0xffffffffu, z, off);
        const float inv = z > 0.f ? 1.f / z : 0.f;
        for (int j = lane; j < n_u; j += 32) wt[h * n_u + j] *= inv;
    }
    // warp w: head w (+ kComputeWarps for a second pass), lane: dims 4 lane .. + 3
    float4 acc[2] = {make_float4(0.f, 0.f, 0.f, 0.f), make_float4(0.f, 0.f, 0.f, 0.f)};
    int round = 0;
    for (int c0 = 0; c0 < n_u; c0 += cap, ++round) {
        const int nrow = min(cap, n_u - c0);
        // every thread is done with the previous chunk (and the weights are written)
        ptx::fence_proxy_async_smem();
        ptx::bar_sync(kBarCompute, kComputeThreads);
        if (c0 > 0) issue_rows(c0, nrow);
        if (!ptx::bar_and(kBarComputeAnd, kComputeThreads, wait(&sm.merge_full, round & 1))) {
            // gave up: this round's copies must still land before the CTA's shared memory goes
            const uint64_t t0 = ptx::globaltimer();
            while (!ptx::mbar_try_wait(&sm.merge_full, round & 1) &&
                   ptx::globaltimer() - t0 < kTimeoutNs) {
            }
            return;
        }
#pragma unroll
        for (int pass = 0; pass < 2; ++pass) {
            const int h = warp + pass * kComputeWarps;
            if (h >= G || !lane_live) continue;
            const float4 *po = reinterpret_cast<const float4 *>(rows + (size_t)h * cap * D) + lane;
            const float *w = wt + h * n_u + c0;
#pragma unroll 4
            for (int j = 0; j < nrow; ++j) {
                const float wj = w[j];
                if (wj != 0.f) {
                    const float4 v = po[(size_t)j * (D / 4)];
                    acc[pass].x = fmaf(wj, v.x, acc[pass].x);
                    acc[pass].y = fmaf(wj, v.y, acc[pass].y);
                    acc[pass].z = fmaf(wj, v.z, acc[pass].z);
                    acc[pass].w = fmaf(wj, v.w, acc[pass].w);
                }
            }
        }
    }
#pragma unroll
    for (int pass = 0; pass < 2; ++pass) {
        const int h = warp + pass * kComputeWarps;
        if (h >= G || !lane_live) continue;
        const size_t oi = ((size_t)b * geo.Hq + qh0 + h) * D + 4 * lane;
        if (a.out_dtype == KL_FP32) {
            *reinterpret_cast<float4 *>(static_cast<float *>(a.out) + oi) = acc[pass];
        } else {
            __nv_bfloat16 *o16 = static_cast<__nv_bfloat16 *>(a.out) + oi;
            *reinterpret_cast<uint2 *>(o16) =
                make_uint2(pack_bf16(acc[pass].x, acc[pass].y), pack_bf16(acc[pass].z, acc[pass].w));
        }
    }
}

// kPerSplit: the CTA runs several splits and writes a state for each (only when the caller
// gets the split states, or the combine kernel merges them, and spc > 1). KH: heads per compute
// warp (8, or 2 when G <= 4).
// kD64: head dim 64 (rows of 64 dims in HBM; the tiles stay 128 wide), else 128.
template <bool kStandard, bool kPerSplit, int KH, bool kExact, bool kD64>
__global__ void __launch_bounds__(Roles<KH>::kThreads, 2)
    decode_tc_kernel(const __grid_constant__ CUtensorMap vmap,
                     const __grid_constant__ CUtensorMap kmap,
                     const __grid_constant__ CUtensorMap wmap,
                     const __grid_constant__ CUtensorMap qmap, const DecodeArgs a) {
    using S = Smem<kStandard>;
    constexpr int NS = Cfg<kStandard>::kStages;
    constexpr int kComputeWarps = Roles<KH>::kComputeWarps;
    constexpr int kComputeThreads = Roles<KH>::kComputeThreads;
    constexpr int kProducerWarp = Roles<KH>::kProducerWarp;
    constexpr int kMmaWarp = Roles<KH>::kMmaWarp;
    constexpr int kPvWarp = Roles<KH>::kPvWarp;
    extern __shared__ uint8_t smem_raw[];
    S &sm = *reinterpret_cast<S *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                   ~uintptr_t(1023));

    const Geometry &geo = a.geo;
    // A CTA runs geo.spc consecutive splits of one (b, g) (one split unless a launch of one CTA
    // per split would not fit in one wave); it keeps one softmax state per split. A group of
    // more than 8 query heads is served by geo.nhb sibling CTAs, adjacent in blockIdx.x, each
    // for up to 8 of its heads: the siblings read the same pages at about the same time, so
    // the second and later reads of a page are served by L2.
    // At head dim 64 a CTA takes two value heads g and g + 1 (geo.vpc = 2): their rows sit side
    // by side in the 128-wide tile (dims 0-63: head g, 64-127: head g + 1), W^R[g] and W^R[g + 1]
    // form the diagonal blocks of a block-diagonal routing tile, and each query head keeps the
    // half of its routed query that belongs to its value head, so the 128-wide MMAs compute
    // both heads' products at once.
    const int hb = blockIdx.x % geo.nhb, cta = blockIdx.x / geo.nhb;
    const int g = blockIdx.y * geo.vpc, b = blockIdx.z;
    const int split0 = cta * geo.spc;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool pair = kD64 && geo.vpc == 2;
    const int G = pair ? 2 * geo.G : min(kNG, geo.G - kNG * hb);   // query heads of this CTA
    const int qh0 = g * geo.G + kNG * hb;         // its first query head within the sequence
    // Head dim of the rows in HBM: 128, or 64. Without a second value head, a 64-dim row lands
    // in the first 64-dim half of its tile row; the second halves, the rows past 64 of a W^R
    // tile and the second half of the query operand are zero for the whole launch, so the
    // 128-dim MMAs give the 64-dim products. (With two heads only the routing tile's
    // off-diagonal blocks rely on the zeros.)
    constexpr int D = kD64 ? 64 : kD;
    // The tile dims that CTA head h reads and writes, as its first output dim: [dim0(h),
    // dim0(h) + D).
    auto dim0 = [&](int h) { return pair && h >= geo.G ? 64 : 0; };

    // The routing runs on the tensor cores: W^R[g] (one per value head) or the G matrices
    // W^R[qh0 + h] (one per query head) arrive by TMA as ring positions 0 .. route_tiles - 1,
    // with the group's query rows, and the cache tiles follow.
    // routing on the tensor cores unless the query arrives routed: pre-routed fp32 queries, or
    // the composed query q = x W^Q W^R of Section 2.1 (no W^R given)
    const bool tc_route = !kStandard && a.q_routed == nullptr && a.w_r != nullptr;
    const bool route_pq = tc_route && geo.wr_per_qh;
    const int route_tiles = !tc_route ? 0 : route_pq ? G : 1;
    const int ro = route_tiles;
    const uint32_t tmem_cols = route_pq ? kTmemColsPq : kTmemCols;

    // Loads that do not depend on one another go out first, so their latency overlaps the
    // set-up: the length, the append position and (producer) the split's first block-table
    // entries, 32 pages per warp load, two batches.
    const int L_raw = a.seq_lens[b];
    const int pos_raw = a.v_new ? a.positions[b] : -1;
    const int t_begin = split0 * geo.chunk;
    const int first_page = t_begin / geo.P;
    const int32_t *bt = a.block_table + (size_t)b * geo.max_pages;
    int bt_cur = -1, bt_nxt = -1;
    if (warp == kProducerWarp) {
        if (first_page + lane < geo.max_pages) bt_cur = bt[first_page + lane];
        if (first_page + 32 + lane < geo.max_pages) bt_nxt = bt[first_page + 32 + lane];
    }

    if (tid == 0) {
        for (int s = 0; s < NS; ++s) {
            ptx::mbar_init(&sm.full[s], 1);
            ptx::mbar_init(&sm.empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(&sm.s_full[i], 1);
            ptx::mbar_init(&sm.s_empty[i], kComputeWarps);
            ptx::mbar_init(&sm.p_full[i], kComputeWarps);
            ptx::mbar_init(&sm.o_full[i], 1);
            ptx::mbar_init(&sm.o_empty[i], kComputeWarps);
        }
        ptx::mbar_init(&sm.qr_full, kComputeWarps);
        ptx::mbar_init(&sm.q_ready, kComputeWarps);
        ptx::mbar_init(&sm.r_full, 1);
        ptx::mbar_init(&sm.merge_full, 1);
        ptx::mbar_init(&sm.drain, 1);
        ptx::mbar_init(&sm.drain2, 1);
        sm.abort = 0;
        ptx::fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        ptx::tmem_alloc(&sm.tmem_base, tmem_cols);
        ptx::tmem_relinquish();
    }
    if (D != kD) {
        // zeros under the halves that TMA never writes (the ring and the query operand); the
        // fence orders these writes before the copies and MMAs issued after the barrier below
        uint4 *z = reinterpret_cast<uint4 *>(&sm.tiles[0][0][0]);
        for (uint32_t i = tid; i < sizeof(sm.tiles) / 16; i += blockDim.x) z[i] = make_uint4(0, 0, 0, 0);
        uint4 *zq = reinterpret_cast<uint4 *>(sm.qr);
        for (uint32_t i = tid; i < sizeof(sm.qr) / 16; i += blockDim.x) zq[i] = make_uint4(0, 0, 0, 0);
        ptx::fence_proxy_async_smem();
    }
    if (warp == kProducerWarp && lane == 0) {
        ptx::prefetch_tensormap(&vmap);
        if (kStandard) ptx::prefetch_tensormap(&kmap);
        if (tc_route) {
            ptx::prefetch_tensormap(&wmap);
            ptx::prefetch_tensormap(&qmap);
        }
    }
    // Ring position r < route_tiles: W^R as the MN-major A operand [j half][128 k rows][128 B];
    // position 0 also brings the group's query rows as the K-major B operand (rows 0..G-1 of
    // the q_r buffer). Issued by the producer warp.
    auto issue_route = [&](int r) {
        const int s = r % NS;
        if (lane == 0) {
            // W^R: two 64-column halves of 128 rows; or (head dim 64) one box of 64 x 64 at
            // the top left, and with two value heads the second head's box at the bottom
            // right (rows and columns 64-127; per query head: the box of the head's half).
            // The query rows go to both 64-dim halves of the operand when two heads share
            // the tile (each head keeps its own half of the result).
            const int wrow = (route_pq ? qh0 + r : g) * D;
            const bool two_q = D == kD || pair;
            const int nbox = D == kD ? 2 : (pair && !route_pq) ? 2 : 1;
            const uint32_t w_off = pair && route_pq && r >= geo.G ? kHalfBytes + 64u * 128u : 0u;
            ptx::mbar_arrive_expect_tx(&sm.full[s], (D == kD ? kTileBytes : (uint32_t)nbox * 64u * 128u) +
                                                        (r == 0 ? (two_q ? 2u : 1u) * (uint32_t)geo.qbox * 128u : 0u));
            if (D == kD) {
                ptx::tma_load_2d(sm.tiles[s][0], &wmap, &sm.full[s], 0, wrow);
                ptx::tma_load_2d(sm.tiles[s][0] + kHalfBytes, &wmap, &sm.full[s], 64, wrow);
            } else {
                ptx::tma_load_2d(sm.tiles[s][0] + w_off, &wmap, &sm.full[s], 0, wrow);
                if (nbox == 2)
                    ptx::tma_load_2d(sm.tiles[s][0] + kHalfBytes + 64u * 128u, &wmap, &sm.full[s], 0,
                                     wrow + D);
            }
            if (r == 0) {
                ptx::tma_load_2d(sm.qr, &qmap, &sm.full[s], 0, b * geo.Hq + qh0);
                if (two_q)
                    ptx::tma_load_2d(sm.qr + kN * 128, &qmap, &sm.full[s], D == kD ? 64 : 0,
                                     b * geo.Hq + qh0);
            }
        }
        __syncwarp();
    };

    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    // a kernel launched behind this one as a programmatic dependent (the combine of the split
    // states, the latent expansion) may start setting up once every CTA is here
    grid_dep_launch();
    // The routing loads that fit the ring depend on nothing the CTA still reads (the length,
    // the block table), so they go out at once: the routed query is then ready about when
    // the first cache tile lands.
    const int early_route = route_tiles < NS ? route_tiles : NS;
    if (warp == kProducerWarp)
        for (int r = 0; r < early_route; ++r) issue_route(r);

    int L = L_raw;
    if (L < 0 || L > geo.max_pages * geo.P) {
        if (tid == 0 && cta == 0 && g == 0) raise_flag(a.err, KL_FLAG_BAD_LENGTH);
        L = 0;
    }
    const int t_end = min(t_begin + geo.spc * geo.chunk, L);
    const int n_tiles = t_end > t_begin ? (t_end - t_begin + kTile - 1) / kTile : 0;

    // Fused append: the CTA whose splits hold row positions[b] owns the current token's row.
    const bool pos_ok = pos_raw >= 0 && pos_raw < geo.max_pages * geo.P;
    if (a.v_new && !pos_ok && tid == 0 && cta == 0 && g == 0)
        raise_flag(a.err, KL_FLAG_BAD_POSITION);
    const bool app_owner = a.v_new && pos_ok && pos_raw / (geo.chunk * geo.spc) == cta;

    // Empty split, no pipeline: in the split-state layout an empty state; otherwise the split
    // of a zero-length sequence writes the zero output, and the empty splits of a longer
    // sequence take no part (the merge counts only the splits that hold tokens).
    if (n_tiles == 0) {
        if (app_owner && warp < geo.vpc) {
            const int page = bt[pos_raw / geo.P];
            const int gv = g + warp;                  // one warp per value head of the CTA
            if (page >= 0 && page < geo.num_pages) {
                const size_t off = (((size_t)page * geo.Hkv + gv) * geo.P + pos_raw % geo.P) * D;
                const uint16_t *src = a.v_new + ((size_t)b * geo.Hkv + gv) * D;
                if (D == kD)
                    reinterpret_cast<uint2 *>(a.cache_rw + off)[lane] = reinterpret_cast<const uint2 *>(src)[lane];
                else
                    reinterpret_cast<uint32_t *>(a.cache_rw + off)[lane] = reinterpret_cast<const uint32_t *>(src)[lane];
            } else if (lane == 0) {
                raise_flag(a.err, KL_FLAG_BAD_PAGE);
            }
        }
        if (tid < D) {
            for (int h = 0; h < G; ++h) {
                const size_t bh = (size_t)b * geo.Hq + qh0 + h;
                if (a.merge_inside) {
                    if (L == 0 && cta == 0) {
                        if (a.out_dtype == KL_FP32) static_cast<float *>(a.out)[bh * D + tid] = 0.f;
                        else static_cast<__nv_bfloat16 *>(a.out)[bh * D + tid] = __float2bfloat16_rn(0.f);
                    }
                } else if (a.direct_out) {
                    if (a.out_dtype == KL_FP32) static_cast<float *>(a.out)[bh * D + tid] = 0.f;
                    else static_cast<__nv_bfloat16 *>(a.out)[bh * D + tid] = __float2bfloat16_rn(0.f);
                } else {
                    for (int sp = split0; sp < min(split0 + geo.spc, geo.S); ++sp) {
                        const size_t slot = bh * geo.S + sp;
                        a.part_o[slot * D + tid] = 0.f;
                        if (tid == 0) {
                            a.part_ml[slot * 2] = -INFINITY;
                            a.part_ml[slot * 2 + 1] = 0.f;
                        }
                    }
                }
            }
        }
        if (warp == kMmaWarp) ptx::tmem_dealloc(sm.tmem_base, tmem_cols);
        // the routing loads issued at the start land before the shared memory goes away
        if (warp == kProducerWarp) {
            for (int r = 0; r < early_route; ++r) {
                const uint64_t t0 = ptx::globaltimer();
                while (!ptx::mbar_try_wait(&sm.full[r], 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
                }
            }
        }
        return;
    }

    const uint32_t tmem = sm.tmem_base;
    int issued = 0;                 // ring uses whose copies the producer issued
    const Waiter<kExact> wait{&sm.abort, a.err, a.wait_ns};

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------------ producer ----
        const int P = geo.P;
        const int ppt = kTile / P;                   // pages per tile (<= 8)
        const int end_page = (t_end + P - 1) / P;
        const uint32_t page_bytes = (uint32_t)P * 128u;   // one half of one page
        bool bad = false;
        issued = 0;
        // The new token's row (fused append), 8 bytes per lane, written just before the loads of
        // the tile that holds it (or first, when it lies past the sequence's end).
        // (head dim 64: 4 bytes per lane, and with two value heads the second head's row in
        // app_val.y; the rows of one page and position lie P * D elements apart)
        int app_tile = -1;
        size_t app_off = 0;
        uint2 app_val = make_uint2(0, 0);
        if (app_owner) {
            const int page = bt[pos_raw / P];
            if (page >= 0 && page < geo.num_pages) {
                app_tile = pos_raw < t_end ? (pos_raw - t_begin) / kTile : 0;
                app_off = (((size_t)page * geo.Hkv + g) * P + pos_raw % P) * D;
                const uint16_t *src = a.v_new + ((size_t)b * geo.Hkv + g) * D;
                if (D == kD)
                    app_val = reinterpret_cast<const uint2 *>(src)[lane];
                else
                    app_val = make_uint2(reinterpret_cast<const uint32_t *>(src)[lane],
                                         pair ? reinterpret_cast<const uint32_t *>(src + D)[lane] : 0u);
            } else if (lane == 0) {
                raise_flag(a.err, KL_FLAG_BAD_PAGE);
            }
        }
        // Ring positions 0 .. route_tiles - 1: the W^R matrices (the first early_route of them
        // went out at the start).
        for (int r = 0; r < route_tiles; ++r) {
            if (r >= early_route) {
                if (r >= NS && !wait(&sm.empty[r % NS], ((r / NS) & 1) ^ 1)) break;
                issue_route(r);
            }
            issued = r + 1;
        }
        // Block-table entries of the split, 32 pages per warp load, one batch ahead (the
        // first two batches were loaded before the set-up).
        const int split_pages = end_page - first_page;
        int bt_batch = 0;
        for (int i = 0; i < n_tiles; ++i) {
            const int r = i + ro, s = r % NS;
            const int p0 = i * ppt;                       // first page of the tile in the split
            if ((p0 >> 5) != bt_batch) {
                bt_batch = p0 >> 5;
                bt_cur = bt_nxt;
                const int q = (bt_batch + 1) * 32 + lane;
                bt_nxt = q < split_pages ? bt[first_page + q] : -1;
            }
            int page = __shfl_sync(0xffffffffu, bt_cur, ((p0 & 31) + lane) & 31);
            const bool exists = lane < ppt && p0 + lane < split_pages;
            // with the ring full, a programmatic dependent sleeps until the routed queries exist
            if (a.pdl && r == NS) grid_dep_wait();
            if (r >= NS && !wait(&sm.empty[s], ((r / NS) & 1) ^ 1)) break;
            const bool in_range = exists && page >= 0 && page < geo.num_pages;
            if (exists && !in_range) bad = true;
            if (i == app_tile) {
                if (D == kD) {
                    reinterpret_cast<uint2 *>(a.cache_rw + app_off)[lane] = app_val;
                } else {
                    reinterpret_cast<uint32_t *>(a.cache_rw + app_off)[lane] = app_val.x;
                    if (pair)
                        reinterpret_cast<uint32_t *>(a.cache_rw + app_off + (size_t)P * D)[lane] = app_val.y;
                }
                ptx::fence_proxy_async_global();
                __syncwarp();
            }
            const unsigned mask = __ballot_sync(0xffffffffu, in_range);
            // two boxes per page: the 64-dim halves of one head's rows, or (head dim 64, two
            // value heads) head g's and head g + 1's rows; one box for a lone 64-dim head
            const bool two = D == kD || pair;
            const int x2 = D == kD ? 64 : 0;
            const int r2 = D == kD ? 0 : P;
            if (lane == 0)
                ptx::mbar_arrive_expect_tx(&sm.full[s], __popc(mask) * page_bytes * (two ? 2u : 1u) *
                                                            Cfg<kStandard>::kTilesPerStage);
            __syncwarp();
            if (in_range) {
                const int row = (page * geo.Hkv + g) * P;
                uint8_t *dst = sm.tiles[s][0] + lane * page_bytes;
                ptx::tma_load_2d(dst, &vmap, &sm.full[s], 0, row);
                if (two) ptx::tma_load_2d(dst + kHalfBytes, &vmap, &sm.full[s], x2, row + r2);
                if constexpr (kStandard) {
                    uint8_t *kd = sm.tiles[s][1] + lane * page_bytes;
                    ptx::tma_load_2d(kd, &kmap, &sm.full[s], 0, row);
                    if (two) ptx::tma_load_2d(kd + kHalfBytes, &kmap, &sm.full[s], x2, row + r2);
                }
            }
            issued = r + 1;
        }
        if (__any_sync(0xffffffffu, bad) && lane == 0) raise_flag(a.err, KL_FLAG_BAD_PAGE);

    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------- score MMA issuer -------
        // (a programmatic dependent sleeps until the routed queries exist instead of polling)
        if (a.pdl) grid_dep_wait();
        // Descriptors are formed once; a k step or a ring stage only moves the start address
        // (the low field, in 16-byte units; shared addresses stay below 256 KiB).
        constexpr uint32_t idesc_s = ptx::idesc_bf16(128, kN, false, false);
        constexpr uint32_t kStageBytes = sizeof(sm.tiles[0]);
        const uint32_t qr_addr = ptx::smem_addr(sm.qr);
        const uint64_t q_desc = ptx::smem_desc(qr_addr, 16, 1024, ptx::kSwizzle128B);
        const uint64_t k_desc = ptx::smem_desc(
            ptx::smem_addr(sm.tiles[0][Cfg<kStandard>::kTilesPerStage - 1]), 16, 1024, ptx::kSwizzle128B);
        bool ok = true;
        if (tc_route) {
            // q_r^T[128 j x 16] = W^R^T (MN-major, ring slot) . q^T (K-major rows of the q_r
            // buffer). One W^R per value head: into the columns of O buffer 0, which the first
            // output MMA reuses. One per query head: matrix h into its own 16 columns
            // (64 + 16 h), of which column h is q_r of head h.
            constexpr uint32_t idesc_r = ptx::idesc_bf16(128, kN, true, false);
            for (int r = 0; ok && r < route_tiles; ++r) {
                const int s = r % NS;
                ok = wait(&sm.full[s], (r / NS) & 1);
                if (!ok) break;
                ptx::tc_fence_after();
                if (lane == 0) {
                    const uint64_t w_desc = ptx::smem_desc(ptx::smem_addr(sm.tiles[s][0]), kHalfBytes,
                                                           1024, ptx::kSwizzle128B);
                    const uint32_t dst = route_pq ? tmem + 64 + 16 * r : tmem + 2 * kN;
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        const uint32_t qoff = (kk >> 2) * (kN * 128) + (kk & 3) * 32;
                        ptx::mma_bf16(dst, w_desc + ((kk * 2048) >> 4), q_desc + (qoff >> 4), idesc_r,
                                      kk > 0);
                    }
                    ptx::mma_commit(&sm.empty[s]);
                    if (r == route_tiles - 1) ptx::mma_commit(&sm.r_full);
                }
                __syncwarp();
            }
        }
        ok = ok && wait(&sm.qr_full, 0);
        if (ok) ptx::tc_fence_after();
        for (int i = 0; ok && i < n_tiles; ++i) {
            const int s = (i + ro) % NS, sb = i & 1;
            if (!wait(&sm.full[s], ((i + ro) / NS) & 1)) break;
            if (i >= 2 && !wait(&sm.s_empty[sb], ((i >> 1) - 1) & 1)) break;
            ptx::tc_fence_after();
            if (lane == 0) {
                const uint64_t a0 = k_desc + ((s * kStageBytes) >> 4);
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
        // Drain: every MMA this warp issued completes before TMEM is freed.
        if (lane == 0) ptx::mma_commit(&sm.drain);
        __syncwarp();
        {
            const uint64_t t0 = ptx::globaltimer();
            while (!ptx::mbar_try_wait(&sm.drain, 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
            }
        }
    } else if (warp == kPvWarp) {
        // ------------------------------------------------------ output MMA issuer -------
        if (a.pdl) grid_dep_wait();
        // A = V^T: MN-major SW128, 64-dim halves kHalfBytes apart (LBO), 8-token row groups
        //          1 KiB apart (SBO); 16 tokens per step.
        // B = P^T: MN-major, no swizzle; hi/lo blocks 128 B apart (SBO), 8-token groups 256 B
        //          apart (LBO).
        constexpr uint32_t idesc_o = ptx::idesc_bf16(128, kN, true, true);
        constexpr uint32_t kStageBytes = sizeof(sm.tiles[0]);
        const uint64_t v_desc =
            ptx::smem_desc(ptx::smem_addr(sm.tiles[0][0]), kHalfBytes, 1024, ptx::kSwizzle128B);
        const uint64_t p_desc = ptx::smem_desc(ptx::smem_addr(sm.p[0]), 256, 128, ptx::kSwizzleNone);
        constexpr uint32_t kPBytes = sizeof(sm.p[0]);
        for (int j = 0; j < n_tiles; ++j) {
            const int s = (j + ro) % NS, pb = j & 1;
            if (!wait(&sm.p_full[pb], (j >> 1) & 1)) break;
            if (j >= 2 && !wait(&sm.o_empty[pb], ((j >> 1) - 1) & 1)) break;
            ptx::tc_fence_after();
            const int nvalid = min(kTile, t_end - (t_begin + j * kTile));
            const int ksteps = (nvalid + 15) >> 4;
            if (lane == 0) {
                const uint64_t a0 = v_desc + ((s * kStageBytes) >> 4);
                const uint64_t b0 = p_desc + ((pb * kPBytes) >> 4);
                for (int kk = 0; kk < ksteps; ++kk)
                    ptx::mma_bf16(tmem + 2 * kN + pb * kN, a0 + ((kk * 2048) >> 4),
                                  b0 + ((kk * 512) >> 4), idesc_o, kk > 0);
                ptx::mma_commit(&sm.o_full[pb]);
                ptx::mma_commit(&sm.empty[s]);
            }
            __syncwarp();
        }
        if (lane == 0) ptx::mma_commit(&sm.drain2);
        __syncwarp();
        {
            const uint64_t t0 = ptx::globaltimer();
            while (!ptx::mbar_try_wait(&sm.drain2, 0) && ptx::globaltimer() - t0 < kTimeoutNs) {
            }
        }
    } else {
        // ------------------------------------------------------------------ compute -----
        // Warp w: TMEM lane quarter qd = w % 4 (thread t = 32 qd + lane is token t of a tile for
        // S and P, output dim t for O) and the KH heads h0 .. h0 + KH - 1, h0 = KH (w / 4).
        // Register arrays are indexed by constants only: the upper head block is picked with a
        // select, never with a warp-dependent index.
        const int qd = warp & 3;
        const int t = qd * 32 + lane;
        const bool hh = KH != 8 && warp >= 4;
        const int h0 = hh ? KH : 0;
        const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
        float *qf = reinterpret_cast<float *>(sm.p[0]);     // [k][8] raw query (prologue only)
        const float sl2 = geo.scale * kLog2e;
        bool ok = true;

        // Routing prologue: thread t obtains q_r[h][t] for its heads in fp32 from the routing
        // MMAs in TMEM, from the caller's pre-routed queries, or the query itself (already
        // composed with W^R, or unrouted for the K+V comparison).
        float acc[KH];
#pragma unroll
        for (int e = 0; e < KH; ++e) acc[e] = 0.f;
        if (tc_route) {
            ok = wait(&sm.r_full, 0);
            if (ok) {
                ptx::tc_fence_after();
                if (route_pq) {
#pragma unroll
                    for (int e = 0; e < KH; ++e)
                        acc[e] = h0 + e < G ? ptx::tmem_ld1(tmem + 64 + 17 * (h0 + e) + lane_base)
                                            : 0.f;
                } else {
                    float rv[16];
                    ptx::tmem_ld16(tmem + 2 * kN + lane_base, rv);
#pragma unroll
                    for (int e = 0; e < KH; ++e)
                        acc[e] = h0 + e < G ? head_col<KH>(rv, 0, hh, e) : 0.f;
                }
                ptx::tc_fence_before();
                // the q rows in the q_r buffer were read by the routing MMA; now overwrite them
                ptx::fence_proxy_async_smem();
            }
        } else if (a.q_routed) {
            if (a.pdl) grid_dep_wait();
#pragma unroll
            for (int e = 0; e < KH; ++e)
                acc[e] = h0 + e < G && t < D ? a.q_routed[((size_t)b * geo.Hq + qh0 + h0 + e) * D + t] : 0.f;
        } else {
            for (int i = tid; i < kD * kNG; i += kComputeThreads) {
                const int k = i >> 3, h = i & 7;
                const int kd = k - dim0(h);      // the head's own dims only
                qf[i] = h < G && kd >= 0 && kd < D
                            ? __uint_as_float((uint32_t)a.q[((size_t)b * geo.Hq + qh0 + h) * D + kd] << 16)
                            : 0.f;
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.q_ready);
            ok = wait(&sm.q_ready, 0);
            if (ok) {
#pragma unroll
                for (int e = 0; e < KH; ++e) acc[e] = qf[t * kNG + h0 + e];
            }
        }
        if (pair) {
            // two value heads: head h keeps the half of its routed query that its value head's
            // rows occupy (the other half holds the other diagonal block's product)
#pragma unroll
            for (int e = 0; e < KH; ++e)
                if ((t >> 6) != (dim0(h0 + e) >> 6)) acc[e] = 0.f;
        }
        if (ok) {
            // split-bf16 operand rows: n = h (hi), n = 8 + h (lo); column k = t. With KH = 2
            // the rows of heads 4-7 are zeros, written by the upper warps.
#pragma unroll
            for (int e = 0; e < KH; ++e) {
                const float v = acc[e] * sl2;
                const __nv_bfloat16 hi = __float2bfloat16_rn(v);
                const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
                *reinterpret_cast<__nv_bfloat16 *>(sm.qr + qr_offset(h0 + e, t)) = hi;
                *reinterpret_cast<__nv_bfloat16 *>(sm.qr + qr_offset(kNG + h0 + e, t)) = lo;
            }
            if (KH == 2 && hh) {
#pragma unroll
                for (int h = 4; h < kNG; ++h) {
                    *reinterpret_cast<uint16_t *>(sm.qr + qr_offset(h, t)) = 0;
                    *reinterpret_cast<uint16_t *>(sm.qr + qr_offset(kNG + h, t)) = 0;
                }
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.qr_full);
        }

        // every decision below is taken by the compute warps together
        ok = ptx::bar_and(kBarComputeAnd, kComputeThreads, ok);
        if (KH == 2 && hh) {
            // P^T columns of heads 4-7 (bytes 8-15 of a token's hi and lo rows) stay zero; the
            // raw query in the first P buffer has been read by now
#pragma unroll
            for (int pb = 0; pb < 2; ++pb) {
                uint8_t *row = sm.p[pb] + (t >> 3) * 256 + (t & 7) * 16;
                *reinterpret_cast<uint2 *>(row + 8) = make_uint2(0, 0);
                *reinterpret_cast<uint2 *>(row + 128 + 8) = make_uint2(0, 0);
            }
        }

        // Lazy reference: a tile's weights are 2^(s - m) with the head's current reference m,
        // which moves to the running maximum (rescaling the running sums) only when a weight
        // passes kLazyW (a score passes m + 2), so the weights stay at most 4 and most tiles need
        // one vote of the compute warps instead of an exchange of their maxima. When the state
        // leaves the kernel (exact_m), mx holds the thread's largest score of it, so that the
        // state carries its true largest score.
        const bool exact_m = !a.direct_out && !a.merge_inside;
        float m[KH], mx[KH], lsum[KH], o[KH];
        Vec<KH> alpha_prev;
#pragma unroll
        for (int e = 0; e < KH; ++e) {
            m[e] = -INFINITY;
            mx[e] = -INFINITY;
            lsum[e] = 0.f;
            o[e] = 0.f;
            alpha_prev.v[e] = 0.f;
        }
        // The CTA's largest score of each head of the current state into sm.mred (the caller's
        // next CTA barrier makes it visible).
        auto head_max = [&]() {
            float x[KH];
#pragma unroll
            for (int e = 0; e < KH; ++e) x[e] = mx[e];
            const float wm = warp_max_k<KH>(x, lane);
            if (max_writer<KH>(lane)) sm.mred[qd][h0 + max_head<KH>(lane)] = wm;
        };

        // O accumulation of tile j: o = o * alpha_j + O_j (thread = output dim t).
        auto correct = [&](int j, const Vec<KH> alpha) -> bool {
            const int ob = j & 1;
            if (!ptx::bar_and(kBarComputeAnd, kComputeThreads, wait(&sm.o_full[ob], (j >> 1) & 1)))
                return false;
            ptx::tc_fence_after();
            float ohi[KH], olo[KH];
            tmem_ld_heads<KH>(tmem + 2 * kN + ob * kN + lane_base, h0, ohi, olo);
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.o_empty[ob]);
#pragma unroll
            for (int e = 0; e < KH; ++e)
                o[e] = fmaf(o[e], alpha.v[e], ohi[e] + olo[e]);
            return true;
        };

        // Splits inside the CTA's run: tile i opens split split0 + i / tps. When the caller
        // gets the split states (or the combine kernel merges them), each split starts from a
        // fresh state (reference -inf, so the first alpha is 0 and its O starts over) and the
        // closed split's state is written once its last O is in. When this kernel merges the
        // splits itself, the run's splits are folded as they go: the online softmax simply
        // continues across the boundary (the merge of adjacent states is associative), and
        // the run leaves one state for the final merge.
        const int tps = geo.chunk / kTile;
        // The state of split sp from the running o, lsum and m (all of its O folded in).
        auto emit_state = [&](int sp) {
            float l[KH];
#pragma unroll
            for (int e = 0; e < KH; ++e) l[e] = lsum[e];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1)
#pragma unroll
                for (int e = 0; e < KH; ++e) l[e] += __shfl_xor_sync(0xffffffffu, l[e], off);
            if (lane == 0) {
#pragma unroll
                for (int e = 0; e < KH; ++e) sm.lred[qd][h0 + e] = l[e];
            }
            head_max();
            ptx::bar_sync(kBarCompute, kComputeThreads);
#pragma unroll
            for (int e = 0; e < KH; ++e) {
                const int h = h0 + e;
                if (h >= G) continue;
                const float lt = (sm.lred[0][h] + sm.lred[1][h]) + (sm.lred[2][h] + sm.lred[3][h]);
                const size_t slot = ((size_t)b * geo.Hq + qh0 + h) * geo.S + sp;
                const int dd = t - dim0(h);
                if (dd >= 0 && dd < D) a.part_o[slot * D + dd] = o[e] / lt;
                if (t == 0) {
                    // the state with its largest score M: l = sum 2^(s - M) = lt 2^(m - M)
                    const float M = fmaxf(fmaxf(sm.mred[0][h], sm.mred[1][h]),
                                          fmaxf(sm.mred[2][h], sm.mred[3][h]));
                    a.part_ml[slot * 2] = M * kLn2;
                    a.part_ml[slot * 2 + 1] = lt * exp2f(m[e] - M);
                }
            }
            ptx::bar_sync(kBarCompute, kComputeThreads);      // lred is free for the next split
        };

        for (int i = 0; ok && i < n_tiles; ++i) {
            const int sb = i & 1;
            if (!ptx::bar_and(kBarComputeAnd, kComputeThreads, wait(&sm.s_full[sb], (i >> 1) & 1))) {
                ok = false;
                break;
            }
            const bool opens = kPerSplit && i > 0 && i % tps == 0;   // tile i opens a split
            if (opens) {
                // close the previous split: its last O, its state, then a fresh state
                if (!correct(i - 1, alpha_prev)) {
                    ok = false;
                    break;
                }
                emit_state(split0 + i / tps - 1);
#pragma unroll
                for (int e = 0; e < KH; ++e) {
                    o[e] = 0.f;
                    lsum[e] = 0.f;
                    m[e] = -INFINITY;
                    mx[e] = -INFINITY;
                }
            }
            ptx::tc_fence_after();
            float shi[KH], slo[KH];
            tmem_ld_heads<KH>(tmem + sb * kN + lane_base, h0, shi, slo);
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.s_empty[sb]);

            // A padded head (h >= G) has a zero query row: its scores are 0, it follows the
            // same steps as a live head with finite values and is never written out.
            const int nvalid = min(kTile, t_end - (t_begin + i * kTile));
            float s[KH];
#pragma unroll
            for (int e = 0; e < KH; ++e) s[e] = shi[e] + slo[e];
            if (nvalid < kTile && t >= nvalid) {
#pragma unroll
                for (int e = 0; e < KH; ++e) s[e] = -INFINITY;      // tokens past the end
            }
            if (exact_m) {
#pragma unroll
                for (int e = 0; e < KH; ++e) mx[e] = fmaxf(mx[e], s[e]);
            }
            // the weights against the current references (0 past the end: s = -inf)
            float p[KH];
#pragma unroll
            for (int e = 0; e < KH; ++e) p[e] = ptx::ex2(s[e] - m[e]);
            float pmax = p[0];
#pragma unroll
            for (int e = 1; e < KH; ++e) pmax = fmaxf(pmax, p[e]);
            const bool grow = pmax > kLazyW;
            Vec<KH> alpha;
#pragma unroll
            for (int e = 0; e < KH; ++e) alpha.v[e] = 1.f;
            // (a state's first tile always sets the reference: no vote)
            const bool first = i == 0 || (kPerSplit && i % tps == 0);
            if (first || ptx::bar_popc(kBarComputeAnd, kComputeThreads, grow) != 0) {
                // a score passed its reference: the per-head maximum over the tile's 128 tokens
                // (warp reduce, then across the 4 lane quarters) becomes the reference
                float x[KH];
#pragma unroll
                for (int e = 0; e < KH; ++e) x[e] = s[e];
                const float wm = warp_max_k<KH>(x, lane);
                if (max_writer<KH>(lane)) sm.red[sb][qd][h0 + max_head<KH>(lane)] = wm;
                ptx::bar_sync(kBarCompute, kComputeThreads);
#pragma unroll
                for (int e = 0; e < KH; ++e) {
                    const int h = h0 + e;
                    float tmax = sm.red[sb][0][h];
#pragma unroll
                    for (int q = 1; q < 4; ++q) tmax = fmaxf(tmax, sm.red[sb][q][h]);
                    const float mn = fmaxf(m[e], tmax);
                    alpha.v[e] = ptx::ex2(m[e] - mn);             // 0 for the first tile
                    lsum[e] *= alpha.v[e];
                    m[e] = mn;
                    p[e] = ptx::ex2(s[e] - mn);
                }
            }
#pragma unroll
            for (int e = 0; e < KH; ++e) lsum[e] += p[e];
            // P^T row of token t, this warp's heads: hi and lo halves.
            {
                uint32_t ph[KH / 2], pl[KH / 2];
#pragma unroll
                for (int e = 0; e < KH / 2; ++e) split_bf16x2(p[2 * e], p[2 * e + 1], ph[e], pl[e]);
                uint8_t *row = sm.p[sb] + (t >> 3) * 256 + (t & 7) * 16 + 2 * h0;
                if constexpr (KH == 8) {
                    *reinterpret_cast<uint4 *>(row) = make_uint4(ph[0], ph[1], ph[2], ph[3]);
                    *reinterpret_cast<uint4 *>(row + 128) = make_uint4(pl[0], pl[1], pl[2], pl[3]);
                } else if constexpr (KH == 4) {
                    *reinterpret_cast<uint2 *>(row) = make_uint2(ph[0], ph[1]);
                    *reinterpret_cast<uint2 *>(row + 128) = make_uint2(pl[0], pl[1]);
                } else {
                    *reinterpret_cast<uint32_t *>(row) = ph[0];
                    *reinterpret_cast<uint32_t *>(row + 128) = pl[0];
                }
            }
            // Rows past the end inside the last 16-token MMA step must be finite: zero them
            // (with two warps per lane quarter, each clears one 64-dim half).
            if (nvalid < kTile) {
                const int st = (i + ro) % NS;
                if (ptx::bar_and(kBarComputeAnd, kComputeThreads,
                                 wait(&sm.full[st], ((i + ro) / NS) & 1)) &&
                    t >= nvalid && t < ((nvalid + 15) & ~15)) {
                    uint4 *r0 = reinterpret_cast<uint4 *>(sm.tiles[st][0] + (hh ? kHalfBytes : 0u) +
                                                          t * 128);
                    uint4 *r1 = reinterpret_cast<uint4 *>(sm.tiles[st][0] + kHalfBytes + t * 128);
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        r0[c] = make_uint4(0, 0, 0, 0);
                        if (KH == 8) r1[c] = make_uint4(0, 0, 0, 0);
                    }
                }
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&sm.p_full[sb]);

            if (i >= 1 && !opens && !correct(i - 1, alpha_prev)) { ok = false; break; }
            alpha_prev = alpha;
        }
        if (ok) ok = correct(n_tiles - 1, alpha_prev);

        if (ok) {
            // l totals over the 128 tokens-threads, then the output or the split state
#pragma unroll
            for (int off = 16; off > 0; off >>= 1)
#pragma unroll
                for (int e = 0; e < KH; ++e) lsum[e] += __shfl_xor_sync(0xffffffffu, lsum[e], off);
            const int rb = n_tiles & 1;   // red buffer not read by the last tile's exchange
            if (lane == 0) {
#pragma unroll
                for (int e = 0; e < KH; ++e) sm.red[rb][qd][h0 + e] = lsum[e];
            }
            // States that leave the kernel (for the caller or the combine kernel) carry their
            // true largest score; the merge inside the kernel takes any reference (l = sum
            // 2^(s - m) for the m it is given), so its states keep the lazy one.
            if (exact_m) head_max();
            ptx::bar_sync(kBarCompute, kComputeThreads);
            {
                // Merged here: one state per CTA run that holds tokens (slot cta; a single one
                // writes the output itself). Otherwise: the state of the split closed last.
                const int n_cta_u = (L + geo.chunk * geo.spc - 1) / (geo.chunk * geo.spc);
                const int sp_last = a.merge_inside ? cta : split0 + (n_tiles - 1) / tps;
                const bool write_out = a.direct_out || (a.merge_inside && n_cta_u == 1);
#pragma unroll
                for (int e = 0; e < KH; ++e) {
                    const int h = h0 + e;
                    if (h >= G) continue;
                    float lt = 0.f;
#pragma unroll
                    for (int q = 0; q < 4; ++q) lt += sm.red[rb][q][h];
                    const float val = o[e] / lt;
                    const size_t bh = (size_t)b * geo.Hq + qh0 + h;
                    const int dd = t - dim0(h);             // this thread's output dim of head h
                    const bool mine = dd >= 0 && dd < D;
                    if (write_out) {
                        if (!mine) continue;
                        if (a.out_dtype == KL_FP32) static_cast<float *>(a.out)[bh * D + dd] = val;
                        else static_cast<__nv_bfloat16 *>(a.out)[bh * D + dd] = __float2bfloat16_rn(val);
                    } else {
                        const size_t slot = bh * geo.S + sp_last;
                        if (mine) a.part_o[slot * D + dd] = val;
                        if (t == 0) {
                            // the state with its largest score M (l = lt 2^(m - M)), or with the
                            // lazy reference m for the merge inside the kernel
                            const float M = exact_m ? fmaxf(fmaxf(sm.mred[0][h], sm.mred[1][h]),
                                                            fmaxf(sm.mred[2][h], sm.mred[3][h]))
                                                    : m[e];
                            a.part_ml[slot * 2] = M * kLn2;
                            a.part_ml[slot * 2 + 1] = exact_m ? lt * exp2f(m[e] - M) : lt;
                        }
                        // splits of the run past the sequence's end: empty states
                        if (!a.merge_inside) {
                            for (int sp = sp_last + 1; sp < min(split0 + geo.spc, geo.S); ++sp) {
                                const size_t es = bh * geo.S + sp;
                                if (mine) a.part_o[es * D + dd] = 0.f;
                                if (t == 0) {
                                    a.part_ml[es * 2] = -INFINITY;
                                    a.part_ml[es * 2 + 1] = 0.f;
                                }
                            }
                        }
                    }
                }
                if (a.merge_inside && !write_out) {
                    // The last CTA of (b, g) to finish merges the n_cta_u states (as kl_combine).
                    ptx::bar_sync(kBarCompute, kComputeThreads);
                    if (tid == 0)
                        sm.is_last = arrive_last(
                            a.counters + ((size_t)b * geo.Hkv + g) * geo.nhb + hb, n_cta_u) ? 1 : 0;
                    ptx::bar_sync(kBarCompute, kComputeThreads);
                    if (sm.is_last) merge_states<KH, D>(sm, a, b, qh0, G, n_cta_u, tid, warp, lane, wait);
                }
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, tmem_cols);
    }
    // A CTA that gave up (every role has left its loop by now, so the flag is final): the cache
    // copies still in flight land before its shared memory goes away.
    if (warp == kProducerWarp && sm.abort) {
        for (int i = max(0, issued - NS); i < issued; ++i) {
            const uint64_t t0 = ptx::globaltimer();
            while (!ptx::mbar_try_wait(&sm.full[i % NS], (i / NS) & 1) &&
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

// 2-D bf16 tensor map over `rows` rows of `dim` (128 or 64) dims, box = 64 dims x box_rows
// (one 128-byte swizzle span), 128-byte swizzle.
bool make_map(CUtensorMap *map, const void *base, int dim, uint64_t rows, uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)dim, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)dim * 2};
    const cuuint32_t box[2] = {64, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <bool kStandard, bool kPerSplit, int KH, bool kExact, bool kD64>
cudaError_t launch_kernel(const DecodeArgs &la, const CUtensorMap &vmap, const CUtensorMap &kmap,
                          const CUtensorMap &wmap, const CUtensorMap &qmap) {
    const Geometry &g = la.geo;
    const size_t smem = sizeof(Smem<kStandard>) + 1024;
    static PerDeviceOnce once;
    const cudaError_t e = once.run([&] {
        return cudaFuncSetAttribute(decode_tc_kernel<kStandard, kPerSplit, KH, kExact, kD64>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((g.S + g.spc - 1) / g.spc * g.nhb, g.Hkv / g.vpc, g.B);
    cfg.blockDim = dim3(Roles<KH>::kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = la.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    if (la.pdl) {
        cfg.attrs = attr;
        cfg.numAttrs = 1;
    }
    return cudaLaunchKernelEx(&cfg, decode_tc_kernel<kStandard, kPerSplit, KH, kExact, kD64>, vmap, kmap,
                              wmap, qmap, la);
}

// The launches of one head dim (kD64) and wait mode: the per-split and merged variants.
template <bool kStandard, int KH, bool kExact, bool kD64>
cudaError_t launch_dim(const DecodeArgs &la, bool per_split, const CUtensorMap &vmap,
                       const CUtensorMap &kmap, const CUtensorMap &wmap, const CUtensorMap &qmap) {
    return per_split ? launch_kernel<kStandard, true, KH, kExact, kD64>(la, vmap, kmap, wmap, qmap)
                     : launch_kernel<kStandard, false, KH, kExact, kD64>(la, vmap, kmap, wmap, qmap);
}

}  // namespace

// The head-dim-64 launches (kl_decode_tc64.cu): K+V comparison or keyless, KH heads per compute
// warp (2 or 8), exact short waits or not.
cudaError_t launch_tc_head64(const DecodeArgs &la, bool per_split, bool standard, int KH, bool exact,
                             const CUtensorMap &vmap, const CUtensorMap &kmap,
                             const CUtensorMap &wmap, const CUtensorMap &qmap);
// The head-dim-128 launches of groups of more than 8 heads (kl_decode_tc_groups.cu): K+V
// comparison or keyless, 4 heads per compute warp, exact short waits or not.
cudaError_t launch_tc_groups(const DecodeArgs &la, bool per_split, bool standard, bool exact,
                             const CUtensorMap &vmap, const CUtensorMap &kmap,
                             const CUtensorMap &wmap, const CUtensorMap &qmap);

}  // namespace kl
