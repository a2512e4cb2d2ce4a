// CUDA-core split-sequence decode: the general path (head_dim 64 or 128, group size <= 8)
// and the cross-check of the tensor-core kernel.
//
// Grid (S, Hkv, B): one CTA per (split, value head, sequence), 4 warps. The CTA first forms
// the routed query of every head of its group (Section 2.2: q_r = q W^R, fp32), then its
// warps take the split's tokens round-robin. A warp reads one cached value row per step
// (32 lanes x D/32 bf16, one coalesced row) and uses it twice, as the Value-Only Cache
// decode prescribes (Section 3): for the G scores <q_r, v_t> (warp-shuffle sums) and for the
// G output accumulators, with an online softmax in base 2 (scores pre-multiplied by
// scale * log2 e). The four warp states are merged in shared memory and the CTA writes either
// the final output (S == 1) or its split state (normalized o, natural-log m, l).
#include <math.h>

#include "kl_internal.cuh"

namespace kl {
namespace {

constexpr int kWarps = 4;
constexpr int kMaxGroup = 8;

template <int E>
__device__ __forceinline__ void load_row(const uint16_t *p, float (&x)[E]) {
    if constexpr (E == 4) {
        const uint2 w = *reinterpret_cast<const uint2 *>(p);
        x[0] = bf16lo(w.x); x[1] = bf16hi(w.x); x[2] = bf16lo(w.y); x[3] = bf16hi(w.y);
    } else {
        const uint32_t w = *reinterpret_cast<const uint32_t *>(p);
        x[0] = bf16lo(w); x[1] = bf16hi(w);
    }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <int D, bool kStandard>
__global__ void __launch_bounds__(kWarps * 32) decode_simt_kernel(DecodeArgs a) {
    constexpr int E = D / 32;
    __shared__ float q_in[kMaxGroup][D];
    __shared__ float qs[kMaxGroup][D];
    __shared__ float sm_m[kWarps][kMaxGroup], sm_l[kWarps][kMaxGroup];
    __shared__ float sm_acc[kWarps][kMaxGroup][D];

    const Geometry &geo = a.geo;
    const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = geo.G;

    int L = a.seq_lens[b];
    if (L < 0 || L > geo.max_pages * geo.P) {
        if (tid == 0 && split == 0 && g == 0) raise_flag(a.err, KL_FLAG_BAD_LENGTH);
        L = 0;
    }
    const int t0 = split * geo.chunk;
    const int t1 = min(t0 + geo.chunk, L);

    // Fused append (kl_decode_step): the CTA whose split holds row positions[b] writes the
    // current token's value row there before any row is read.
    if (a.v_new) {
        const int pos = a.positions[b];
        if (pos < 0 || pos >= geo.max_pages * geo.P) {
            if (tid == 0 && split == 0 && g == 0) raise_flag(a.err, KL_FLAG_BAD_POSITION);
        } else if (pos / geo.chunk == split) {
            const int page = a.block_table[(size_t)b * geo.max_pages + pos / geo.P];
            if (page >= 0 && page < geo.num_pages) {
                if (tid < D / 8)
                    reinterpret_cast<uint4 *>(a.cache_rw + (((size_t)page * geo.Hkv + g) * geo.P +
                                                            pos % geo.P) * D)[tid] =
                        reinterpret_cast<const uint4 *>(a.v_new + ((size_t)b * geo.Hkv + g) * D)[tid];
            } else if (tid == 0) {
                raise_flag(a.err, KL_FLAG_BAD_PAGE);
            }
        }
        __syncthreads();
    }

    // Routed, pre-scaled query of every head of the group.
    for (int i = tid; i < G * D; i += kWarps * 32) {
        const int h = i / D, k = i % D;
        q_in[h][k] = __uint_as_float((uint32_t)a.q[((size_t)b * geo.Hq + g * G + h) * D + k] << 16);
    }
    __syncthreads();
    const float sl2 = geo.scale * kLog2e;
    if (t1 > t0) {
        for (int i = tid; i < G * D; i += kWarps * 32) {
            const int h = i / D, j = i % D;
            float acc;
            if (kStandard || a.w_r == nullptr) {
                acc = q_in[h][j];      // unrouted (K+V) or already composed (q = x W^Q W^R)
            } else {
                const uint16_t *W = a.w_r + (size_t)(geo.wr_per_qh ? g * G + h : g) * D * D;
                acc = 0.f;
#pragma unroll 8
                for (int k = 0; k < D; ++k)
                    acc = fmaf(q_in[h][k], __uint_as_float((uint32_t)W[(size_t)k * D + j] << 16), acc);
            }
            qs[h][j] = acc * sl2;
        }
    }
    __syncthreads();

    float qreg[kMaxGroup][E];
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h)
#pragma unroll
        for (int i = 0; i < E; ++i) qreg[h][i] = (h < G) ? qs[h][lane * E + i] : 0.f;

    float m[kMaxGroup], l[kMaxGroup], acc[kMaxGroup][E];
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int i = 0; i < E; ++i) acc[h][i] = 0.f;
    }

    const int32_t *bt = a.block_table + (size_t)b * geo.max_pages;
    const uint16_t *score_cache = kStandard ? a.k_cache : a.v_cache;
    bool bad_page = false;
    for (int t = t0 + warp; t < t1; t += kWarps) {
        const int page = bt[t / geo.P];
        if (page < 0 || page >= geo.num_pages) {
            bad_page = true;
            continue;
        }
        const size_t off = (((size_t)page * geo.Hkv + g) * geo.P + t % geo.P) * D + lane * E;
        float v[E], k[E];
        load_row<E>(a.v_cache + off, v);
        if constexpr (kStandard) load_row<E>(score_cache + off, k);
#pragma unroll
        for (int h = 0; h < kMaxGroup; ++h) {
            if (h < G) {
                float part = 0.f;
#pragma unroll
                for (int i = 0; i < E; ++i) part = fmaf(qreg[h][i], kStandard ? k[i] : v[i], part);
                const float s = warp_sum(part);
                const float mn = fmaxf(m[h], s);
                const float alpha = exp2f(m[h] - mn);
                const float p = exp2f(s - mn);
                l[h] = fmaf(l[h], alpha, p);
#pragma unroll
                for (int i = 0; i < E; ++i) acc[h][i] = fmaf(acc[h][i], alpha, p * v[i]);
                m[h] = mn;
            }
        }
    }
    if (bad_page && lane == 0) raise_flag(a.err, KL_FLAG_BAD_PAGE);

    if (lane == 0) {
#pragma unroll
        for (int h = 0; h < kMaxGroup; ++h) {
            sm_m[warp][h] = m[h];
            sm_l[warp][h] = l[h];
        }
    }
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h)
        if (h < G)
#pragma unroll
            for (int i = 0; i < E; ++i) sm_acc[warp][h][lane * E + i] = acc[h][i];
    __syncthreads();

    for (int i = tid; i < G * D; i += kWarps * 32) {
        const int h = i / D, j = i % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sm_m[w][h]);
        float z = 0.f, o = 0.f;
        if (M != -INFINITY) {
#pragma unroll
            for (int w = 0; w < kWarps; ++w) {
                const float f = exp2f(sm_m[w][h] - M);
                z = fmaf(sm_l[w][h], f, z);
                o = fmaf(sm_acc[w][h][j], f, o);
            }
            o = o / z;
        }
        const size_t bh = (size_t)b * geo.Hq + g * G + h;
        if (a.direct_out) {
            if (a.out_dtype == KL_FP32)
                static_cast<float *>(a.out)[bh * D + j] = o;
            else
                static_cast<__nv_bfloat16 *>(a.out)[bh * D + j] = __float2bfloat16_rn(o);
        } else {
            const size_t slot = bh * geo.S + split;
            a.part_o[slot * D + j] = o;
            if (j == 0) {
                a.part_ml[slot * 2] = (M == -INFINITY) ? -INFINITY : M * kLn2;
                a.part_ml[slot * 2 + 1] = z;
            }
        }
    }
}

}  // namespace

cudaError_t launch_decode_simt(const DecodeArgs &a, bool standard) {
    const Geometry &g = a.geo;
    if (g.B == 0) return cudaSuccess;
    const dim3 grid(g.S, g.Hkv, g.B), block(kWarps * 32);
    if (g.D == 128) {
        if (standard) decode_simt_kernel<128, true><<<grid, block, 0, a.stream>>>(a);
        else decode_simt_kernel<128, false><<<grid, block, 0, a.stream>>>(a);
    } else {
        if (standard) decode_simt_kernel<64, true><<<grid, block, 0, a.stream>>>(a);
        else decode_simt_kernel<64, false><<<grid, block, 0, a.stream>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace kl
