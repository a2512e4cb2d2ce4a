// Value-cache append, standalone routing projection and the split-state combine.
#include <math.h>

#include "kl_internal.cuh"

namespace kl {
namespace {

// Append (Section 3): one CTA per sequence copies the Hkv value rows of the current token
// into row pos % P of page block_table[b][pos / P]. 16-byte copies; D is a multiple of 8.
__global__ void __launch_bounds__(128) append_kernel(int Hkv, int D, int P, int num_pages,
                                                     int max_pages, const uint4 *__restrict__ v_new,
                                                     const int32_t *__restrict__ block_table,
                                                     const int32_t *__restrict__ positions,
                                                     uint4 *__restrict__ v_cache, int32_t *err) {
    const int b = blockIdx.x;
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
    const int slot = pos % P;
    const int cpr = D / 8;  // 16-byte chunks per row
    for (int i = threadIdx.x; i < Hkv * cpr; i += blockDim.x) {
        const int g = i / cpr, c = i % cpr;
        v_cache[(((size_t)page * Hkv + g) * P + slot) * cpr + c] =
            v_new[((size_t)b * Hkv + g) * cpr + c];
    }
}

// Routing projection (Section 2.2): one CTA per (h, b), thread j computes
// q_r[j] = sum_k q[k] W^R[k][j]; the W^R reads of a k step are one coalesced row.
__global__ void route_kernel(int Hq, int G, int D, int wr_per_qh, const uint16_t *__restrict__ q,
                             const uint16_t *__restrict__ w_r, float *__restrict__ q_r) {
    __shared__ float qs[128];
    const int h = blockIdx.x, b = blockIdx.y, j = threadIdx.x;
    const size_t row = ((size_t)b * Hq + h) * D;
    qs[j] = __uint_as_float((uint32_t)q[row + j] << 16);
    __syncthreads();
    const uint16_t *W = w_r + (size_t)(wr_per_qh ? h : h / G) * D * D;
    float acc = 0.f;
#pragma unroll 8
    for (int k = 0; k < D; ++k)
        acc = fmaf(qs[k], __uint_as_float((uint32_t)W[(size_t)k * D + j] << 16), acc);
    q_r[row + j] = acc;
}

// Combine: one CTA per (h, b); thread j merges column j of the S split states.
__global__ void combine_kernel(int Hq, int D, int S, const float *__restrict__ part_o,
                               const float2 *__restrict__ part_ml, void *out, int out_fp32) {
    __shared__ float red[4];
    const int h = blockIdx.x, b = blockIdx.y, j = threadIdx.x;
    const size_t bh = (size_t)b * Hq + h;
    const float2 *ml = part_ml + bh * S;

    float M = -INFINITY;
    for (int s = j; s < S; s += blockDim.x) {
        const float2 v = ml[s];
        if (v.y > 0.f) M = fmaxf(M, v.x);
    }
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    if ((j & 31) == 0) red[j >> 5] = M;
    __syncthreads();
    M = red[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) M = fmaxf(M, red[w]);

    float res = 0.f;
    if (M != -INFINITY) {
        float z = 0.f, acc = 0.f;
        const float *po = part_o + bh * S * D + j;
        for (int s = 0; s < S; ++s) {
            const float2 v = ml[s];
            if (v.y > 0.f) {
                const float w = v.y * expf(v.x - M);
                z += w;
                acc = fmaf(w, po[(size_t)s * D], acc);
            }
        }
        res = acc / z;
    }
    const size_t oi = bh * D + j;
    if (out_fp32)
        static_cast<float *>(out)[oi] = res;
    else
        static_cast<__nv_bfloat16 *>(out)[oi] = __float2bfloat16_rn(res);
}

}  // namespace

cudaError_t launch_append(const Geometry &g, const uint16_t *v_new, const int32_t *block_table,
                          const int32_t *positions, uint16_t *v_cache, int32_t *err,
                          cudaStream_t stream) {
    if (g.B == 0) return cudaSuccess;
    append_kernel<<<g.B, 128, 0, stream>>>(g.Hkv, g.D, g.P, g.num_pages, g.max_pages,
                                           reinterpret_cast<const uint4 *>(v_new), block_table,
                                           positions, reinterpret_cast<uint4 *>(v_cache), err);
    return cudaGetLastError();
}

cudaError_t launch_route(const Geometry &g, const uint16_t *q, const uint16_t *w_r, float *q_r,
                         cudaStream_t stream) {
    if (g.B == 0) return cudaSuccess;
    route_kernel<<<dim3(g.Hq, g.B), g.D, 0, stream>>>(g.Hq, g.G, g.D, g.wr_per_qh, q, w_r, q_r);
    return cudaGetLastError();
}

cudaError_t launch_combine(int B, int Hq, int D, int S, const float *part_o,
                           const float *part_ml, void *out, kl_dtype out_dtype,
                           cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    combine_kernel<<<dim3(Hq, B), D, 0, stream>>>(Hq, D, S, part_o,
                                                 reinterpret_cast<const float2 *>(part_ml), out,
                                                 out_dtype == KL_FP32);
    return cudaGetLastError();
}

}  // namespace kl
