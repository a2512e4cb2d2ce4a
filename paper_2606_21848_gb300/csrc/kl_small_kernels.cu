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

// Combine: one CTA of 4 warps per (h, b). The split weights w_s = l_s exp(m_s - M) are formed
// once in shared memory; then warp w folds the states s = w, w + 4, ... (each lane 4 dims of
// one state row, float4 loads), and the four warp sums are added and normalized.
constexpr int kCombineWarps = 4;
constexpr int kCombineMaxSplits = 1024;

__global__ void __launch_bounds__(kCombineWarps * 32)
    combine_kernel(int Hq, int D, int S, const float *__restrict__ part_o,
                   const float2 *__restrict__ part_ml, void *out, int out_fp32) {
    __shared__ float w_s[kCombineMaxSplits];
    __shared__ float red[kCombineWarps];
    __shared__ float4 acc_s[kCombineWarps][32];
    const int h = blockIdx.x, b = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const size_t bh = (size_t)b * Hq + h;
    const float2 *ml = part_ml + bh * S;
    // behind a decode as its programmatic dependent: the decode's states are complete and
    // visible past this point (an ordinary launch returns at once)
    grid_dep_wait();

    float M = -INFINITY;
    for (int s = tid; s < S; s += blockDim.x) {
        const float2 v = ml[s];
        if (v.y > 0.f) M = fmaxf(M, v.x);
    }
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    if (lane == 0) red[warp] = M;
    __syncthreads();
    M = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
    __syncthreads();

    float z = 0.f;
    for (int s = tid; s < S; s += blockDim.x) {
        const float2 v = ml[s];
        const float w = (v.y > 0.f && M != -INFINITY) ? v.y * expf(v.x - M) : 0.f;
        w_s[s] = w;
        z += w;
    }
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if (lane == 0) red[warp] = z;
    __syncthreads();
    z = red[0] + red[1] + red[2] + red[3];

    // D / 4 lanes hold 4 dims each (D = 128: all 32 lanes; D = 64: 16 lanes)
    const int nl = D / 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (lane < nl) {
        const float4 *po = reinterpret_cast<const float4 *>(part_o + bh * S * D) + lane;
#pragma unroll 4
        for (int s = warp; s < S; s += kCombineWarps) {
            const float w = w_s[s];
            if (w != 0.f) {
                const float4 v = po[(size_t)s * nl];
                acc.x = fmaf(w, v.x, acc.x);
                acc.y = fmaf(w, v.y, acc.y);
                acc.z = fmaf(w, v.z, acc.z);
                acc.w = fmaf(w, v.w, acc.w);
            }
        }
    }
    acc_s[warp][lane] = acc;
    __syncthreads();
    if (tid < D) {
        const int l = tid >> 2, c = tid & 3;
        float r = 0.f;
#pragma unroll
        for (int w = 0; w < kCombineWarps; ++w) r += reinterpret_cast<const float *>(&acc_s[w][l])[c];
        r = z > 0.f ? r / z : 0.f;
        const size_t oi = bh * D + tid;
        if (out_fp32)
            static_cast<float *>(out)[oi] = r;
        else
            static_cast<__nv_bfloat16 *>(out)[oi] = __float2bfloat16_rn(r);
    }
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
                           cudaStream_t stream, bool dependent) {
    if (B == 0) return cudaSuccess;
    if (S > kCombineMaxSplits) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(Hq, B);
    cfg.blockDim = dim3(kCombineWarps * 32);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    if (dependent) {
        cfg.attrs = attr;
        cfg.numAttrs = 1;
    }
    return cudaLaunchKernelEx(&cfg, combine_kernel, Hq, D, S, part_o,
                              reinterpret_cast<const float2 *>(part_ml), out,
                              (int)(out_dtype == KL_FP32));
}

}  // namespace kl
