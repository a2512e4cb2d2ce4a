// Latent value-only cache (Section 3, "Multihead with Latent Value-only Cache"): the absorbed
// query and the output expansion around the decode over the latent rows.
//
//   q*_h  = (q_h W^R[w(h)]) W^V_{h,post}^T      query width D -> latent width r
//   o*_h  = softmax(scale q*_h V*^T) V*          the tensor-core decode, pre-routed mode
//   out_h = o*_h W^V_{h,post}                    latent width r -> head width D
//
// Both projections are small per (sequence, head) and share their matrices across the batch,
// so one CTA per (head, block of sequences) stages the matrices in shared memory once (bf16,
// 16-byte copies) and runs the products for every sequence of the block, four sequences per
// pass so that each thread keeps four independent accumulation chains; fp32 accumulation.
#include "kl_internal.cuh"

namespace kl {
namespace {

constexpr int kSeqBlock = 8;       // sequences per CTA
constexpr int kSeqPass = 4;        // sequences per pass (independent chains per thread)
constexpr int kMaxDim = 128;       // D and r are at most 128

__device__ __forceinline__ float bf(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }

// Copy `rows` rows of `cols` bf16 values (cols a multiple of 8, 16-byte aligned) into shared
// memory with a row stride of `stride` values, 16 bytes per copy. The loads go out in batches of
// eight before their stores, so a cold matrix costs a few memory round trips, not one per copy.
__device__ __forceinline__ void stage_rows(uint16_t *dst, const uint16_t *src, int rows, int cols,
                                           int stride) {
    constexpr int kBatch = 8;
    const int vpr = cols / 8, n = rows * vpr;
    const uint4 *s4 = reinterpret_cast<const uint4 *>(src);
    for (int v0 = threadIdx.x; v0 < n; v0 += kBatch * blockDim.x) {
        uint4 w[kBatch];
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int v = v0 + i * blockDim.x;
            if (v < n) w[i] = __ldg(s4 + v);
        }
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int v = v0 + i * blockDim.x;
            if (v < n) *reinterpret_cast<uint4 *>(dst + (v / vpr) * stride + (v % vpr) * 8) = w[i];
        }
    }
}

// One CTA per (query head h, block of sequences), kMaxDim threads. Shared (bf16): W^R[w(h)] as
// [k][j] (thread j of the first product reads column j: consecutive threads, consecutive
// halves) and W_post[h] as [k][j] with rows padded by 16 bytes (thread k of the second product
// reads its own row 16 bytes at a time; the padding spreads eight such rows over all banks).
__global__ void __launch_bounds__(kMaxDim)
    latent_query_kernel(int B, int Hq, int G, int D, int r, int wr_per_qh,
                        const uint16_t *__restrict__ q, const uint16_t *__restrict__ w_r,
                        const uint16_t *__restrict__ w_post, float *__restrict__ q_lat) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int ps = D + 8;                   // padded row stride of W_post (values)
    uint16_t *wr = reinterpret_cast<uint16_t *>(smem_raw);             // [D][D]
    uint16_t *wp = wr + D * D;                                         // [r][ps]
    // per-sequence vectors as [dim][sequence]: one 16-byte load feeds four FMAs
    float4 *qv = reinterpret_cast<float4 *>(wp + r * ps);              // [D] x 4 sequences
    float4 *qr = qv + D;                                               // [D] x 4 sequences
    const int h = blockIdx.x, b0 = blockIdx.y * kSeqBlock, t = threadIdx.x;
    stage_rows(wr, w_r + (size_t)(wr_per_qh ? h : h / G) * D * D, D, D, D);
    stage_rows(wp, w_post + (size_t)h * r * D, r, D, ps);
    __syncthreads();
    const int b_end = min(B, b0 + kSeqBlock);
    for (int b = b0; b < b_end; b += kSeqPass) {
        const int nb = min(kSeqPass, b_end - b);
        if (t < D) {
            float v[kSeqPass];
#pragma unroll
            for (int s = 0; s < kSeqPass; ++s)
                v[s] = s < nb ? bf(q[((size_t)(b + s) * Hq + h) * D + t]) : 0.f;
            qv[t] = make_float4(v[0], v[1], v[2], v[3]);
        }
        __syncthreads();
        if (t < D) {
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
            for (int k = 0; k < D; ++k) {
                const float w = bf(wr[k * D + t]);
                const float4 x = qv[k];
                acc.x = fmaf(x.x, w, acc.x);
                acc.y = fmaf(x.y, w, acc.y);
                acc.z = fmaf(x.z, w, acc.z);
                acc.w = fmaf(x.w, w, acc.w);
            }
            qr[t] = acc;
        }
        __syncthreads();
        if (t < r) {
            float acc[kSeqPass] = {0.f, 0.f, 0.f, 0.f};
            const uint4 *row = reinterpret_cast<const uint4 *>(wp + t * ps);
            for (int c = 0; c < D / 8; ++c) {
                const uint4 w4 = row[c];
                const uint32_t u[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int j = 8 * c + 2 * e;
                    const float w0 = bf16lo(u[e]), w1 = bf16hi(u[e]);
                    const float4 x0 = qr[j], x1 = qr[j + 1];
                    acc[0] = fmaf(x1.x, w1, fmaf(x0.x, w0, acc[0]));
                    acc[1] = fmaf(x1.y, w1, fmaf(x0.y, w0, acc[1]));
                    acc[2] = fmaf(x1.z, w1, fmaf(x0.z, w0, acc[2]));
                    acc[3] = fmaf(x1.w, w1, fmaf(x0.w, w0, acc[3]));
                }
            }
#pragma unroll
            for (int s = 0; s < kSeqPass; ++s)
                if (s < nb) q_lat[((size_t)(b + s) * Hq + h) * r + t] = acc[s];
        }
        __syncthreads();
    }
}

// One CTA per (query head h, block of sequences), kMaxDim threads; W_post[h] [k][j] in shared
// memory (bf16); thread j: out[j] = sum_k o*[k] W_post[h][k][j].
__global__ void __launch_bounds__(kMaxDim)
    latent_expand_kernel(int B, int Hq, int D, int r, const float *__restrict__ o_lat,
                         const uint16_t *__restrict__ w_post, void *out, int out_fp32) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    uint16_t *wp = reinterpret_cast<uint16_t *>(smem_raw);             // [r][D]
    float4 *ov = reinterpret_cast<float4 *>(wp + r * D);               // [r] x 4 sequences
    const int h = blockIdx.x, b0 = blockIdx.y * kSeqBlock, t = threadIdx.x;
    stage_rows(wp, w_post + (size_t)h * r * D, r, D, D);
    __syncthreads();
    const int b_end = min(B, b0 + kSeqBlock);
    for (int b = b0; b < b_end; b += kSeqPass) {
        const int nb = min(kSeqPass, b_end - b);
        if (t < r) {
            float v[kSeqPass];
#pragma unroll
            for (int s = 0; s < kSeqPass; ++s)
                v[s] = s < nb ? o_lat[((size_t)(b + s) * Hq + h) * r + t] : 0.f;
            ov[t] = make_float4(v[0], v[1], v[2], v[3]);
        }
        __syncthreads();
        if (t < D) {
            float acc[kSeqPass] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
            for (int k = 0; k < r; ++k) {
                const float w = bf(wp[k * D + t]);
                const float4 x = ov[k];
                acc[0] = fmaf(x.x, w, acc[0]);
                acc[1] = fmaf(x.y, w, acc[1]);
                acc[2] = fmaf(x.z, w, acc[2]);
                acc[3] = fmaf(x.w, w, acc[3]);
            }
#pragma unroll
            for (int s = 0; s < kSeqPass; ++s) {
                if (s >= nb) continue;
                const size_t oi = ((size_t)(b + s) * Hq + h) * D + t;
                if (out_fp32)
                    static_cast<float *>(out)[oi] = acc[s];
                else
                    static_cast<__nv_bfloat16 *>(out)[oi] = __float2bfloat16_rn(acc[s]);
            }
        }
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_latent_query(int B, int Hq, int G, int D, int r, int wr_per_qh,
                                const uint16_t *q, const uint16_t *w_r, const uint16_t *w_post,
                                float *q_lat, cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    if (D > kMaxDim || r > kMaxDim || D % 8 || r % 8) return cudaErrorInvalidValue;
    const size_t smem = (size_t)(D * D + r * (D + 8)) * 2 + 2 * D * sizeof(float4);
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(
            latent_query_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
            (int)((kMaxDim * kMaxDim + kMaxDim * (kMaxDim + 8)) * 2 +
                  2 * kSeqPass * kMaxDim * sizeof(float)));
        if (e != cudaSuccess) return e;
        configured = true;
    }
    const dim3 grid(Hq, (B + kSeqBlock - 1) / kSeqBlock);
    latent_query_kernel<<<grid, kMaxDim, smem, stream>>>(B, Hq, G, D, r, wr_per_qh, q, w_r, w_post,
                                                          q_lat);
    return cudaGetLastError();
}

cudaError_t launch_latent_expand(int B, int Hq, int D, int r, const float *o_lat,
                                 const uint16_t *w_post, void *out, kl_dtype out_dtype,
                                 cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    if (D > kMaxDim || r > kMaxDim || D % 8 || r % 8) return cudaErrorInvalidValue;
    const size_t smem = (size_t)r * D * 2 + r * sizeof(float4);
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(
            latent_expand_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
            (int)(kMaxDim * kMaxDim * 2 + kSeqPass * kMaxDim * sizeof(float)));
        if (e != cudaSuccess) return e;
        configured = true;
    }
    const dim3 grid(Hq, (B + kSeqBlock - 1) / kSeqBlock);
    latent_expand_kernel<<<grid, kMaxDim, smem, stream>>>(B, Hq, D, r, o_lat, w_post, out,
                                                           out_dtype == KL_FP32);
    return cudaGetLastError();
}

}  // namespace kl
