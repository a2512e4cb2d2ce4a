// FP8 value cache, the writing side: the quantizing append of one row per (sequence, value
// head) and the conversion of a whole bf16 cache. A row of 128 values becomes 128 OCP E4M3 codes
// and one fp32 scale: scale = max |v| / 448 in fp32, code = E4M3(v / scale), rounded to nearest
// even and saturating (the conversion intrinsic of cuda_fp8.h; an all-zero row gets scale 0).
#include "kl_fp8_quant.cuh"

namespace kl {
namespace {

constexpr int kD = 128;

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
        float s;
        const uint32_t packed = quantize_row4(w, s);
        const size_t row = ((size_t)page * Hkv + g) * P + pos % P;
        reinterpret_cast<uint32_t *>(codes + row * kD)[lane] = packed;
        if (lane == 0) scales[row] = s;
    }
}

// Quantize a whole bf16 cache [rows][128] into codes [rows][128] and row scales [rows], with the
// arithmetic of the append: one warp per row, 4 values per lane; each warp loads 4 rows before
// reducing any of them, so that enough loads are in flight to keep HBM busy.
__device__ __forceinline__ void quantize_row_regs(const uint2 w, int lane, uint8_t *__restrict__ codes,
                                                  float *__restrict__ scales, size_t row) {
    float s;
    const uint32_t packed = quantize_row4(w, s);
    reinterpret_cast<uint32_t *>(codes + row * kD)[lane] = packed;
    if (lane == 0) scales[row] = s;
}

__global__ void __launch_bounds__(256)
    quantize_rows_kernel(size_t rows, const uint16_t *__restrict__ v, uint8_t *__restrict__ codes,
                         float *__restrict__ scales) {
    constexpr int kRowsPerWarp = 4;
    const int lane = threadIdx.x & 31;
    const size_t warps = (size_t)gridDim.x * (blockDim.x >> 5);
    const size_t w0 = (size_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    for (size_t r0 = w0 * kRowsPerWarp; r0 < rows; r0 += warps * kRowsPerWarp) {
        uint2 w[kRowsPerWarp];
#pragma unroll
        for (int i = 0; i < kRowsPerWarp; ++i)
            if (r0 + i < rows) w[i] = __ldcs(reinterpret_cast<const uint2 *>(v + (r0 + i) * kD) + lane);
#pragma unroll
        for (int i = 0; i < kRowsPerWarp; ++i)
            if (r0 + i < rows) quantize_row_regs(w[i], lane, codes, scales, r0 + i);
    }
}

}  // namespace

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
    const size_t blocks = (rows + 31) / 32;                 // 8 warps of 4 rows each
    const unsigned grid = (unsigned)(blocks < 65535 * 16 ? blocks : 65535 * 16);
    quantize_rows_kernel<<<grid, 256, 0, stream>>>(rows, v, codes, scales);
    return cudaGetLastError();
}

}  // namespace kl
