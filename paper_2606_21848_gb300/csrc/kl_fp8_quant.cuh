// OCP FP8 E4M3 quantization of one cached value row, shared by every writer of the FP8 cache (the
// quantizing append, the cache quantizer and the decode step's fused append), so that all of them
// produce the same codes and scales.
#pragma once

#include <cuda_fp8.h>

#include "kl_internal.cuh"

namespace kl {

// One 128-value row held by a warp, lane j holding values 4j .. 4j + 3 (bf16 pairs in w):
// scale = max |v| / 448 in fp32, code = E4M3(v / scale) rounded to nearest even and saturating
// (the conversion intrinsic of cuda_fp8.h); an all-zero row gets scale 0 and zero codes. Returns
// the lane's four codes packed (value 4j in the low byte) and the row's scale in every lane.
__device__ __forceinline__ uint32_t quantize_row4(const uint2 w, float &scale) {
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
    scale = s;
    return packed;
}

}  // namespace kl
