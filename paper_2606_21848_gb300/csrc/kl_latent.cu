// Latent value-only cache (Section 3, "Multihead with Latent Value-only Cache"): the absorbed
// query and the output expansion around the decode over the latent rows.
//
//   q*_h  = (q_h W^R[w(h)]) W^V_{h,post}^T      query width D -> latent width r
//   o*_h  = softmax(scale q*_h V*^T) V*          the tensor-core decode, pre-routed mode
//   out_h = o*_h W^V_{h,post}                    latent width r -> head width D
//
// Both projections are, per query head h, a product of a block of up to 128 sequences with
// matrices the whole batch shares, so each runs on the tensor cores: one CTA per (head, block
// of 128 sequences), the sequences as the MMA rows (M = 128; rows past the batch read as zeros
// and are never stored), the shared matrices staged once by TMA (128-byte swizzle), the
// accumulators in TMEM, and the results leaving through TMA stores.
//
//   query      Q_r = Q . W^R[w(h)]                  M = 128, N = D,   K = D      (bf16 x bf16)
//              Q*  = Q_r . W_post[h]^T              M = 128, N = r,   K = 2 x D  (hi + lo)
//   expansion  O   = O* . W_post[h]                 M = 128, N = D,   K = 2 x r  (hi + lo)
//
// The fp32 intermediates (Q_r, and the decode's fp32 output O*) enter the second products as a
// pair of bf16 operands x = hi + lo, hi = bf16(x), lo = bf16(x - hi), which keeps about 16
// significant bits; the pairs go from registers into TMEM and feed the MMAs as A operands from
// there. Products and sums are fp32 on the tensor cores.
//
// Each row of a result is one TMEM lane, read by the thread of that lane and written to shared
// memory in the 128-byte-swizzled box layout that a TMA store reads (16-byte chunk j of row t at
// chunk j ^ (t % 8)), so that neither the writes nor the stores conflict; the expansion reads
// the O* rows from TMA boxes of the same layout.
//
// The three kernels overlap at their seams by programmatic dependent launch: the decode and the
// expansion are launched as dependents of the kernel ahead of them. The query kernel lets the
// decode launch once its MMAs are done, so the decode sets up and fills its ring of cache tiles
// while the absorbed queries are stored; the decode lets the expansion launch at its set-up, so
// the expansion stages W_post during the decode's tail. Each waits for its predecessor only
// before reading that kernel's output.
//
// Roles (160 threads): warps 0-3 read and write the TMEM lanes (thread t = row t of the block);
// warp 4 owns TMEM, issues the TMA copies and (one lane) the MMAs. Every wait is bounded (about
// one second); a wait that runs out raises KL_FLAG_TIMEOUT and the CTA leaves after its copies
// and MMAs have drained.
#include <cudaTypedefs.h>

#include "kl_internal.cuh"
#include "kl_tc_ptx.cuh"

namespace kl {
namespace {

constexpr int kBM = 128;                 // sequences per CTA (MMA rows, TMEM lanes)
constexpr int kR = 128;                  // latent width r
constexpr int kThreads = 5 * 32;
constexpr int kCtlWarp = 4;
constexpr uint32_t kBox = 16384;         // one 128-row x 128-byte swizzled box
constexpr uint32_t kTmemCols = 256;
constexpr uint64_t kTimeoutNs = 1000000000ull;

// Shared memory of both kernels (1024-byte aligned). Query: stage = Q (boxes 0-1, the 64-dim
// halves) and W^R (boxes 2-3, 64-column halves), w = W_post[h] (64-column halves); the result
// (four 32-value column boxes) is staged over Q and W^R. Expansion: w = W_post[h], stage = the
// O* rows (four 32-value column boxes), then the result.
struct __align__(1024) LatentSmem {
    uint8_t stage[4 * kBox];
    uint8_t w[2 * kBox];
    uint64_t full, wfull, r_full, a_ready, d_full, drain;
    uint32_t tmem_base;
    int abort;
};

// Bounded wait on an mbarrier phase (every lane of the warp calls it; all get the same answer).
__device__ bool wait_bar(LatentSmem &sm, uint64_t *bar, uint32_t parity, int32_t *err) {
    bool ok = ptx::mbar_try_wait(bar, parity);
    if (!ok) {
        const uint64_t t0 = ptx::globaltimer();
        while (true) {
            if (ptx::mbar_try_wait(bar, parity)) { ok = true; break; }
            if (*reinterpret_cast<volatile int *>(&sm.abort)) break;
            if (ptx::globaltimer() - t0 > kTimeoutNs) {
                sm.abort = 1;
                raise_flag(err, KL_FLAG_TIMEOUT);
                break;
            }
        }
    }
    return __all_sync(0xffffffffu, ok);
}

// Bounded wait, no flag: the copies or MMAs tracked by `bar` have landed (teardown only).
__device__ void settle(uint64_t *bar, uint32_t parity) {
    const uint64_t t0 = ptx::globaltimer();
    while (!ptx::mbar_try_wait(bar, parity) && ptx::globaltimer() - t0 < kTimeoutNs) {
    }
}

// x = hi + lo with hi = bf16(x), lo = bf16(x - hi), for two values packed as bf16 pairs.
__device__ __forceinline__ void split2(float x0, float x1, uint32_t &hi, uint32_t &lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
    const float2 hf = __bfloat1622float2(h);
    const __nv_bfloat162 l = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t x, uint32_t y, uint32_t z,
                                             uint32_t w) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(x), "r"(y), "r"(z),
                 "r"(w)
                 : "memory");
}

__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(addr)
                 : "memory");
    return v;
}

// Shared address of the 16-byte chunk j of row t in the swizzled box at `box`.
__device__ __forceinline__ uint32_t box_chunk(uint32_t box, int t, int j) {
    return box + t * 128 + ((j ^ (t & 7)) << 4);
}

// K-major SW128 operand of 64-value halves kBox apart: start-address step of k step kk (16
// values: 32 bytes inside a half, the next half every 4 steps), in 16-byte units.
__device__ __forceinline__ uint32_t kstep(int kk) { return ((kk >> 2) * kBox + (kk & 3) * 32) >> 4; }

__device__ __forceinline__ LatentSmem &smem_of(uint8_t *raw) {
    return *reinterpret_cast<LatentSmem *>((reinterpret_cast<uintptr_t>(raw) + 1023) &
                                           ~uintptr_t(1023));
}

// Barriers, TMEM, and the set-up fences common to both kernels.
__device__ void setup(LatentSmem &sm, int warp) {
    if (threadIdx.x == 0) {
        ptx::mbar_init(&sm.full, 1);
        ptx::mbar_init(&sm.wfull, 1);
        ptx::mbar_init(&sm.r_full, 1);
        ptx::mbar_init(&sm.a_ready, 4);
        ptx::mbar_init(&sm.d_full, 1);
        ptx::mbar_init(&sm.drain, 1);
        sm.abort = 0;
        ptx::fence_mbar_init();
    }
    if (warp == kCtlWarp) {
        ptx::tmem_alloc(&sm.tmem_base, kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
}

// Every MMA of the control warp has completed, all threads meet, TMEM is freed.
__device__ void teardown(LatentSmem &sm, int warp, int lane) {
    if (warp == kCtlWarp) {
        if (lane == 0) {
            ptx::mma_commit(&sm.drain);
            settle(&sm.drain, 0);
        }
        __syncwarp();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == kCtlWarp) ptx::tmem_dealloc(sm.tmem_base, kTmemCols);
}

// ------------------------------------------------------------------- absorbed query ----
// CTA (h, block): Q_r = Q . W^R into TMEM columns 0 .. D-1; Q_r as hi | lo pairs into columns
// 128 .. 191 | 192 .. 255; Q* = Q_r . W_post^T into columns 0 .. 127; then q_lat.
__global__ void __launch_bounds__(kThreads, 1)
    latent_query_kernel(const __grid_constant__ CUtensorMap qmap,
                        const __grid_constant__ CUtensorMap wrmap,
                        const __grid_constant__ CUtensorMap wpmap,
                        const __grid_constant__ CUtensorMap qlmap, int D, int G, int wr_per_qh,
                        int32_t *err) {
    extern __shared__ uint8_t smem_raw[];
    LatentSmem &sm = smem_of(smem_raw);
    const int h = blockIdx.x, b0 = blockIdx.y * kBM;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nh = D / 64;                     // 64-value halves of a query row
    setup(sm, warp);
    const uint32_t tmem = sm.tmem_base;
    uint8_t *const q_s = sm.stage, *const wr_s = sm.stage + 2 * kBox;

    if (warp == kCtlWarp) {
        if (lane == 0) {
            ptx::prefetch_tensormap(&qmap);
            ptx::prefetch_tensormap(&wrmap);
            ptx::prefetch_tensormap(&wpmap);
            ptx::prefetch_tensormap(&qlmap);
            // Q rows (rows past the batch read as zeros), W^R[w(h)] (D k rows per half),
            // W_post[h] (128 latent rows per half)
            ptx::mbar_arrive_expect_tx(&sm.full, nh * (2 * kBox + (uint32_t)D * 128));
            const int wrow = (wr_per_qh ? h : h / G) * D;
            for (int x = 0; x < nh; ++x) {
                ptx::tma_load_3d(q_s + x * kBox, &qmap, &sm.full, 64 * x, h, b0);
                ptx::tma_load_2d(wr_s + x * kBox, &wrmap, &sm.full, 64 * x, wrow);
                ptx::tma_load_2d(sm.w + x * kBox, &wpmap, &sm.full, 64 * x, h * kR);
            }
        }
        __syncwarp();
        bool ok = wait_bar(sm, &sm.full, 0, err);
        if (ok) {
            ptx::tc_fence_after();
            if (lane == 0) {
                // Q_r = Q . W^R: A = Q (K-major), B = W^R (N = output dim, MN-major: halves kBox
                // apart, 16 k rows = 2 KiB per step)
                const uint64_t qd = ptx::smem_desc(ptx::smem_addr(q_s), 16, 1024, ptx::kSwizzle128B);
                const uint64_t wd = ptx::smem_desc(ptx::smem_addr(wr_s), kBox, 1024, ptx::kSwizzle128B);
                const uint32_t idesc = ptx::idesc_bf16(kBM, D, false, true);
                for (int kk = 0; kk < D / 16; ++kk)
                    ptx::mma_bf16(tmem, qd + kstep(kk), wd + ((kk * 2048) >> 4), idesc, kk > 0);
                ptx::mma_commit(&sm.r_full);
            }
            __syncwarp();
            ok = wait_bar(sm, &sm.a_ready, 0, err);
        } else if (lane == 0) {
            settle(&sm.full, 0);      // copies in flight land before shared memory goes away
        }
        if (ok) {
            ptx::tc_fence_after();
            if (lane == 0) {
                // Q* = Q_hi . W_post^T + Q_lo . W_post^T: A = the pairs in TMEM (8 packed
                // columns per step), B = W_post[h] (N = the r latent rows, K-major over D)
                const uint64_t pd = ptx::smem_desc(ptx::smem_addr(sm.w), 16, 1024, ptx::kSwizzle128B);
                const uint32_t idesc = ptx::idesc_bf16(kBM, kR, false, false);
                const int ks = D / 16;
                for (int kk = 0; kk < 2 * ks; ++kk) {
                    const int k = kk % ks;
                    ptx::mma_bf16_ts(tmem, tmem + 128 + (kk >= ks ? 64u : 0u) + 8 * k,
                                     pd + kstep(k), idesc, kk > 0);
                }
                ptx::mma_commit(&sm.d_full);
            }
            __syncwarp();
        }
        grid_dep_launch();
    } else {
        const int t = tid;                                   // row of the block = TMEM lane
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        bool ok = wait_bar(sm, &sm.r_full, 0, err);
        if (ok) {
            ptx::tc_fence_after();
            for (int c = 0; c < nh; ++c) {
                uint32_t u0[32], u1[32], hi[32], lo[32];
                ptx::tmem_ld32(tmem + lane_base + 64 * c, u0);
                ptx::tmem_ld32(tmem + lane_base + 64 * c + 32, u1);
                ptx::tmem_wait_ld();
                ptx::reg_fence(u0);
                ptx::reg_fence(u1);
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    split2(__uint_as_float(u0[2 * e]), __uint_as_float(u0[2 * e + 1]), hi[e], lo[e]);
                    split2(__uint_as_float(u1[2 * e]), __uint_as_float(u1[2 * e + 1]), hi[16 + e],
                           lo[16 + e]);
                }
                ptx::tmem_st32(tmem + lane_base + 128 + 32 * c, hi);
                ptx::tmem_st32(tmem + lane_base + 192 + 32 * c, lo);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
        }
        __syncwarp();
        if (ok && lane == 0) ptx::mbar_arrive(&sm.a_ready);
        ok = ok && wait_bar(sm, &sm.d_full, 0, err);
        // The decode behind this kernel may start setting up now, during the store: launched
        // earlier, its CTAs slow this kernel's TMEM passes on the SMs they share.
        grid_dep_launch();
        if (ok) {
            // Q* row t -> four 32-value boxes over Q and W^R (their MMAs have completed)
            ptx::tc_fence_after();
            const uint32_t stage = ptx::smem_addr(sm.stage);
#pragma unroll
            for (int c = 0; c < kR / 32; ++c) {
                uint32_t u[32];
                ptx::tmem_ld32(tmem + lane_base + 32 * c, u);
                ptx::tmem_wait_ld();
                ptx::reg_fence(u);
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    st_shared_v4(box_chunk(stage + c * kBox, t, j), u[4 * j], u[4 * j + 1],
                                 u[4 * j + 2], u[4 * j + 3]);
            }
            ptx::fence_proxy_async_smem();
        }
        ptx::tc_fence_before();
        if (ptx::bar_and(1, 128, ok) && t == 0) {
            for (int c = 0; c < kR / 32; ++c)
                ptx::tma_store_3d(&qlmap, sm.stage + c * kBox, 32 * c, h, b0);
            ptx::bulk_commit();
            ptx::bulk_wait_read();
        }
    }
    teardown(sm, warp, lane);
}

// -------------------------------------------------------------------------- expansion ----
// CTA (h, block): W_post[h] staged before the wait on the decode; the O* rows by TMA; the pairs
// into TMEM columns 0 .. 63 | 64 .. 127; O = O* . W_post into columns 128 .. 128 + D - 1; then
// out (bf16 or fp32).
__global__ void __launch_bounds__(kThreads, 1)
    latent_expand_kernel(const __grid_constant__ CUtensorMap olmap,
                         const __grid_constant__ CUtensorMap wpmap,
                         const __grid_constant__ CUtensorMap outmap, int D, int out_fp32,
                         int32_t *err) {
    extern __shared__ uint8_t smem_raw[];
    LatentSmem &sm = smem_of(smem_raw);
    const int h = blockIdx.x, b0 = blockIdx.y * kBM;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    setup(sm, warp);
    const uint32_t tmem = sm.tmem_base;

    if (warp == kCtlWarp) {
        if (lane == 0) {
            ptx::prefetch_tensormap(&olmap);
            ptx::prefetch_tensormap(&wpmap);
            ptx::prefetch_tensormap(&outmap);
            ptx::mbar_arrive_expect_tx(&sm.wfull, (D / 64) * kBox);
            for (int x = 0; x < D / 64; ++x)
                ptx::tma_load_2d(sm.w + x * kBox, &wpmap, &sm.wfull, 64 * x, h * kR);
            // O* is the decode's output: wait for the decode, then its rows (past the batch:
            // zeros)
            grid_dep_wait();
            ptx::mbar_arrive_expect_tx(&sm.full, 4 * kBox);
            for (int c = 0; c < 4; ++c)
                ptx::tma_load_3d(sm.stage + c * kBox, &olmap, &sm.full, 32 * c, h, b0);
        }
        __syncwarp();
        bool ok = wait_bar(sm, &sm.wfull, 0, err);
        ok = ok && wait_bar(sm, &sm.a_ready, 0, err);
        if (ok) {
            ptx::tc_fence_after();
            if (lane == 0) {
                // O = O*_hi . W_post + O*_lo . W_post: A = the pairs in TMEM, B = W_post[h]
                // (N = output dim, MN-major: halves kBox apart, 16 latent rows = 2 KiB per step)
                const uint64_t pd = ptx::smem_desc(ptx::smem_addr(sm.w), kBox, 1024, ptx::kSwizzle128B);
                const uint32_t idesc = ptx::idesc_bf16(kBM, D, false, true);
                for (int kk = 0; kk < 2 * kR / 16; ++kk)
                    ptx::mma_bf16_ts(tmem + 128, tmem + (kk >= 8 ? 64u : 0u) + 8 * (kk & 7),
                                     pd + (((kk & 7) * 2048) >> 4), idesc, kk > 0);
                ptx::mma_commit(&sm.d_full);
            }
            __syncwarp();
        } else if (lane == 0) {
            settle(&sm.wfull, 0);
            settle(&sm.full, 0);
        }
    } else {
        const int t = tid;
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        const uint32_t stage = ptx::smem_addr(sm.stage);
        bool ok = wait_bar(sm, &sm.full, 0, err);
        if (ok) {
            // row t of O*: box 2c + q holds values 64c + 32q .. + 31, four per chunk
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                uint32_t hi[32], lo[32];
#pragma unroll
                for (int q = 0; q < 2; ++q) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint4 v = ld_shared_v4(box_chunk(stage + (2 * c + q) * kBox, t, j));
                        split2(__uint_as_float(v.x), __uint_as_float(v.y), hi[16 * q + 2 * j],
                               lo[16 * q + 2 * j]);
                        split2(__uint_as_float(v.z), __uint_as_float(v.w), hi[16 * q + 2 * j + 1],
                               lo[16 * q + 2 * j + 1]);
                    }
                }
                ptx::tmem_st32(tmem + lane_base + 32 * c, hi);
                ptx::tmem_st32(tmem + lane_base + 64 + 32 * c, lo);
            }
            ptx::tmem_wait_st();
            ptx::tc_fence_before();
        }
        __syncwarp();
        if (ok && lane == 0) ptx::mbar_arrive(&sm.a_ready);
        // d_full follows every thread's arrival, so all O* rows have been read: the result is
        // staged over them
        ok = ok && wait_bar(sm, &sm.d_full, 0, err);
        const int box_cols = out_fp32 ? 32 : 64;
        if (ok) {
            ptx::tc_fence_after();
            for (int c = 0; c < D / 32; ++c) {
                uint32_t u[32];
                ptx::tmem_ld32(tmem + lane_base + 128 + 32 * c, u);
                ptx::tmem_wait_ld();
                ptx::reg_fence(u);
                if (out_fp32) {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        st_shared_v4(box_chunk(stage + c * kBox, t, j), u[4 * j], u[4 * j + 1],
                                     u[4 * j + 2], u[4 * j + 3]);
                } else {
                    // 32 values = 64 bytes: chunks 4 (c % 2) .. + 3 of box c / 2
                    const uint32_t box = stage + (c >> 1) * kBox;
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        uint32_t p[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const __nv_bfloat162 v =
                                __floats2bfloat162_rn(__uint_as_float(u[8 * j + 2 * e]),
                                                      __uint_as_float(u[8 * j + 2 * e + 1]));
                            p[e] = *reinterpret_cast<const uint32_t *>(&v);
                        }
                        st_shared_v4(box_chunk(box, t, 4 * (c & 1) + j), p[0], p[1], p[2], p[3]);
                    }
                }
            }
            ptx::fence_proxy_async_smem();
        }
        ptx::tc_fence_before();
        if (ptx::bar_and(1, 128, ok) && t == 0) {
            for (int c = 0; c < D / box_cols; ++c)
                ptx::tma_store_3d(&outmap, sm.stage + c * kBox, box_cols * c, h, b0);
            ptx::bulk_commit();
            ptx::bulk_wait_read();
        }
    }
    teardown(sm, warp, lane);
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

// Tensor map with the 128-byte swizzle: dims innermost first, strides in bytes (rank - 1).
bool encode(CUtensorMap *map, CUtensorMapDataType type, int rank, const void *base,
            const cuuint64_t *dims, const cuuint64_t *strides, const cuuint32_t *box) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, type, rank, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Rows [B][Hq][cols] of `esize`-byte values; one box = `box_cols` columns (128 bytes) of one
// head for 128 consecutive sequences.
bool rows_map(CUtensorMap *map, CUtensorMapDataType type, size_t esize, const void *base, int B,
              int Hq, int cols, int box_cols) {
    const cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)Hq, (cuuint64_t)B};
    const cuuint64_t strides[2] = {(cuuint64_t)cols * esize, (cuuint64_t)Hq * cols * esize};
    const cuuint32_t box[3] = {(cuuint32_t)box_cols, 1, kBM};
    return encode(map, type, 3, base, dims, strides, box);
}

// `rows` rows of `cols` bf16 values; one box = 64 columns x `box_rows` rows.
bool matrix_map(CUtensorMap *map, const void *base, uint64_t rows, int cols, int box_rows) {
    const cuuint64_t dims[2] = {(cuuint64_t)cols, rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box);
}

constexpr size_t kSmemBytes = sizeof(LatentSmem) + 1024;

template <typename Kernel>
cudaError_t configure(Kernel kernel, PerDeviceOnce &once) {
    return once.run([&] {
        return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)kSmemBytes);
    });
}

}  // namespace

cudaError_t launch_latent_query(int B, int Hq, int G, int D, int r, int wr_per_qh,
                                const uint16_t *q, const uint16_t *w_r, const uint16_t *w_post,
                                float *q_lat, int32_t *err, cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    if ((D != 64 && D != 128) || r != kR || G <= 0 || Hq % G) return cudaErrorInvalidValue;
    const int Hw = wr_per_qh ? Hq : Hq / G;
    CUtensorMap qmap, wrmap, wpmap, qlmap;
    if (!rows_map(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, q, B, Hq, D, 64) ||
        !matrix_map(&wrmap, w_r, (uint64_t)Hw * D, D, D) ||
        !matrix_map(&wpmap, w_post, (uint64_t)Hq * kR, D, kR) ||
        !rows_map(&qlmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, q_lat, B, Hq, kR, 32))
        return cudaErrorInvalidValue;
    static PerDeviceOnce once;
    cudaError_t e = configure(latent_query_kernel, once);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(Hq, (B + kBM - 1) / kBM);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = stream;
    return cudaLaunchKernelEx(&cfg, latent_query_kernel, qmap, wrmap, wpmap, qlmap, D, G, wr_per_qh,
                              err);
}

cudaError_t launch_latent_expand(int B, int Hq, int D, int r, const float *o_lat,
                                 const uint16_t *w_post, void *out, kl_dtype out_dtype,
                                 int32_t *err, cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    if ((D != 64 && D != 128) || r != kR) return cudaErrorInvalidValue;
    const bool fp32 = out_dtype == KL_FP32;
    CUtensorMap olmap, wpmap, outmap;
    if (!rows_map(&olmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, o_lat, B, Hq, kR, 32) ||
        !matrix_map(&wpmap, w_post, (uint64_t)Hq * kR, D, kR) ||
        !rows_map(&outmap, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                  fp32 ? 4 : 2, out, B, Hq, D, fp32 ? 32 : 64))
        return cudaErrorInvalidValue;
    static PerDeviceOnce once;
    cudaError_t e = configure(latent_expand_kernel, once);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(Hq, (B + kBM - 1) / kBM);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = stream;
    // a programmatic dependent of the decode (or of its combine kernel)
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, latent_expand_kernel, olmap, wpmap, outmap, D, (int)fp32, err);
}

}  // namespace kl
