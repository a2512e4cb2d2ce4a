// Internal declarations shared by the translation units of libkeyless.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "keyless.h"

namespace kl {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr uint64_t kDefaultWaitNs = 1000000000ull;   // about one second
// Wait limits below this are kept exactly: the decodes are then launched in a variant whose
// waits poll without suspending (a suspended try_wait can outlast such a limit).
constexpr uint64_t kExactWaitNs = 100000ull;

// The pipeline-wait limit in force (kl_set_wait_timeout_ns; the default unless set).
uint64_t current_wait_ns();

// Geometry of one decode call, resolved on the host.
struct Geometry {
    int B, Hq, Hkv, G, D, P, num_pages, max_pages, wr_per_qh;
    float scale;       // lambda / sqrt(d_k)
    int S;             // split count
    int chunk;         // tokens per split (a multiple of 128)
    int spc = 1;       // splits per CTA of the tensor-core decode (consecutive, same (b, g))
    int nhb = 1;       // CTAs per (run of splits, b, g): blocks of up to 8 query heads
    int qbox = 8;      // query rows of one CTA: min(G, 8), or 2 G with two value heads
    int vpc = 1;       // value heads per CTA of the tensor-core decode: 2 at head dim 64 (the
                       // two heads' rows side by side in one 128-wide tile), else 1
};

// Arguments of a decode launch (keyless or the standard K+V comparison).
struct DecodeArgs {
    Geometry geo;
    const uint16_t *q;        // [B][Hq][D] bf16
    const uint16_t *w_r;      // [Hw][D][D] bf16 (keyless only)
    // Pre-routed queries (tensor-core kernel only): when set, q and w_r are unused and the
    // kernel scores with q_routed[b][h][:] (fp32, [B][Hq][D]) as the routed query, e.g. the
    // absorbed query of a latent value-only cache.
    const float *q_routed;
    const uint16_t *k_cache;  // [num_pages][Hkv][P][D] bf16 (standard only)
    const uint16_t *v_cache;  // [num_pages][Hkv][P][D] bf16
    const int32_t *block_table;
    const int32_t *seq_lens;
    // Fused append (kl_decode_step): when v_new is set, the CTA whose split holds row
    // positions[b] writes v_new[b][g] there (into cache_rw, the value cache) before it reads it.
    const uint16_t *v_new;            // [B][Hkv][D] bf16 or nullptr
    const int32_t *positions;         // [B]
    uint16_t *cache_rw;
    // FP8 step (kl_decode_step_fp8): the row positions[b] of the code and scale caches receives
    // v_new[b][g] quantized, in the same way, from the CTA whose split holds it.
    uint8_t *codes_rw = nullptr;
    float *scales_rw = nullptr;
    float *part_o;            // [B][Hq][S][D]   split states (unless direct_out)
    float *part_ml;           // [B][Hq][S][2]
    void *out;                // [B][Hq][D]
    bool direct_out;          // true: S == 1 and the CTA writes `out` itself (no split states)
    bool merge_inside;        // true: the last split of each (b, g) merges the split states
                              // into `out` (tensor-core kernel), using the workspace counters
    unsigned int *counters;   // [B][Hkv][nhb] arrivals of the current call (zero between calls)
    kl_dtype out_dtype;
    int32_t *err;
    cudaStream_t stream;
    // Limit of each pipeline wait of the tensor-core decodes (ns); the drains of a CTA that gave
    // up keep the full default so that its copies and MMAs complete before it exits.
    uint64_t wait_ns = kDefaultWaitNs;
    // Latent path: the launch is a programmatic dependent of the absorbed-query kernel ahead of
    // it; the CTAs set up and fill their ring of cache tiles at once, every role then sleeps in
    // grid_dep_wait until that kernel has finished (the compute warps before reading q_routed),
    // and every CTA lets the expansion kernel behind it launch early (grid_dep_launch).
    bool pdl = false;
};

// Arguments of a chunked-prefill launch (kl_prefill_attention). Sequence b's query rows are
// cu_q[b] .. cu_q[b + 1] - 1 of q / out ([total_q][Hq][D]); they are the last n_b rows of its
// seq_lens[b] cached rows, so query row i sits at position seq_lens[b] - n_b + i.
struct PrefillArgs {
    Geometry geo;             // S and chunk unused
    int total_q;              // rows of q and out
    int max_q;                // host bound on n_b (grid sizing)
    const uint16_t *q;        // [total_q][Hq][D] bf16
    const uint16_t *w_r;      // [Hw][D][D] bf16
    const uint16_t *v_cache;  // [num_pages][Hkv][P][D] bf16
    const int32_t *block_table;
    const int32_t *seq_lens;
    const int32_t *cu_q;      // [B + 1]
    void *out;                // [total_q][Hq][D]
    kl_dtype out_dtype;
    int32_t *err;
    cudaStream_t stream;
};

// bf16 bit helpers (a bf16 value is the upper half of a binary32 value).
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ void raise_flag(int32_t *err, int32_t bits) {
    if (err) atomicOr(err, bits);
}

// Programmatic dependent launch. A kernel launched with programmatic stream serialization may
// start before the kernel ahead of it in the stream has finished: grid_dep_wait() blocks the
// calling thread until that kernel has completed and its writes are visible (it returns at once
// for an ordinary launch), and grid_dep_launch() lets such a follower start once every CTA of
// the calling grid has signalled or exited.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launchers (each returns cudaGetLastError() of its launch).
cudaError_t launch_append(const Geometry &g, const uint16_t *v_new, const int32_t *block_table,
                          const int32_t *positions, uint16_t *v_cache, int32_t *err,
                          cudaStream_t stream);
cudaError_t launch_route(const Geometry &g, const uint16_t *q, const uint16_t *w_r, float *q_r,
                         cudaStream_t stream);
// dependent: launched as a programmatic dependent of the decode just before it in the stream
// (it starts once every decode CTA has set up and waits for the decode to complete)
cudaError_t launch_combine(int B, int Hq, int D, int S, const float *part_o,
                           const float *part_ml, void *out, kl_dtype out_dtype,
                           cudaStream_t stream, bool dependent = false);
cudaError_t launch_decode_simt(const DecodeArgs &a, bool standard);
// Merges the split states of a finished decode into `out` unless it wrote `out` directly or
// the caller asked for the states.
cudaError_t finish_decode(const DecodeArgs &a, bool states_requested);

// Tensor-core path: whether it supports a geometry, and its launcher.
bool tc_supported(const Geometry &g, bool standard);
// Whether the tensor-core kernel can merge this geometry's split states itself.
bool tc_merge_inside(const Geometry &g, bool standard);
cudaError_t launch_decode_tc(const DecodeArgs &a, bool standard);

// Chunked prefill on the tensor cores (head_dim 128, compute capability 10.3) and the
// chunk append.
bool prefill_tc_supported(const Geometry &g);
cudaError_t launch_prefill_tc(const PrefillArgs &a);
cudaError_t launch_append_chunk(const Geometry &g, int total_q, int max_q, const uint16_t *v_new,
                                const int32_t *block_table, const int32_t *seq_lens,
                                const int32_t *cu_q, uint16_t *v_cache, int32_t *err,
                                cudaStream_t stream);

// FP8 value cache (E4M3 codes [num_pages][Hkv][P][D] with fp32 row scales [num_pages][Hkv][P]):
// the decode on the tensor cores (a.v_cache holds the codes; states or direct output, merged by
// the combine kernel) and the quantizing append.
cudaError_t launch_decode_fp8(const DecodeArgs &a, const float *v_scales);
cudaError_t launch_append_fp8(const Geometry &g, const uint16_t *v_new, const int32_t *block_table,
                              const int32_t *positions, uint8_t *codes, float *scales, int32_t *err,
                              cudaStream_t stream);
cudaError_t launch_quantize_fp8(size_t rows, const uint16_t *v, uint8_t *codes, float *scales,
                                cudaStream_t stream);

// Latent value-only cache (head_dim D of queries and outputs, latent width r):
// q_lat[b][h] = (q[b][h] W^R[w(h)]) W_post[h]^T and out[b][h] = o_lat[b][h] W_post[h].
// Tensor-core kernels (D 64 or 128, r 128); the expansion is launched as a programmatic
// dependent of the kernel ahead of it.
cudaError_t launch_latent_query(int B, int Hq, int G, int D, int r, int wr_per_qh,
                                const uint16_t *q, const uint16_t *w_r, const uint16_t *w_post,
                                float *q_lat, int32_t *err, cudaStream_t stream);
cudaError_t launch_latent_expand(int B, int Hq, int D, int r, const float *o_lat,
                                 const uint16_t *w_post, void *out, kl_dtype out_dtype,
                                 int32_t *err, cudaStream_t stream);

// Number of SMs of the current device (cached per device).
int device_sm_count();

// A launch site's one-time set-up of its kernel (a function attribute, which belongs to the
// function on the current device): run once per device (ordinals below 64; others every time).
struct PerDeviceOnce {
    std::atomic<uint64_t> done{0};
    template <typename F>
    cudaError_t run(F &&setup) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        const uint64_t bit = dev >= 0 && dev < 64 ? 1ull << dev : 0ull;
        if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
        e = setup();
        if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
        return e;
    }
};

}  // namespace kl
