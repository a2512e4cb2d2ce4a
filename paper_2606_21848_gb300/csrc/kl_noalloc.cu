// kl_decode_attention_noalloc: the keyless decode for callers that cannot allocate device
// memory. The split states that kl_decode_attention keeps in a caller-provided workspace live
// here in one fixed, file-scope device array instead.
#include <cudaTypedefs.h>

#include <mutex>

#include "kl_internal.cuh"

namespace kl {
namespace {

// Fixed scratch for split states: [B][Hq][S][D] fp32 outputs, then [B][Hq][S][2] fp32 {m, l}.
// Every GPU that loads this library holds these bytes until the process exits.
constexpr size_t kScratchBytes = (size_t)KL_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_split_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
// Per device: the device address of the scratch array and the id of the CUDA context it was
// looked up in. The address belongs to the module loaded into that context, so a new context on
// the device (after cudaDeviceReset, say) gets its own lookup.
void *g_scratch_ptr[kMaxDevices] = {nullptr};
unsigned long long g_scratch_ctx[kMaxDevices] = {0};

// The unique id of the calling thread's current context (0 if it cannot be read).
unsigned long long current_context_id() {
    static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
    static PFN_cuCtxGetId_v12000 get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
    });
    if (!get_current || !get_id) return 0;
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch array for the current device and context. Host code cannot
// use the symbol itself as a device address: cudaGetSymbolAddress translates it, once per
// device and context (the runtime makes the device's primary context current first).
cudaError_t scratch_for_current_device(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    const unsigned long long ctx = current_context_id();
    if (!g_scratch_ptr[dev] || ctx == 0 || ctx != g_scratch_ctx[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_split_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
        // the context id is read again after the lookup, which may have created the context
        g_scratch_ctx[dev] = current_context_id();
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

size_t round_up256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace
}  // namespace kl

extern "C" kl_status kl_decode_attention_noalloc(const kl_shape *shape, const void *q,
                                                 const void *w_r, const void *v_cache,
                                                 const int32_t *block_table,
                                                 const int32_t *seq_lens, int32_t num_splits,
                                                 void *out, kl_dtype out_dtype, int32_t *err,
                                                 kl_stream_t stream) {
    using namespace kl;
    if (!shape || num_splits < 0) return KL_ERR_INVALID_ARG;
    const int32_t S = kl_decode_num_splits(shape, num_splits);
    if (S <= 0) return KL_ERR_INVALID_ARG;
    if (S == 1)   // no split states: the ordinary path needs no workspace either
        return kl_decode_attention(shape, q, w_r, v_cache, block_table, seq_lens, 1, out,
                                   out_dtype, nullptr, 0, err, stream);
    const size_t rows = (size_t)shape->num_seqs * shape->num_q_heads * S;
    const size_t o_bytes = round_up256(rows * shape->head_dim * sizeof(float));
    const size_t ml_bytes = round_up256(rows * 2 * sizeof(float));
    if (o_bytes + ml_bytes > kScratchBytes) return KL_ERR_WORKSPACE;
    // the decode below writes split states, not `out`, so `out` is checked here as
    // kl_decode_attention checks it
    if (!out || (reinterpret_cast<uintptr_t>(out) & 15u) != 0) return KL_ERR_INVALID_ARG;

    void *base = nullptr;
    if (scratch_for_current_device(&base) != cudaSuccess) return KL_ERR_CUDA;
    float *part_o = static_cast<float *>(base);
    float *part_ml = reinterpret_cast<float *>(static_cast<unsigned char *>(base) + o_bytes);
    kl_decode_options opts{S, KL_KERNEL_AUTO, part_o, part_ml};
    kl_status st = kl_decode_attention_ex(shape, q, w_r, v_cache, block_table, seq_lens, &opts,
                                          nullptr, out_dtype, nullptr, 0, err, stream);
    if (st != KL_OK) return st;
    return kl_combine(shape, part_o, part_ml, S, out, out_dtype, stream);
}
