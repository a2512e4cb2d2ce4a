// C-ABI entry points of libkeyless: host-side validation, split planning, workspace layout
// and dispatch to the kernels. Nothing here allocates, frees or synchronizes.
#include <math.h>
#include <stdint.h>

#include <atomic>

#include "kl_internal.cuh"

namespace kl {

namespace {
std::atomic<uint64_t> g_wait_ns{0};   // 0: the default
}  // namespace

uint64_t current_wait_ns() {
    const uint64_t v = g_wait_ns.load(std::memory_order_relaxed);
    return v ? v : kDefaultWaitNs;
}

int device_sm_count() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
    int n = 1;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
        n = 1;
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

namespace {

constexpr int kChunkQuantum = 128;  // split boundaries fall on multiples of 128 tokens
constexpr int kSimtMaxGroup = 8;    // query heads per value head of the CUDA-core kernel
constexpr int kMaxSplits = 1024;

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Validate the shape and resolve the split plan. `num_splits` < 0 skips split planning.
kl_status resolve(const kl_shape *s, int32_t num_splits, Geometry *g) {
    if (!s) return KL_ERR_INVALID_ARG;
    if (s->num_seqs < 0 || s->num_q_heads <= 0 || s->num_kv_heads <= 0 || s->page_size <= 0 ||
        s->num_pages <= 0 || s->max_pages_per_seq <= 0 || s->head_dim <= 0)
        return KL_ERR_INVALID_ARG;
    if (s->num_q_heads % s->num_kv_heads != 0) return KL_ERR_INVALID_ARG;
    if (s->head_dim != 64 && s->head_dim != 128) return KL_ERR_UNSUPPORTED;
    if ((int64_t)s->max_pages_per_seq * s->page_size > (int64_t)INT32_MAX / 2)
        return KL_ERR_INVALID_ARG;
    if (!(s->scale == s->scale)) return KL_ERR_INVALID_ARG;  // NaN
    g->B = s->num_seqs;
    g->Hq = s->num_q_heads;
    g->Hkv = s->num_kv_heads;
    g->G = s->num_q_heads / s->num_kv_heads;
    g->D = s->head_dim;
    g->P = s->page_size;
    g->num_pages = s->num_pages;
    g->max_pages = s->max_pages_per_seq;
    g->wr_per_qh = s->wr_per_query_head ? 1 : 0;
    g->scale = s->scale > 0.f ? s->scale : 1.0f / sqrtf((float)s->head_dim);
    g->S = 1;
    g->chunk = 0;
    g->nhb = (g->G + 7) / 8;
    g->qbox = g->G < 8 ? g->G : 8;
    // head dim 64: a tensor-core CTA takes two value heads (even Hkv, groups of up to 4)
    g->vpc = (g->D == 64 && g->Hkv % 2 == 0 && g->G <= 4) ? 2 : 1;
    if (g->vpc == 2) g->qbox = 2 * g->G;
    if (num_splits < 0) return KL_OK;
    if (num_splits > kMaxSplits) return KL_ERR_INVALID_ARG;

    const int64_t Lmax = (int64_t)g->max_pages * g->P;
    int64_t S = num_splits;
    if (S == 0) {
        // As many splits as fit one wave of two CTAs per SM over the (value head, sequence)
        // units, and splits of at most 8192 tokens so that ragged batches balance; never
        // below 256 tokens per split.
        const int64_t units = (int64_t)(g->B > 0 ? g->B : 1) * (g->Hkv / g->vpc) * g->nhb;
        const int64_t slots = 2 * (int64_t)device_sm_count();
        const int64_t fill = units < slots ? slots / units : 1;
        const int64_t cap = (Lmax + 8191) / 8192;
        S = fill > cap ? fill : cap;
        const int64_t smax = (Lmax + 255) / 256;
        if (S > smax) S = smax;
        if (S > kMaxSplits) S = kMaxSplits;
        if (S < 1) S = 1;
    }
    int64_t chunk = (Lmax + S - 1) / S;
    chunk = (chunk + kChunkQuantum - 1) / kChunkQuantum * kChunkQuantum;
    g->chunk = (int)chunk;
    g->S = (int)((Lmax + chunk - 1) / chunk);
    if (g->S < 1) g->S = 1;
    return KL_OK;
}

struct WorkspaceLayout {
    size_t part_o, part_ml, counters, total;
};

// [B][Hkv][nhb] u32 merge counters (one per sequence and block of up to 8 query heads of a
// value head) in a region of at least kCounterFloor counters at the front, then [B][Hq][S][D]
// fp32 states and [B][Hq][S][2] fp32 {m, l}. Every shape with at most kCounterFloor counters
// keeps them in the same region, which no split state ever covers, so the counters that a call
// leaves at zero stay zero whatever shape uses the workspace next.
constexpr size_t kCounterFloor = 16384;
WorkspaceLayout layout(const Geometry &g) {
    WorkspaceLayout w{0, 0, 0, 0};
    if (g.S <= 1) return w;
    const size_t rows = (size_t)g.B * g.Hq * g.S;
    const size_t counters = (size_t)g.B * g.Hkv * g.nhb;
    w.counters = 0;
    w.part_o = round_up((counters > kCounterFloor ? counters : kCounterFloor) * sizeof(unsigned int),
                        256);
    w.part_ml = w.part_o + round_up(rows * g.D * sizeof(float), 256);
    w.total = w.part_ml + round_up(rows * 2 * sizeof(float), 256);
    return w;
}

kl_status from_cuda(cudaError_t e) { return e == cudaSuccess ? KL_OK : KL_ERR_CUDA; }

kl_status decode_common(bool standard, const kl_shape *shape, const void *q, const void *w_r,
                        const void *k_cache, const void *v_cache, const int32_t *block_table,
                        const int32_t *seq_lens, const kl_decode_options *opts, void *out,
                        kl_dtype out_dtype, void *workspace, size_t workspace_bytes,
                        int32_t *err, kl_stream_t stream, const void *v_new = nullptr,
                        const int32_t *positions = nullptr, const float *q_routed = nullptr,
                        bool pdl = false) {
    const int32_t ns = opts ? opts->num_splits : 0;
    const int32_t kernel = opts ? opts->kernel : KL_KERNEL_AUTO;
    if (ns < 0 || kernel < KL_KERNEL_AUTO || kernel > KL_KERNEL_SIMT) return KL_ERR_INVALID_ARG;
    if (out_dtype != KL_BF16 && out_dtype != KL_FP32) return KL_ERR_INVALID_ARG;
    Geometry g;
    kl_status st = resolve(shape, ns, &g);
    if (st != KL_OK) return st;
    if (g.B == 0) return KL_OK;
    if ((!q && !q_routed) || !v_cache || !block_table || !seq_lens) return KL_ERR_INVALID_ARG;
    if (standard && !k_cache) return KL_ERR_INVALID_ARG;   // keyless: w_r == NULL = composed q
    if ((q && !aligned(q, 16)) || !aligned(v_cache, 16) || (w_r && !aligned(w_r, 16)) ||
        (k_cache && !aligned(k_cache, 16)) || (out && !aligned(out, 16)))
        return KL_ERR_INVALID_ARG;

    const bool states = opts && opts->partial_o && opts->partial_ml;
    if (opts && (!opts->partial_o) != (!opts->partial_ml)) return KL_ERR_INVALID_ARG;
    if (!states && !out) return KL_ERR_INVALID_ARG;
    if (states && (!aligned(opts->partial_o, 16) || !aligned(opts->partial_ml, 8)))
        return KL_ERR_INVALID_ARG;
    const WorkspaceLayout wl = states ? WorkspaceLayout{0, 0, 0} : layout(g);
    if (wl.total > 0 && (!workspace || workspace_bytes < wl.total || !aligned(workspace, 256)))
        return KL_ERR_WORKSPACE;

    DecodeArgs a;
    a.geo = g;
    a.q = static_cast<const uint16_t *>(q);
    a.w_r = static_cast<const uint16_t *>(w_r);
    a.q_routed = q_routed;
    a.k_cache = static_cast<const uint16_t *>(k_cache);
    a.v_cache = static_cast<const uint16_t *>(v_cache);
    a.block_table = block_table;
    a.seq_lens = seq_lens;
    a.v_new = static_cast<const uint16_t *>(v_new);
    a.positions = positions;
    a.cache_rw = static_cast<uint16_t *>(const_cast<void *>(v_cache));
    char *ws = static_cast<char *>(workspace);
    a.part_o = states ? opts->partial_o : wl.total ? reinterpret_cast<float *>(ws + wl.part_o) : nullptr;
    a.part_ml = states ? opts->partial_ml : wl.total ? reinterpret_cast<float *>(ws + wl.part_ml) : nullptr;
    a.out = out;
    a.direct_out = !states && g.S == 1;
    a.merge_inside = false;
    a.counters = wl.total ? reinterpret_cast<unsigned int *>(ws + wl.counters) : nullptr;
    a.out_dtype = out_dtype;
    a.err = err;
    a.stream = reinterpret_cast<cudaStream_t>(stream);
    a.pdl = pdl;
    a.wait_ns = current_wait_ns();

    bool use_tc = false;
    if (q_routed && !tc_supported(g, standard)) return KL_ERR_UNSUPPORTED;
    if (q_routed && kernel == KL_KERNEL_SIMT) return KL_ERR_UNSUPPORTED;
    if (kernel == KL_KERNEL_TENSOR || q_routed) {
        if (!tc_supported(g, standard)) return KL_ERR_UNSUPPORTED;
        use_tc = true;
    } else if (kernel == KL_KERNEL_AUTO) {
        use_tc = tc_supported(g, standard);
    }
    // the CUDA-core kernel serves groups of up to 8 query heads
    if (!use_tc && g.G > kSimtMaxGroup) return KL_ERR_UNSUPPORTED;
    a.merge_inside = use_tc && !states && tc_merge_inside(g, standard);
    cudaError_t e = use_tc ? launch_decode_tc(a, standard) : launch_decode_simt(a, standard);
    if (e == cudaSuccess) e = finish_decode(a, states);
    return from_cuda(e);
}

}  // namespace

cudaError_t finish_decode(const DecodeArgs &a, bool states_requested) {
    if (a.direct_out || a.merge_inside || states_requested) return cudaSuccess;
    return launch_combine(a.geo.B, a.geo.Hq, a.geo.D, a.geo.S, a.part_o, a.part_ml, a.out,
                          a.out_dtype, a.stream, true);
}

}  // namespace kl

using namespace kl;

extern "C" {

kl_status kl_route_query(const kl_shape *shape, const void *q, const void *w_r, float *q_r,
                         kl_stream_t stream) {
    Geometry g;
    kl_status st = resolve(shape, -1, &g);
    if (st != KL_OK) return st;
    if (g.B == 0) return KL_OK;
    if (!q || !w_r || !q_r) return KL_ERR_INVALID_ARG;
    return from_cuda(launch_route(g, static_cast<const uint16_t *>(q),
                                  static_cast<const uint16_t *>(w_r), q_r,
                                  reinterpret_cast<cudaStream_t>(stream)));
}

kl_status kl_append_v(const kl_shape *shape, const void *v_new, const int32_t *block_table,
                      const int32_t *positions, void *v_cache, int32_t *err, kl_stream_t stream) {
    Geometry g;
    kl_status st = resolve(shape, -1, &g);
    if (st != KL_OK) return st;
    if (g.B == 0) return KL_OK;
    if (!v_new || !block_table || !positions || !v_cache) return KL_ERR_INVALID_ARG;
    if (!aligned(v_new, 16) || !aligned(v_cache, 16)) return KL_ERR_INVALID_ARG;
    return from_cuda(launch_append(g, static_cast<const uint16_t *>(v_new), block_table,
                                   positions, static_cast<uint16_t *>(v_cache), err,
                                   reinterpret_cast<cudaStream_t>(stream)));
}

size_t kl_decode_workspace_size(const kl_shape *shape, int32_t num_splits) {
    Geometry g;
    if (num_splits < 0 || resolve(shape, num_splits, &g) != KL_OK) return 0;
    return layout(g).total;
}

int32_t kl_decode_num_splits(const kl_shape *shape, int32_t num_splits) {
    Geometry g;
    if (num_splits < 0 || resolve(shape, num_splits, &g) != KL_OK) return 0;
    return g.S;
}

kl_status kl_decode_attention(const kl_shape *shape, const void *q, const void *w_r,
                              const void *v_cache, const int32_t *block_table,
                              const int32_t *seq_lens, int32_t num_splits, void *out,
                              kl_dtype out_dtype, void *workspace, size_t workspace_bytes,
                              int32_t *err, kl_stream_t stream) {
    kl_decode_options o{num_splits, KL_KERNEL_AUTO, nullptr, nullptr};
    return decode_common(false, shape, q, w_r, nullptr, v_cache, block_table, seq_lens, &o, out,
                         out_dtype, workspace, workspace_bytes, err, stream);
}

kl_status kl_decode_attention_ex(const kl_shape *shape, const void *q, const void *w_r,
                                 const void *v_cache, const int32_t *block_table,
                                 const int32_t *seq_lens, const kl_decode_options *opts,
                                 void *out, kl_dtype out_dtype, void *workspace,
                                 size_t workspace_bytes, int32_t *err, kl_stream_t stream) {
    return decode_common(false, shape, q, w_r, nullptr, v_cache, block_table, seq_lens, opts,
                         out, out_dtype, workspace, workspace_bytes, err, stream);
}

kl_status kl_decode_step(const kl_shape *shape, const void *q, const void *w_r,
                         const void *v_new, const int32_t *positions, void *v_cache,
                         const int32_t *block_table, const int32_t *seq_lens,
                         const kl_decode_options *opts, void *out, kl_dtype out_dtype,
                         void *workspace, size_t workspace_bytes, int32_t *err,
                         kl_stream_t stream) {
    if (!v_new || !positions) return KL_ERR_INVALID_ARG;
    if (!aligned(v_new, 16)) return KL_ERR_INVALID_ARG;
    return decode_common(false, shape, q, w_r, nullptr, v_cache, block_table, seq_lens, opts,
                         out, out_dtype, workspace, workspace_bytes, err, stream, v_new,
                         positions);
}

kl_status kl_standard_decode(const kl_shape *shape, const void *q, const void *k_cache,
                             const void *v_cache, const int32_t *block_table,
                             const int32_t *seq_lens, const kl_decode_options *opts, void *out,
                             kl_dtype out_dtype, void *workspace, size_t workspace_bytes,
                             int32_t *err, kl_stream_t stream) {
    return decode_common(true, shape, q, nullptr, k_cache, v_cache, block_table, seq_lens, opts,
                         out, out_dtype, workspace, workspace_bytes, err, stream);
}

kl_status kl_combine(const kl_shape *shape, const float *partial_o, const float *partial_ml,
                     int32_t num_splits, void *out, kl_dtype out_dtype, kl_stream_t stream) {
    Geometry g;
    kl_status st = resolve(shape, -1, &g);
    if (st != KL_OK) return st;
    if (num_splits <= 0 || num_splits > kMaxSplits) return KL_ERR_INVALID_ARG;
    if (out_dtype != KL_BF16 && out_dtype != KL_FP32) return KL_ERR_INVALID_ARG;
    if (g.B == 0) return KL_OK;
    if (!partial_o || !partial_ml || !out) return KL_ERR_INVALID_ARG;
    if (!aligned(partial_ml, 8)) return KL_ERR_INVALID_ARG;
    return from_cuda(launch_combine(g.B, g.Hq, g.D, num_splits, partial_o, partial_ml, out,
                                    out_dtype, reinterpret_cast<cudaStream_t>(stream)));
}

kl_status kl_append_v_chunk(const kl_shape *shape, const void *v_new, const int32_t *block_table,
                            const int32_t *seq_lens, const int32_t *cu_q_lens, int32_t total_q,
                            int32_t max_q_len, void *v_cache, int32_t *err, kl_stream_t stream) {
    Geometry g;
    kl_status st = resolve(shape, -1, &g);
    if (st != KL_OK) return st;
    if (total_q < 0 || max_q_len < 0) return KL_ERR_INVALID_ARG;
    if (g.B == 0 || total_q == 0 || max_q_len == 0) return KL_OK;
    if (!v_new || !block_table || !seq_lens || !cu_q_lens || !v_cache) return KL_ERR_INVALID_ARG;
    if (!aligned(v_new, 16) || !aligned(v_cache, 16)) return KL_ERR_INVALID_ARG;
    return from_cuda(launch_append_chunk(g, total_q, max_q_len, static_cast<const uint16_t *>(v_new),
                                         block_table, seq_lens, cu_q_lens,
                                         static_cast<uint16_t *>(v_cache), err,
                                         reinterpret_cast<cudaStream_t>(stream)));
}

kl_status kl_prefill_attention(const kl_shape *shape, const void *q, const void *w_r,
                               const void *v_cache, const int32_t *block_table,
                               const int32_t *seq_lens, const int32_t *cu_q_lens,
                               int32_t total_q, int32_t max_q_len, void *out, kl_dtype out_dtype,
                               int32_t *err, kl_stream_t stream) {
    Geometry g;
    kl_status st = resolve(shape, -1, &g);
    if (st != KL_OK) return st;
    if (total_q < 0 || max_q_len < 0) return KL_ERR_INVALID_ARG;
    if (out_dtype != KL_BF16 && out_dtype != KL_FP32) return KL_ERR_INVALID_ARG;
    if (!prefill_tc_supported(g)) return KL_ERR_UNSUPPORTED;
    if (g.B == 0 || total_q == 0 || max_q_len == 0) return KL_OK;
    if (!q || !w_r || !v_cache || !block_table || !seq_lens || !cu_q_lens || !out)
        return KL_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(w_r, 16) || !aligned(v_cache, 16) || !aligned(out, 16))
        return KL_ERR_INVALID_ARG;
    if ((int64_t)max_q_len > (int64_t)65535 * 128) return KL_ERR_UNSUPPORTED;
    PrefillArgs a;
    a.geo = g;
    a.total_q = total_q;
    a.max_q = max_q_len;
    a.q = static_cast<const uint16_t *>(q);
    a.w_r = static_cast<const uint16_t *>(w_r);
    a.v_cache = static_cast<const uint16_t *>(v_cache);
    a.block_table = block_table;
    a.seq_lens = seq_lens;
    a.cu_q = cu_q_lens;
    a.out = out;
    a.out_dtype = out_dtype;
    a.err = err;
    a.stream = reinterpret_cast<cudaStream_t>(stream);
    return from_cuda(launch_prefill_tc(a));
}

}  // extern "C"

namespace {

// The decode geometry over the latent rows (value heads = latent groups, head_dim = r) and the
// workspace carve: q* and o* ([B][Hq][r] fp32 each), then the decode's own workspace.
struct LatentPlan {
    kl_shape dec;
    size_t q_lat, o_lat, dec_ws, total;
};

kl_status latent_plan(const kl_latent_shape *s, int32_t num_splits, LatentPlan *p) {
    if (!s) return KL_ERR_INVALID_ARG;
    if (s->num_seqs < 0 || s->num_q_heads <= 0 || s->num_latent_heads <= 0 || s->head_dim <= 0 ||
        s->latent_dim <= 0)
        return KL_ERR_INVALID_ARG;
    if (s->num_q_heads % s->num_latent_heads != 0) return KL_ERR_INVALID_ARG;
    if (s->latent_dim != 128 || (s->head_dim != 64 && s->head_dim != 128)) return KL_ERR_UNSUPPORTED;
    if (num_splits < 0) return KL_ERR_INVALID_ARG;
    p->dec = kl_shape{s->num_seqs, s->num_q_heads, s->num_latent_heads, s->latent_dim, s->page_size,
                      s->num_pages, s->max_pages_per_seq, 0,
                      s->scale > 0.f ? s->scale : 1.0f / sqrtf((float)s->latent_dim)};
    Geometry g;
    kl_status st = resolve(&p->dec, num_splits, &g);
    if (st != KL_OK) return st;
    if (g.G > 8) return KL_ERR_UNSUPPORTED;
    const size_t rows = (size_t)s->num_seqs * s->num_q_heads * s->latent_dim * sizeof(float);
    // the decode's part first, so that its merge counters sit in the same front region as
    // those of every other decode sharing the workspace (reserved even when S = 1)
    const size_t dec = layout(g).total;
    const size_t floor_bytes = kCounterFloor * sizeof(unsigned int);
    p->dec_ws = 0;
    p->q_lat = round_up(dec > floor_bytes ? dec : floor_bytes, 256);
    p->o_lat = p->q_lat + round_up(rows, 256);
    p->total = p->o_lat + round_up(rows, 256);
    return KL_OK;
}

}  // namespace

extern "C" {

kl_status kl_append_v_fp8(const kl_shape *shape, const void *v_new, const int32_t *block_table,
                          const int32_t *positions, void *v_codes, float *v_scales, int32_t *err,
                          kl_stream_t stream) {
    Geometry g;
    kl_status st = resolve(shape, -1, &g);
    if (st != KL_OK) return st;
    if (g.D != 128) return KL_ERR_UNSUPPORTED;
    if (g.B == 0) return KL_OK;
    if (!v_new || !block_table || !positions || !v_codes || !v_scales) return KL_ERR_INVALID_ARG;
    if (!aligned(v_new, 16) || !aligned(v_codes, 16) || !aligned(v_scales, 16))
        return KL_ERR_INVALID_ARG;
    return from_cuda(launch_append_fp8(g, static_cast<const uint16_t *>(v_new), block_table,
                                       positions, static_cast<uint8_t *>(v_codes), v_scales, err,
                                       reinterpret_cast<cudaStream_t>(stream)));
}

kl_status kl_quantize_cache_fp8(const kl_shape *shape, const void *v_cache, void *v_codes,
                                float *v_scales, kl_stream_t stream) {
    Geometry g;
    kl_status st = resolve(shape, -1, &g);
    if (st != KL_OK) return st;
    if (g.D != 128) return KL_ERR_UNSUPPORTED;
    if (!v_cache || !v_codes || !v_scales) return KL_ERR_INVALID_ARG;
    if (!aligned(v_cache, 16) || !aligned(v_codes, 16) || !aligned(v_scales, 16))
        return KL_ERR_INVALID_ARG;
    const size_t rows = (size_t)g.num_pages * g.Hkv * g.P;
    return from_cuda(launch_quantize_fp8(rows, static_cast<const uint16_t *>(v_cache),
                                         static_cast<uint8_t *>(v_codes), v_scales,
                                         reinterpret_cast<cudaStream_t>(stream)));
}

}  // extern "C"

namespace {

// kl_decode_attention_fp8, with the fused quantizing append of kl_decode_step_fp8 when v_new
// is set.
kl_status decode_fp8(const kl_shape *shape, const void *q, const void *w_r, const void *v_codes,
                     const float *v_scales, const int32_t *block_table, const int32_t *seq_lens,
                     int32_t num_splits, void *out, kl_dtype out_dtype, void *workspace,
                     size_t workspace_bytes, int32_t *err, kl_stream_t stream,
                     const void *v_new, const int32_t *positions) {
    if (num_splits < 0) return KL_ERR_INVALID_ARG;
    if (out_dtype != KL_BF16 && out_dtype != KL_FP32) return KL_ERR_INVALID_ARG;
    Geometry g;
    kl_status st = resolve(shape, num_splits, &g);
    if (st != KL_OK) return st;
    if (g.D != 128 || g.wr_per_qh || !tc_supported(g, false)) return KL_ERR_UNSUPPORTED;
    if (g.P < 4) return KL_ERR_UNSUPPORTED;
    if (g.B == 0) return KL_OK;
    // Runs of splits: when one CTA per split would overflow a wave of two CTAs per SM while the
    // (b, g) units alone would not fill it, each CTA takes the fewest consecutive splits that
    // fit and folds them as it goes (the online softmax continues across the boundary, the
    // associative merge of adjacent states): the split chunk widens by that factor. The split
    // states stay internal to this entry point (merged by the combine kernel).
    {
        const int64_t units = (int64_t)g.B * g.Hkv * g.nhb;
        const int64_t slots = 2 * (int64_t)device_sm_count();
        int spc = 1;
        if (g.S > 1 && units < slots)
            while ((int64_t)((g.S + spc - 1) / spc) * units > slots) ++spc;
        if (spc > 1) {
            const int64_t Lmax = (int64_t)g.max_pages * g.P;
            g.chunk *= spc;
            g.S = (int)((Lmax + g.chunk - 1) / g.chunk);
        }
    }
    if (!q || !v_codes || !v_scales || !block_table || !seq_lens || !out) return KL_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(v_codes, 16) || !aligned(v_scales, 16) || !aligned(out, 16) ||
        (w_r && !aligned(w_r, 16)))
        return KL_ERR_INVALID_ARG;
    const WorkspaceLayout wl = layout(g);
    if (wl.total > 0 && (!workspace || workspace_bytes < wl.total || !aligned(workspace, 256)))
        return KL_ERR_WORKSPACE;
    DecodeArgs a{};
    a.geo = g;
    a.q = static_cast<const uint16_t *>(q);
    a.w_r = static_cast<const uint16_t *>(w_r);
    a.q_routed = nullptr;
    a.k_cache = nullptr;
    a.v_cache = static_cast<const uint16_t *>(v_codes);
    a.block_table = block_table;
    a.seq_lens = seq_lens;
    a.v_new = static_cast<const uint16_t *>(v_new);
    a.positions = positions;
    a.cache_rw = nullptr;
    a.codes_rw = static_cast<uint8_t *>(const_cast<void *>(v_codes));
    a.scales_rw = const_cast<float *>(v_scales);
    char *ws = static_cast<char *>(workspace);
    a.part_o = wl.total ? reinterpret_cast<float *>(ws + wl.part_o) : nullptr;
    a.part_ml = wl.total ? reinterpret_cast<float *>(ws + wl.part_ml) : nullptr;
    a.out = out;
    a.direct_out = g.S == 1;
    a.merge_inside = false;
    a.counters = nullptr;
    a.out_dtype = out_dtype;
    a.err = err;
    a.stream = reinterpret_cast<cudaStream_t>(stream);
    a.wait_ns = current_wait_ns();
    cudaError_t e = launch_decode_fp8(a, v_scales);
    if (e == cudaSuccess) e = finish_decode(a, false);
    return from_cuda(e);
}

}  // namespace

extern "C" {

kl_status kl_decode_attention_fp8(const kl_shape *shape, const void *q, const void *w_r,
                                  const void *v_codes, const float *v_scales,
                                  const int32_t *block_table, const int32_t *seq_lens,
                                  int32_t num_splits, void *out, kl_dtype out_dtype,
                                  void *workspace, size_t workspace_bytes, int32_t *err,
                                  kl_stream_t stream) {
    return decode_fp8(shape, q, w_r, v_codes, v_scales, block_table, seq_lens, num_splits, out,
                      out_dtype, workspace, workspace_bytes, err, stream, nullptr, nullptr);
}

kl_status kl_decode_step_fp8(const kl_shape *shape, const void *q, const void *w_r,
                             const void *v_new, const int32_t *positions, void *v_codes,
                             float *v_scales, const int32_t *block_table, const int32_t *seq_lens,
                             int32_t num_splits, void *out, kl_dtype out_dtype, void *workspace,
                             size_t workspace_bytes, int32_t *err, kl_stream_t stream) {
    if (!v_new || !positions || !aligned(v_new, 16)) return KL_ERR_INVALID_ARG;
    return decode_fp8(shape, q, w_r, v_codes, v_scales, block_table, seq_lens, num_splits, out,
                      out_dtype, workspace, workspace_bytes, err, stream, v_new, positions);
}

size_t kl_latent_workspace_size(const kl_latent_shape *shape, int32_t num_splits) {
    LatentPlan p;
    return latent_plan(shape, num_splits, &p) == KL_OK ? p.total : 0;
}

}  // extern "C"

namespace {

// kl_latent_decode, with the fused append of kl_latent_decode_step when v_new is set.
kl_status latent_decode(const kl_latent_shape *shape, const void *q, const void *w_r,
                        const void *w_post, const void *v_lat, const int32_t *block_table,
                        const int32_t *seq_lens, int32_t num_splits, void *out,
                        kl_dtype out_dtype, void *workspace, size_t workspace_bytes, int32_t *err,
                        kl_stream_t stream, const void *v_new, const int32_t *positions) {
    LatentPlan p;
    kl_status st = latent_plan(shape, num_splits, &p);
    if (st != KL_OK) return st;
    if (out_dtype != KL_BF16 && out_dtype != KL_FP32) return KL_ERR_INVALID_ARG;
    if (shape->num_seqs == 0) return KL_OK;
    if (!q || !w_r || !w_post || !v_lat || !block_table || !seq_lens || !out)
        return KL_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(w_r, 16) || !aligned(w_post, 16) || !aligned(v_lat, 16) ||
        !aligned(out, 16))
        return KL_ERR_INVALID_ARG;
    if (!workspace || workspace_bytes < p.total || !aligned(workspace, 256)) return KL_ERR_WORKSPACE;
    Geometry g;
    resolve(&p.dec, num_splits, &g);
    if (!tc_supported(g, false)) return KL_ERR_UNSUPPORTED;
    char *ws = static_cast<char *>(workspace);
    float *q_lat = reinterpret_cast<float *>(ws + p.q_lat);
    float *o_lat = reinterpret_cast<float *>(ws + p.o_lat);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int B = shape->num_seqs, Hq = shape->num_q_heads, D = shape->head_dim,
              r = shape->latent_dim;
    cudaError_t e = launch_latent_query(B, Hq, Hq / shape->num_latent_heads, D, r,
                                        shape->wr_per_query_head ? 1 : 0,
                                        static_cast<const uint16_t *>(q),
                                        static_cast<const uint16_t *>(w_r),
                                        static_cast<const uint16_t *>(w_post), q_lat, err, s);
    if (e != cudaSuccess) return KL_ERR_CUDA;
    kl_decode_options o{num_splits, KL_KERNEL_TENSOR, nullptr, nullptr};
    st = decode_common(false, &p.dec, nullptr, nullptr, nullptr, v_lat, block_table, seq_lens, &o,
                       o_lat, KL_FP32, ws + p.dec_ws, workspace_bytes - p.dec_ws, err, stream,
                       v_new, positions, q_lat, /*pdl=*/true);
    if (st != KL_OK) return st;
    return from_cuda(launch_latent_expand(B, Hq, D, r, o_lat, static_cast<const uint16_t *>(w_post),
                                          out, out_dtype, err, s));
}

}  // namespace

extern "C" {

kl_status kl_latent_decode(const kl_latent_shape *shape, const void *q, const void *w_r,
                           const void *w_post, const void *v_lat, const int32_t *block_table,
                           const int32_t *seq_lens, int32_t num_splits, void *out,
                           kl_dtype out_dtype, void *workspace, size_t workspace_bytes,
                           int32_t *err, kl_stream_t stream) {
    return latent_decode(shape, q, w_r, w_post, v_lat, block_table, seq_lens, num_splits, out,
                         out_dtype, workspace, workspace_bytes, err, stream, nullptr, nullptr);
}

kl_status kl_latent_decode_step(const kl_latent_shape *shape, const void *q, const void *w_r,
                                const void *w_post, const void *v_new, const int32_t *positions,
                                void *v_lat, const int32_t *block_table, const int32_t *seq_lens,
                                int32_t num_splits, void *out, kl_dtype out_dtype,
                                void *workspace, size_t workspace_bytes, int32_t *err,
                                kl_stream_t stream) {
    if (!v_new || !positions || !aligned(v_new, 16)) return KL_ERR_INVALID_ARG;
    return latent_decode(shape, q, w_r, w_post, v_lat, block_table, seq_lens, num_splits, out,
                         out_dtype, workspace, workspace_bytes, err, stream, v_new, positions);
}

int32_t kl_decode_kernel_available(const kl_shape *shape, int32_t kernel, int32_t standard) {
    Geometry g;
    if (resolve(shape, 1, &g) != KL_OK) return 0;
    const bool tc = tc_supported(g, standard != 0);
    const bool simt = g.G <= kSimtMaxGroup;
    if (kernel == KL_KERNEL_SIMT) return simt ? 1 : 0;
    if (kernel == KL_KERNEL_AUTO) return (tc || simt) ? 1 : 0;
    if (kernel == KL_KERNEL_TENSOR) return tc ? 1 : 0;
    return 0;
}

uint64_t kl_set_wait_timeout_ns(uint64_t ns) {
    const uint64_t old = g_wait_ns.exchange(ns, std::memory_order_relaxed);
    return old ? old : kDefaultWaitNs;
}

const char *kl_status_string(kl_status s) {
    switch (s) {
        case KL_OK: return "ok";
        case KL_ERR_INVALID_ARG: return "invalid argument";
        case KL_ERR_UNSUPPORTED: return "unsupported shape or option";
        case KL_ERR_WORKSPACE: return "workspace missing or too small";
        case KL_ERR_CUDA: return "CUDA error";
    }
    return "unknown status";
}

}  // extern "C"
