/*
 * keyless.h -- C ABI of libkeyless: the decode step of Keyless Attention over a paged
 * Value-Only Cache, as hand-written CUDA for sm_103a (GB300).
 *
 * The method ("Keyless Attention: Value-Space Routing and Value-Only Caching for Efficient
 * Transformers") drops the key projection: a query row is routed into value space by W^R
 * (Section 2.2, Eq. 4) and scored directly against the cached value rows, and the same rows
 * form the output (Section 3, decode formula for O_{n+1}):
 *
 *     q_r      = q W^R
 *     alpha_i  = exp(scale * <q_r, v_i>) / sum_i' exp(scale * <q_r, v_i'>),  i = 1 .. n+1
 *     O_{n+1}  = sum_i alpha_i v_i
 *
 * with MHA / MQA / GQA head sharing as in Section 3: query head h reads value head
 * h / (Hq / Hkv).
 *
 * Conventions for every entry point:
 *   - Pointers are device memory owned by the caller (except `shape` and `opts`, which are
 *     host structs read during the call). The library never allocates, frees or
 *     synchronizes; every launch is asynchronous on `stream` (NULL = legacy default stream).
 *   - bf16 tensors are passed as `const void *` holding IEEE bfloat16 values.
 *   - The return value reports synchronous host-side validation and launch errors; on any
 *     error nothing is launched.
 *   - Data-dependent violations found on the device (a page id outside [0, num_pages), a
 *     position or length beyond max_pages_per_seq * page_size) skip the offending access
 *     and OR a KL_FLAG_* bit into the caller's device word `*err` (which may be NULL to
 *     ignore them). The caller reads `*err` after synchronizing; the kernels never trap.
 *   - Paging follows PagedAttention: token t of sequence b is row t % P of physical page
 *     block_table[b * max_pages_per_seq + t / P]; the value cache is laid out as
 *     [num_pages][Hkv][P][D] bf16, so one (page, head) tile is P * D * 2 contiguous bytes.
 *     Filling the block table (page allocation) is the caller's job.
 */
#ifndef KEYLESS_H
#define KEYLESS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st *kl_stream_t;

typedef enum kl_status {
    KL_OK = 0,
    KL_ERR_INVALID_ARG = 1,  /* null pointer, bad dimension or count */
    KL_ERR_UNSUPPORTED = 2,  /* valid but not implemented (e.g. head_dim not 64 or 128) */
    KL_ERR_WORKSPACE = 3,    /* workspace missing or smaller than kl_decode_workspace_size */
    KL_ERR_CUDA = 4          /* a CUDA runtime call or launch failed */
} kl_status;

/* Bits OR-ed into the device error word. */
#define KL_FLAG_BAD_PAGE 0x1     /* block-table entry outside [0, num_pages) */
#define KL_FLAG_BAD_POSITION 0x2 /* append position outside [0, max_pages_per_seq * P) */
#define KL_FLAG_BAD_LENGTH 0x4   /* seq_len outside [0, max_pages_per_seq * P] */
#define KL_FLAG_TIMEOUT 0x8      /* a bounded pipeline wait gave up (output invalid) */
#define KL_FLAG_RANGE 0x10       /* a non-finite output of kl_prefill_attention (a cached value
                                    beyond its fp16 range, or a non-finite input) */

typedef enum kl_dtype { KL_BF16 = 0, KL_FP32 = 1 } kl_dtype;

typedef struct kl_shape {
    int32_t num_seqs;          /* B */
    int32_t num_q_heads;       /* Hq */
    int32_t num_kv_heads;      /* Hkv, the value heads; Hq % Hkv == 0, G = Hq / Hkv */
    int32_t head_dim;          /* D = d_k; 64 or 128 */
    int32_t page_size;         /* P tokens per page */
    int32_t num_pages;         /* pages in the cache pool */
    int32_t max_pages_per_seq; /* block-table row stride */
    int32_t wr_per_query_head; /* 0: W^R holds Hkv matrices (index h / G); 1: Hq matrices (index h) */
    float scale;               /* lambda / sqrt(d_k); <= 0 selects 1 / sqrt(head_dim) (lambda = 1) */
} kl_shape;

/* Kernel family of the decode. */
typedef enum kl_kernel {
    KL_KERNEL_AUTO = 0,   /* tensor-core kernel where supported, else the CUDA-core one */
    KL_KERNEL_TENSOR = 1, /* tcgen05 + TMA kernel (head_dim 128 or 64; a group of more than 8
                           * query heads is served by CTAs of up to 8 heads each, group size
                           * <= 128) */
    KL_KERNEL_SIMT = 2    /* CUDA-core kernel (group size <= 8) */
} kl_kernel;

typedef struct kl_decode_options {
    int32_t num_splits; /* split-sequence count S; 0 = chosen from the shape and the GPU */
    int32_t kernel;     /* kl_kernel */
    /* Optional split-state outputs. When both are non-NULL the decode writes every split's
     * state there -- partial_o [B][Hq][S][D] fp32 (normalized) and partial_ml [B][Hq][S][2]
     * fp32 ({m, l}, the layout kl_combine reads) -- and neither merges nor writes `out`
     * (which may be NULL); no workspace is needed. This exposes the states for a later
     * kl_combine, e.g. after gathering the states of sequence shards from several devices.
     * Split s holds tokens [s C, (s + 1) C) of every sequence, C = ceil(max_pages_per_seq * P
     * / S) rounded up to a multiple of 128, with S = kl_decode_num_splits(shape, num_splits);
     * a split past a sequence's end has m = -inf, l = 0 and a zero row. m is the split's largest
     * score (natural-log units, scale included) and l = sum_t exp(s_t - m). */
    float *partial_o;
    float *partial_ml;
} kl_decode_options;

/*
 * Routing projection (Section 2.2, Eq. 4; the composed query of Eq. 2):
 *   q_r[b][h][j] = sum_k q[b][h][k] * W^R[w(h)][k][j],   fp32 accumulation.
 * q: [B][Hq][D] bf16. w_r: [Hw][D][D] bf16 row-major (row k = input dimension), Hw = Hkv
 * (w(h) = h / G) or Hq (w(h) = h) per shape->wr_per_query_head. q_r: [B][Hq][D] fp32 out.
 */
kl_status kl_route_query(const kl_shape *shape, const void *q, const void *w_r, float *q_r,
                         kl_stream_t stream);

/*
 * Value-Only Cache append (Section 3: the cache holds the value rows of earlier steps and the
 * row obtained at the current step; no key row is stored):
 *   v_cache[block_table[b][pos_b / P]][g][pos_b % P][:] = v_new[b][g][:]   for all b, g,
 * with pos_b = positions[b]. v_new: [B][Hkv][D] bf16; positions: [B] int32; v_cache is
 * written in place (bit copy). A position outside [0, max_pages_per_seq * P) or a page id
 * outside the pool skips that sequence and raises KL_FLAG_BAD_POSITION / KL_FLAG_BAD_PAGE.
 */
kl_status kl_append_v(const kl_shape *shape, const void *v_new, const int32_t *block_table,
                      const int32_t *positions, void *v_cache, int32_t *err,
                      kl_stream_t stream);

/*
 * Bytes of device workspace kl_decode_attention / kl_decode_step / kl_standard_decode need for
 * `num_splits` (0 = the automatic choice); 0 when no workspace is needed (one split). Returns
 * 0 on invalid shapes. The workspace holds, for the tensor-core kernel, one merge counter per
 * sequence, value head and block of up to 8 of its query heads, then the split states. It must
 * be zero-filled (cudaMemsetAsync) before its first use; every call leaves its counters at zero
 * again. The counters occupy a fixed front region of 64 KiB for every shape with at most 16384
 * of them (larger shapes extend it), where no split state is ever written, so the workspace
 * serves any sequence of calls and shapes -- batch sizes and split counts that change from
 * call to call included -- except after a call that raised KL_FLAG_TIMEOUT, which may leave
 * counters behind, or a switch from a shape with more than 16384 counters: zero the workspace
 * again then. Calls that share a workspace must not overlap on the GPU.
 */
size_t kl_decode_workspace_size(const kl_shape *shape, int32_t num_splits);

/* The split count that `num_splits` (0 = automatic) resolves to for this shape. */
int32_t kl_decode_num_splits(const kl_shape *shape, int32_t num_splits);

/*
 * Keyless decode attention over the paged Value-Only Cache (Section 3, decode formula for
 * O_{n+1}; MHA/MQA/GQA head sharing; the routing projection of Section 2.2 is fused into the
 * kernel's prologue). For every sequence b and query head h:
 *   q_r = q[b][h] W^R[w(h)],  s_t = scale * <q_r, v_t>,  out[b][h] = sum_t softmax(s)_t v_t,
 * over the L_b = seq_lens[b] cached rows t = 0 .. L_b - 1 (the current token's row included,
 * i.e. append first). L_b = 0 writes zeros.
 * q: [B][Hq][D] bf16; w_r: [Hw][D][D] bf16; v_cache: [num_pages][Hkv][P][D] bf16;
 * block_table: [B][max_pages_per_seq] int32; seq_lens: [B] int32; out: [B][Hq][D] of
 * `out_dtype`. The sequence is cut into `num_splits` chunks processed in parallel and merged
 * as in kl_combine (by the last chunk of each sequence to finish, or by a second kernel);
 * `workspace` must hold kl_decode_workspace_size(shape, num_splits) bytes (256-byte aligned,
 * zero-filled before its first use). A bad page id or length raises its flag and leaves that
 * output unspecified.
 * w_r == NULL selects the composed-query form of Section 2.1: at inference W^Q W^R is one
 * precomputed projection, so q already is the routed query (q = x W^Q W^R) and is used as q_r
 * directly (no routing in the kernel). The same holds for every decode entry point below.
 */
kl_status kl_decode_attention(const kl_shape *shape, const void *q, const void *w_r,
                              const void *v_cache, const int32_t *block_table,
                              const int32_t *seq_lens, int32_t num_splits, void *out,
                              kl_dtype out_dtype, void *workspace, size_t workspace_bytes,
                              int32_t *err, kl_stream_t stream);

/*
 * One whole decode step in one pass: the Value-Only Cache append of the current token
 * (Section 3: V holds the rows of the earlier steps and the row obtained at the current step)
 * followed by the keyless decode over the n+1 rows, i.e. kl_append_v then
 * kl_decode_attention_ex, fused: the decode CTA whose split holds row positions[b] writes
 * v_new[b][g] there before reading it, so the new row never makes a separate round trip.
 * v_new: [B][Hkv][D] bf16; positions: [B] int32 (normally seq_lens[b] - 1); v_cache is
 * written in place. Other arguments, layouts and flags as in kl_append_v and
 * kl_decode_attention_ex.
 */
kl_status kl_decode_step(const kl_shape *shape, const void *q, const void *w_r,
                         const void *v_new, const int32_t *positions, void *v_cache,
                         const int32_t *block_table, const int32_t *seq_lens,
                         const kl_decode_options *opts, void *out, kl_dtype out_dtype,
                         void *workspace, size_t workspace_bytes, int32_t *err,
                         kl_stream_t stream);

/* kl_decode_attention with an explicit kernel choice (opts may be NULL = defaults). */
kl_status kl_decode_attention_ex(const kl_shape *shape, const void *q, const void *w_r,
                                 const void *v_cache, const int32_t *block_table,
                                 const int32_t *seq_lens, const kl_decode_options *opts,
                                 void *out, kl_dtype out_dtype, void *workspace,
                                 size_t workspace_bytes, int32_t *err, kl_stream_t stream);

/*
 * Merge of split states into one softmax (the decode formula's normalization applied over
 * the union of the splits). For every (b, h), with split s holding its normalized output
 * o_s = partial_o[b][h][s][:] and {m_s, l_s} = partial_ml[b][h][s][0..1] (m_s = largest
 * score of the split, l_s = sum over the split of exp(s_t - m_s); l_s = 0 marks an empty
 * split):
 *   M = max_{l_s > 0} m_s,  w_s = l_s exp(m_s - M),  out[b][h] = sum_s w_s o_s / sum_s w_s.
 * All splits empty writes zeros. partial_o: [B][Hq][S][D] fp32; partial_ml: [B][Hq][S][2]
 * fp32; out: [B][Hq][D] of out_dtype. Used inside kl_decode_attention and, across devices,
 * to merge the states of sequence shards.
 */
kl_status kl_combine(const kl_shape *shape, const float *partial_o, const float *partial_ml,
                     int32_t num_splits, void *out, kl_dtype out_dtype, kl_stream_t stream);

/*
 * Comparison only: standard decode attention softmax(q K^T * scale) V (Eq. 1) over a paged
 * key cache and a paged value cache of the same layout -- the K+V cache a Value-Only Cache
 * replaces, read by a kernel of the same design. q is used as given (no routing).
 * Arguments as in kl_decode_attention_ex with k_cache added.
 */
kl_status kl_standard_decode(const kl_shape *shape, const void *q, const void *k_cache,
                             const void *v_cache, const int32_t *block_table,
                             const int32_t *seq_lens, const kl_decode_options *opts, void *out,
                             kl_dtype out_dtype, void *workspace, size_t workspace_bytes,
                             int32_t *err, kl_stream_t stream);

/*
 * Chunk append, the prefill counterpart of kl_append_v: sequence b's chunk of
 * n_b = cu_q_lens[b + 1] - cu_q_lens[b] new tokens takes the last n_b of its seq_lens[b] rows,
 *   v_cache[block_table[b][p / P]][g][p % P][:] = v_new[cu_q_lens[b] + i][g][:],
 *   p = seq_lens[b] - n_b + i,  0 <= i < n_b,  all g.
 * v_new: [total_q][Hkv][D] bf16 (total_q = cu_q_lens[B]); cu_q_lens: [B + 1] int32 on the
 * device, non-decreasing from 0; max_q_len: a host-side bound on every n_b (it sizes the grid;
 * rows past it are not written). A length that breaks 0 <= n_b <= seq_lens[b] <=
 * max_pages_per_seq * P raises KL_FLAG_BAD_LENGTH and skips the sequence; a page id outside the
 * pool raises KL_FLAG_BAD_PAGE and skips that row.
 */
kl_status kl_append_v_chunk(const kl_shape *shape, const void *v_new, const int32_t *block_table,
                            const int32_t *seq_lens, const int32_t *cu_q_lens, int32_t total_q,
                            int32_t max_q_len, void *v_cache, int32_t *err, kl_stream_t stream);

/*
 * Chunked keyless prefill: the full attention of Eq. 3 for a chunk of new tokens under the
 * causal mask of an autoregressive model (Section 5), over the paged Value-Only Cache, with
 * the routing projection of Section 2.2 fused into the kernel. Sequence b's chunk is its last
 * n_b = cu_q_lens[b + 1] - cu_q_lens[b] cached rows (append them first, kl_append_v_chunk);
 * query row r = cu_q_lens[b] + i sits at position p = seq_lens[b] - n_b + i and, per query
 * head h,
 *   q_r = q[r][h] W^R[w(h)],  s_t = scale * <q_r, v_t> (t = 0 .. p),
 *   out[r][h] = sum_t softmax(s)_t v_t.
 * A whole prompt is the case n_b = seq_lens[b]; a decode step is n_b = 1.
 * q, out: [total_q][Hq][D] (q bf16, out of out_dtype); w_r, v_cache, block_table as in
 * kl_decode_attention; cu_q_lens: [B + 1] int32 on the device; max_q_len: a host-side bound on
 * every n_b (it sizes the grid; rows past it get no output). head_dim 128 only
 * (KL_ERR_UNSUPPORTED otherwise). Needs no workspace. Flags as in kl_append_v_chunk, and a bad
 * page id leaves the affected outputs unspecified. Precision: the scores are formed from the
 * bf16 cache rows with the routed query carried to about 16 significant bits; the output sum
 * takes the softmax weights and the cached values in fp16 (exact for bf16 values of magnitude
 * 2^-14 to 65280, smaller ones to within 2^-25). A cached value of magnitude 65536 or more has
 * no finite fp16 form: the outputs of the query rows whose 128-token cache tiles hold it come
 * out non-finite, and any non-finite output raises KL_FLAG_RANGE.
 */
kl_status kl_prefill_attention(const kl_shape *shape, const void *q, const void *w_r,
                               const void *v_cache, const int32_t *block_table,
                               const int32_t *seq_lens, const int32_t *cu_q_lens,
                               int32_t total_q, int32_t max_q_len, void *out, kl_dtype out_dtype,
                               int32_t *err, kl_stream_t stream);

/*
 * Shape of a decode over a latent value-only cache (Section 3, "Multihead with Latent Value-only
 * Cache"): the cache holds V* = X W^V_pre, latent_dim (r) wide, one latent row per token and
 * latent group; query head h reads latent group h / (num_q_heads / num_latent_heads) and
 * expands it with its own W^V_{h,post} (r x head_dim).
 */
typedef struct {
    int32_t num_seqs;            /* B */
    int32_t num_q_heads;         /* Hq */
    int32_t num_latent_heads;    /* Hl: latent groups (1 = one latent shared by every head) */
    int32_t head_dim;            /* D: width of q, W^R and the output (64 or 128) */
    int32_t latent_dim;          /* r: width of the cached latent rows (128) */
    int32_t page_size;           /* P */
    int32_t num_pages;           /* latent pool size */
    int32_t max_pages_per_seq;   /* block_table row stride */
    int32_t wr_per_query_head;   /* W^R: Hq matrices (1) or Hl matrices (0) */
    float scale;                 /* <= 0: 1 / sqrt(latent_dim), the paper's 1/sqrt(r) */
} kl_latent_shape;

/* Bytes of device workspace kl_latent_decode needs for `num_splits` (0 = automatic); 0 on an
 * invalid or unsupported shape. Same zero-fill contract as kl_decode_workspace_size (its merge
 * counters sit in the same front region). */
size_t kl_latent_workspace_size(const kl_latent_shape *shape, int32_t num_splits);

/*
 * Keyless decode over a latent value-only cache (Section 3): for every sequence b and query
 * head h of latent group g,
 *   q*  = (q[b][h] W^R[w(h)]) W_post[h]^T          (the absorbed query, width r)
 *   o*  = sum_t softmax(scale <q*, v*_t>)_t v*_t    (over the L_b cached latent rows)
 *   out[b][h] = o* W_post[h]                         (width D)
 * q: [B][Hq][D] bf16; w_r: [Hw][D][D] bf16; w_post: [Hq][r][D] bf16 row-major (row k = latent
 * dimension); v_lat: [num_pages][Hl][P][r] bf16 (append with kl_append_v and a kl_shape whose
 * num_kv_heads = Hl and head_dim = r); block_table, seq_lens, num_splits, out, workspace and
 * flags as in kl_decode_attention. Three launches on `stream`: the absorbed queries, the
 * tensor-core decode over the latent rows, the expansion. latent_dim 128 and compute
 * capability 10.3 only (KL_ERR_UNSUPPORTED otherwise); at most 8 query heads per latent group.
 */
kl_status kl_latent_decode(const kl_latent_shape *shape, const void *q, const void *w_r,
                           const void *w_post, const void *v_lat, const int32_t *block_table,
                           const int32_t *seq_lens, int32_t num_splits, void *out,
                           kl_dtype out_dtype, void *workspace, size_t workspace_bytes,
                           int32_t *err, kl_stream_t stream);

/*
 * One decode step over a latent value-only cache: the current token's latent rows are appended
 * (Section 3: the cache holds every row up to the current one) and the decode of
 * kl_latent_decode runs over the n+1 rows -- kl_append_v into v_lat then kl_latent_decode,
 * fused: the decode CTA whose split holds row positions[b] writes v_new[b][g] there before it
 * reads that row. v_new: [B][Hl][r] bf16, 16-byte aligned; positions: [B] int32 (normally
 * seq_lens[b] - 1); v_lat is written in place. A position outside the block table raises
 * KL_FLAG_BAD_POSITION and a page id outside the pool KL_FLAG_BAD_PAGE in *err (that row is not
 * written). Other arguments, layouts, workspace and flags as in kl_latent_decode.
 */
kl_status kl_latent_decode_step(const kl_latent_shape *shape, const void *q, const void *w_r,
                                const void *w_post, const void *v_new, const int32_t *positions,
                                void *v_lat, const int32_t *block_table, const int32_t *seq_lens,
                                int32_t num_splits, void *out, kl_dtype out_dtype,
                                void *workspace, size_t workspace_bytes, int32_t *err,
                                kl_stream_t stream);

/*
 * FP8 value cache (not in the paper; §3 notes that the value-only cache is orthogonal to other
 * cache-reduction methods, and a quantized cache is one): the same value rows stored in about
 * half the bytes. Each cached row is D OCP FP8 E4M3 codes (1 sign, 4 exponent bits of bias 7,
 * 3 mantissa bits; subnormals m/8 * 2^-6; largest finite value 448) and one fp32 scale, the
 * row's values being scale * value(code):
 *   codes: [num_pages][Hkv][P][D] uint8,   scales: [num_pages][Hkv][P] fp32,
 * both caller-owned device memory, 16-byte aligned (KL_ERR_INVALID_ARG otherwise). head_dim 128
 * only (KL_ERR_UNSUPPORTED otherwise). The library never writes the code 0x7F / 0xFF (NaN); a
 * cache holding them yields NaN outputs.
 *
 * kl_append_v_fp8: quantize v_new[b][g] (bf16, [B][Hkv][D]) into row positions[b] of sequence
 * b -- scale = max |v| / 448 in fp32, code_j = E4M3(v_j / scale) rounded to nearest even and
 * saturating (an all-zero row gets scale 0 and zero codes). A position outside the block table
 * raises KL_FLAG_BAD_POSITION, a page id outside the pool KL_FLAG_BAD_PAGE, in *err; that row is
 * skipped.
 */
kl_status kl_append_v_fp8(const kl_shape *shape, const void *v_new, const int32_t *block_table,
                          const int32_t *positions, void *v_codes, float *v_scales, int32_t *err,
                          kl_stream_t stream);

/* Quantize a whole bf16 value cache [num_pages][Hkv][P][128] (caller-owned device memory,
 * 16-byte aligned) into the FP8 layout, row by row, with the arithmetic of kl_append_v_fp8 (e.g.
 * to move an existing cache to FP8). The results are bit-identical to appending every row. */
kl_status kl_quantize_cache_fp8(const kl_shape *shape, const void *v_cache, void *v_codes,
                                float *v_scales, kl_stream_t stream);

/*
 * kl_decode_attention_fp8: the keyless decode of kl_decode_attention (routing §2.2, one softmax
 * over the cached value rows, each row serving score and output, §3) over the FP8 cache, each
 * cached value being scale * value(code). On the tensor cores with E4M3 products straight on
 * the stored codes and fp32 accumulation; the routed query and the softmax weights enter as
 * sums of E4M3 terms (4 and 3 terms, about 16 and 12 significant bits), each row's scale
 * multiplies its score and its weight. W^R per value head (wr_per_query_head = 0) or
 * w_r == NULL (q is then the composed query); a group of more than 8 query heads is served by
 * CTAs of up to 8 heads each (group size <= 128); page size
 * 16, 32, 64 or 128; compute capability 10.3 (KL_ERR_UNSUPPORTED otherwise). q, w_r, out,
 * num_splits, the workspace (kl_decode_workspace_size of the same shape and split count), the
 * output layout and the error flags are those of kl_decode_attention; with more than one split
 * the split states are merged by the combine kernel in a second launch on the same stream.
 * Returns after enqueueing; nothing is allocated or synchronized.
 */
kl_status kl_decode_attention_fp8(const kl_shape *shape, const void *q, const void *w_r,
                                  const void *v_codes, const float *v_scales,
                                  const int32_t *block_table, const int32_t *seq_lens,
                                  int32_t num_splits, void *out, kl_dtype out_dtype,
                                  void *workspace, size_t workspace_bytes, int32_t *err,
                                  kl_stream_t stream);

/*
 * One decode step over the FP8 cache: kl_append_v_fp8 of the current token's rows followed by
 * kl_decode_attention_fp8 over the n+1 rows, fused -- the decode CTA whose split holds row
 * positions[b] quantizes v_new[b][g] (bit-identical to kl_append_v_fp8) into the code and scale
 * caches before it loads that row. v_new: [B][Hkv][D] bf16, 16-byte aligned; positions: [B]
 * int32 (normally seq_lens[b] - 1); v_codes and v_scales are written in place. Flags as in
 * kl_append_v_fp8 (that row is then not written) and kl_decode_attention_fp8; other arguments
 * as in kl_decode_attention_fp8.
 */
kl_status kl_decode_step_fp8(const kl_shape *shape, const void *q, const void *w_r,
                             const void *v_new, const int32_t *positions, void *v_codes,
                             float *v_scales, const int32_t *block_table, const int32_t *seq_lens,
                             int32_t num_splits, void *out, kl_dtype out_dtype, void *workspace,
                             size_t workspace_bytes, int32_t *err, kl_stream_t stream);

/* Size of the fixed device scratch that kl_decode_attention_noalloc uses (32 MiB). */
#define KL_NOALLOC_SCRATCH_BYTES (32u * 1024u * 1024u)

/*
 * kl_decode_attention without a workspace argument, for callers that must not allocate device
 * memory -- for example code running inside a host framework that owns all device memory
 * through its own pool and does not let its plugins call cudaMalloc, or a latency-critical
 * path that cannot afford an allocation's implicit synchronization and unpredictable cost.
 * The paper has no counterpart: this is a deployment convenience of the library.
 * The split states live in one fixed array of KL_NOALLOC_SCRATCH_BYTES in device memory,
 * which every GPU that loads the library holds until the process exits. The library looks
 * up that array's device address during the first call on each device (with that device
 * current); make that first call before any stream capture. The address belongs to the CUDA
 * context it was looked up in: the library records that context's unique id and looks the
 * address up again when a call finds a different context current on the device (after
 * cudaDeviceReset, for instance), so that call too is a first call. Nothing is allocated and no
 * allocating routine is called. Every call on a device shares the one array and leaves its
 * contents behind, so calls that may overlap on the GPU (different streams, or different
 * host threads without ordering) race and must be serialized by the caller. A shape and
 * split count whose split states need more than KL_NOALLOC_SCRATCH_BYTES is rejected with
 * KL_ERR_WORKSPACE before anything is launched (num_splits = 1 needs no scratch). Other
 * arguments, results and error flags are those of kl_decode_attention.
 */
kl_status kl_decode_attention_noalloc(const kl_shape *shape, const void *q, const void *w_r,
                                      const void *v_cache, const int32_t *block_table,
                                      const int32_t *seq_lens, int32_t num_splits, void *out,
                                      kl_dtype out_dtype, int32_t *err, kl_stream_t stream);

/*
 * Whether kernel family `kernel` (kl_kernel) handles this shape: 1 yes, 0 no. For the keyless
 * decode (standard = 0) or the K+V comparison (standard = 1). A capability query of the
 * library; the paper has no counterpart.
 */
int32_t kl_decode_kernel_available(const kl_shape *shape, int32_t kernel, int32_t standard);

/*
 * Failure detection of the decodes: every wait of a tensor-core decode CTA on its own pipeline
 * (a copy landing, an MMA finishing, another role's hand-off) gives up after a time limit, about
 * one second by default. A CTA whose wait runs out raises KL_FLAG_TIMEOUT, leaves its loops,
 * waits (with the full default bound) for the copies and MMAs it has in flight, frees its tensor
 * memory and exits, so that the call returns and the context stays usable; its outputs are then
 * undefined, and a workspace it used must be zero-filled again before the next call. This sets
 * that limit, in nanoseconds, for every decode launched afterwards by kl_decode_attention(_ex),
 * kl_decode_step, kl_standard_decode, kl_decode_attention_noalloc, the latent decodes and the FP8
 * decodes, process-wide; 0 restores the default. Returns the limit in force before the call. A
 * small value makes the waits run out on purpose: this is how the timeout path is tested. The
 * paper has no counterpart.
 */
uint64_t kl_set_wait_timeout_ns(uint64_t ns);

/* Static description of a status code. */
const char *kl_status_string(kl_status status);

#ifdef __cplusplus
}
#endif

#endif /* KEYLESS_H */
