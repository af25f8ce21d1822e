/*
 * jfkv.h -- C ABI of the GB300 paged 4-bit KV library (libjfkv.so).
 *
 * The library implements the data-parallel hot path of KVExec (Sec. 3.1 and
 * Sec. 3.4 of "JustFit: Just-in-Time State Management for Local LLM Serving"):
 * attention that reads a paged, 4-bit quantized KV cache directly, with a
 * temporary workspace whose size never depends on the history length, plus
 * the quantize-on-append and page-gather checkpoint operations that produce
 * and persist those pages.
 *
 * Conventions for every entry point
 *   - All array pointers are DEVICE pointers owned by the caller.  The library
 *     never allocates, frees or synchronizes; it only enqueues kernels on
 *     `stream` (a cudaStream_t passed as void*, NULL = legacy default stream).
 *   - Return value: JF_OK (0) or a negative JF_ERR_* code.  Arguments are
 *     validated on the host before anything is launched; on an error nothing
 *     is enqueued.  JF_ERR_CUDA means a launch was refused by the runtime.
 *   - Inconsistencies only visible on the device (a page id outside the pool,
 *     a position beyond the page table) never trap: the kernel skips the
 *     affected work and ORs a JF_DEV_* bit into a device status word
 *     (`err_flag`, or the first int32 of `workspace`), which the caller reads
 *     after the stream completes.
 *   - bf16 means IEEE bfloat16 bit patterns (uint16), row-major, contiguous.
 *
 * KV pool formats.  JF_FMT_AFFINE4_G64 (the paper defines TQ4 for KV and only
 * mentions affine Q4 groups for weights, so the affine group layout below is
 * this library's reading) and JF_FMT_TQ4 (documented with jf_tq4_codec):
 *   page record = [K codes: Hkv x P x D/2 bytes][V codes: same]
 *                 [K scale/bias: Hkv x P x D/64 x (bf16 scale, bf16 bias)]
 *                 [V scale/bias: same]
 *   Within a code row, element 2i is the low nibble of byte i (eight 4-bit
 *   indices per little-endian 32-bit word, App. A.1 Table 3).  A 64-element
 *   group reconstructs as x = code * scale + bias.
 *   page_bytes = 2*Hkv*P*(D/2 + 4*D/64); for Hkv 4, P 256, D 256 that is
 *   294,912 bytes, i.e. 1,152 bytes per position per layer (the affine-g64
 *   analogue of Eq. 2's 16,640 bytes per position over 16 layers for TQ4).
 */
#ifndef JFKV_H
#define JFKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes --------------------------------------------------- */
#define JF_OK                       0
#define JF_ERR_INVALID_ARG         (-1)
#define JF_ERR_UNSUPPORTED         (-2)
#define JF_ERR_WORKSPACE_TOO_SMALL (-3)
#define JF_ERR_CUDA                (-4)

/* ---- device status bits (ORed into err_flag / workspace word 0) ------- */
#define JF_DEV_ERR_PAGE_ID    1   /* page id < 0 or >= num_pages          */
#define JF_DEV_ERR_POSITION   2   /* position beyond the page-table row, or
                                     a request index out of range          */
#define JF_DEV_ERR_TIMEOUT    4   /* a bounded wait on a copy gave up      */
#define JF_DEV_ERR_RANGE     16   /* prefill met an affine K/V group whose
                                     fp16 reconstruction can overflow
                                     (|bias| + 15 scale >= 65504, or a
                                     non-finite scale/bias word): outputs
                                     reading it are not reliable           */
#define JF_DEV_ERR_LAYOUT     8   /* the kernel's dynamic shared-memory
                                     window was not 1024-byte aligned (the
                                     swizzled copies need it); the CTA did
                                     no work                               */

/* ---- formats -------------------------------------------------------- */
#define JF_FMT_AFFINE4_G64 0      /* affine 4-bit, 64-element groups (above) */
#define JF_FMT_TQ4         1      /* TQ4 (Sec. 3.1 Eq. 4), see below         */

/*
 * TQ4 format (Sec. 3.1 Eq. 4; App. A.1 Table 3).  A vector x of D elements is
 * stored as D 4-bit indices z into 16 shared centroids c and one fp16 norm:
 *   rho   = fp32 rounding of ||x||_2 (from the fp64 sum of squares),
 *   u     = H_D S x   (H_D the unnormalized Sylvester Hadamard matrix,
 *                      H[i][j] = (-1)^popcount(i & j); S = diag(signs)),
 *   z_j   = #{k in 0..14 : u_j > fp64(fp64(sqrt(D) rho) t_k)},
 *           t_k = fp32(fp32(c_k + c_{k+1}) * 0.5)   (midpoints, strict >),
 *   norm  = fp16 round-to-nearest of min(rho, 65504),
 * and reconstructs as x_hat = norm S H_D c[z] / sqrt(D).  Indices are exact
 * (bit for bit with the reference definition) for bf16 vectors whose
 * nonzero magnitudes span less than 2^37 and whose norm lies in [1e-30, 1e36].
 *   page record = [K indices: Hkv x P x D/2 bytes][V indices: same]
 *                 [K norms: Hkv x P x fp16][V norms: same]
 *   Index j of a vector is nibble j % 8 of little-endian 32-bit word j / 8
 *   (element 2i in the low nibble of byte i).  page_bytes = 2*Hkv*P*(D/2 + 2):
 *   1,040 bytes per position per layer at Hkv 4, D 256, i.e. Eq. 2's 16,640
 *   bytes over 16 layers.
 */
typedef struct jf_tq4_codec {
  float  centroids[16];   /* strictly ascending, |c| < 1 (jf_tq4_codebook)  */
  int8_t signs_k[256];    /* diagonal of S for K: +1 or -1, first D used    */
  int8_t signs_v[256];    /* diagonal of S for V                            */
} jf_tq4_codec;

typedef struct jf_kv_pool {
  void*   base;          /* device pointer to num_pages page records,
                            16-byte aligned                                */
  int64_t num_pages;     /* >= 1                                           */
  int32_t page_size;     /* P: 64, 128 or 256 positions                    */
  int32_t num_kv_heads;  /* Hkv >= 1                                       */
  int32_t head_dim;      /* D: 128 or 256                                  */
  int32_t group_size;    /* 64 (affine format; ignored for TQ4)            */
  int32_t format;        /* JF_FMT_AFFINE4_G64 or JF_FMT_TQ4               */
  const jf_tq4_codec* tq4;  /* host pointer, read during each call;
                               required for JF_FMT_TQ4, else ignored       */
} jf_kv_pool;

/* Bytes of one affine page record (0 if the geometry is unsupported). */
size_t jf_kv_page_bytes(int32_t num_kv_heads, int32_t page_size, int32_t head_dim);

/* Bytes of one page record of the given format (0 if unsupported). */
size_t jf_kv_page_bytes_fmt(int32_t format, int32_t num_kv_heads, int32_t page_size,
                            int32_t head_dim);

/*
 * TQ4 codebook for head dimension head_dim (App. A.1 Table 3), on the host:
 * the 16 fp32 Lloyd-Max centroids of the density (1 - x^2)^((head_dim-3)/2)
 * on [-1, 1], from a 32,768-point grid over [-1 + 1e-6, 1 - 1e-6], quantile
 * start (the first grid point whose cumulative weight reaches (k + 1/2)/16),
 * at most 100 updates (cells by midpoints with strict >, centroid = weighted
 * cell mean, empty cells kept), stopping after the update whose largest
 * change is below 1e-6; computed in fp64 and rounded to fp32.
 *   centroids  host float[16], written in ascending order
 * Returns JF_ERR_INVALID_ARG for head_dim outside [3, 65536] or a NULL pointer.
 */
int jf_tq4_codebook(int32_t head_dim, float* centroids);

/*
 * Workspace bytes jf_paged_decode_attn needs for at most `num_splits`
 * splits per (request, KV head): 256 + roundup(8*B*Hq*S, 256) + 4*B*Hq*S*D
 * bytes (status word, per-split (max, sum) pairs, per-split outputs).  The size
 * depends on batch, heads, splits and head_dim only, never on the context
 * length (Sec. 2, Eq. 3 is the paper's argument for bounding temporaries).
 * Returns 0 for invalid arguments.
 */
size_t jf_attn_workspace_bytes(int32_t batch, int32_t num_q_heads, int32_t num_kv_heads,
                               int32_t head_dim, int32_t num_splits);

/* Workspace bytes jf_prefill_chunk_attn needs (a status word). */
size_t jf_prefill_workspace_bytes(void);

/*
 * Quantize-on-append (Sec. 3.3 "pending cache writes"; Sec. 2 paged pool).
 *
 * For each row i < n_rows, the bf16 vectors k[i, h, :] and v[i, h, :]
 * (layout [n_rows, Hkv, D]) are quantized per 64-element group --
 *   bias  = group minimum (-0 stored as +0),
 *   scale = bf16_rne(fp32(max - min) / 15)            (IEEE, no FMA),
 *   code  = #{k in 0..14 : fp32(x - bias) / scale > k + 1/2}, 0 if scale == 0
 *   (midpoint thresholds with strict >, App. A.1 Table 3) --
 * and written to slot row_pos[i] % P of physical page
 * page_table[row_req[i] * pt_stride + row_pos[i] / P].
 *   page_table  int32 [num_requests, pt_stride]
 *   row_req     int32 [n_rows], 0 <= row_req[i] < num_requests
 *   row_pos     int32 [n_rows], 0 <= row_pos[i] < pt_stride * P
 *   k, v        bf16 [n_rows, Hkv, D], 16-byte aligned
 *   err_flag    device int32 or NULL; JF_DEV_* bits are ORed into it for
 *               rows that were skipped.
 * Rows must not target the same slot twice in one call (the result of such
 * a call is one of the rows, unspecified which).  n_rows == 0 is a no-op.
 * TQ4 pools: each vector is encoded as the TQ4 format block above states
 * (indices and norm), with the codec in pool->tq4.
 */
int jf_kv_quantize_append(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                          int32_t num_requests, const int32_t* row_req, const int32_t* row_pos,
                          const void* k, const void* v, int32_t n_rows, int32_t* err_flag,
                          void* stream);

/*
 * Paged decode attention, one query token per request (Sec. 3.1: the decode
 * kernel reads compressed pages where they are used; Eq. 5 head grouping).
 *
 *   out[b, h, :] = sum_t softmax_t(softmax_scale * <q[b, h], K_t>) V_t
 * over logical positions t < context_lens[b] of request b, with KV head
 * floor(h / (Hq / Hkv)) and K_t, V_t reconstructed from the page named by
 * page_table[b * pt_stride + t / P].  context_lens counts positions already
 * appended, the current token included.  A zero context gives a zero output.
 *
 *   page_table    int32 [batch, pt_stride]
 *   context_lens  int32 [batch], 0 <= ctx <= pt_stride * P
 *   q             bf16 [batch, Hq, D];   out: bf16 [batch, Hq, D]
 *   Hq % Hkv == 0 and Hq / Hkv <= 8.
 *   workspace     device buffer of >= jf_attn_workspace_bytes(batch, Hq,
 *                 Hkv, D, num_splits) bytes, 256-byte aligned.  Its first
 *                 int32 is the device status word (JF_DEV_* bits, ORed);
 *                 the caller zeroes it when it wants a fresh status.
 *   num_splits    >= 1: split-K partitions per (request, KV head) that the
 *                 workspace holds.  Each partition keeps (max, sum, partial
 *                 output) in the workspace; a second kernel merges them.  A
 *                 single request uses at most num_splits; a batch of 2 to
 *                 1,024 requests shares its batch * num_splits partitions,
 *                 cutting every request into pieces of one size chosen for
 *                 the whole batch (so a long request may take more than
 *                 num_splits and a short one fewer, and the split CTAs carry
 *                 equal work).
 * Numerics: K codes and q enter fp16 tensor-core products with fp32
 * accumulation (q is rescaled by a power of two per KV head when max|q| >= 2^14,
 * so any finite bf16 q is accepted); the softmax runs in fp32 with the
 * maximum subtracted; probabilities scaled by the V group scale enter fp16
 * products, so V group scales must stay below 65504; the V bias term
 * sum_t bias_t p_t is accumulated in fp32.  Output rounded RNE.
 * TQ4 pools (pool->tq4 required): the query is rotated once, q' = H S_K q /
 * sqrt(D), and scaled by a power of two into the fp16 range; indices meet
 * fp16 centroids in fp16 tensor-core products with fp32 accumulation, scores
 * are scaled by the K norms, probabilities times V norm times 2^-8 enter
 * fp16 products, and the accumulated output is rotated back by S_V H / sqrt(D)
 * in fp32.  jf_paged_verify_attn and jf_paged_decode_append_attn take TQ4
 * pools the same way (the fused step encodes the new rows exactly as
 * jf_kv_quantize_append does); the no-workspace variant returns
 * JF_ERR_UNSUPPORTED for them.
 */
int jf_paged_decode_attn(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                         const int32_t* context_lens, int32_t batch, const void* q,
                         int32_t num_q_heads, float softmax_scale, void* out, void* workspace,
                         size_t workspace_bytes, int32_t num_splits, void* stream);

/*
 * Packed multi-query verifier (Sec. 3.1, speculative verification of two to
 * four proposed tokens at once; App. A.1 dispatch: causal masks, query
 * lengths 2-4).  Each request b has q_len query tokens at absolute positions
 * context_lens[b] - q_len + i (i < q_len), already appended to the pool;
 * token i attends positions [0, context_lens[b] - q_len + i] causally:
 *   out[b, i, h, :] = sum_t softmax_t(scale * <q[b, i, h], K_t>) V_t.
 * The page reads are shared by the tokens.  With more than 8 (token, head)
 * rows per KV head (G * q_len > 8) a split CTA holds up to 24 of them and its
 * warps work in pairs on each 32-position chunk, each warp for half of D, so
 * every 4-bit code (or TQ4 index) is unpacked once per chunk; more than 24
 * rows take ceil(G * q_len / 24) CTAs per split over the same chunk range.
 * A single request then uses at most one split per SM and CTA of a KV head
 * (min(num_splits, SMs / (Hkv * CTAs)) splits; the workspace row stride
 * stays num_splits).  With 8 rows or fewer, one CTA per split holds them.
 *   q, out        bf16 [batch, q_len, Hq, D]
 *   q_len         1..4 (1 is plain decode)
 *   context_lens  int32 [batch], >= q_len for every request that has tokens
 *                 (a shorter context gives each token the positions it has)
 *   workspace     >= jf_attn_workspace_bytes(batch, q_len * Hq, Hkv, D,
 *                 num_splits) bytes, 256-byte aligned
 * Other arguments, limits, numerics and errors as for jf_paged_decode_attn.
 */
int jf_paged_verify_attn(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                         const int32_t* context_lens, int32_t batch, const void* q,
                         int32_t q_len, int32_t num_q_heads, float softmax_scale, void* out,
                         void* workspace, size_t workspace_bytes, int32_t num_splits,
                         void* stream);

/*
 * Append-then-attend decode step in one launch pair (Sec. 3.3: the step's
 * pending cache write lands before its attention reads the pool; Sec. 3.1
 * decode).  For every request b with context_lens[b] >= 1 the bf16 vectors
 * k_new[b, h, :] and v_new[b, h, :] are quantized exactly as
 * jf_kv_quantize_append does and written to position context_lens[b] - 1,
 * then out is computed exactly as jf_paged_decode_attn computes it over
 * positions [0, context_lens[b]).  The result (pool bytes and out) equals
 * jf_kv_quantize_append with row_req = b, row_pos = context_lens[b] - 1
 * followed by jf_paged_decode_attn; the fused form saves one launch and one
 * grid-wide dependency per step.  Each new row is written by the split that
 * owns its position, before that split reads it.
 *   k_new, v_new  bf16 [batch, Hkv, D], 16-byte aligned
 * Other arguments, limits and errors as for jf_paged_decode_attn; a bad page
 * id for the new row sets JF_DEV_ERR_PAGE_ID in the status word and skips
 * that write.
 */
int jf_paged_decode_append_attn(const jf_kv_pool* pool, const int32_t* page_table,
                                int32_t pt_stride, const int32_t* context_lens, int32_t batch,
                                const void* k_new, const void* v_new, const void* q,
                                int32_t num_q_heads, float softmax_scale, void* out,
                                void* workspace, size_t workspace_bytes, int32_t num_splits,
                                void* stream);

/*
 * Prefill-chunk attention for one request (Sec. 3.1 "decode and prefill need
 * different kernels"; Eq. 5).  chunk_len queries q[i] at absolute positions
 * q_start + i attend positions [0, q_start + i] (causal != 0) or
 * [0, q_start + chunk_len) (causal == 0) of the request's cache, which must
 * already hold the chunk's own rows (append, then attend).
 *   page_table_row  int32 [>= ceil((q_start + chunk_len) / P)]
 *   q, out          bf16 [chunk_len, Hq, D]
 *   workspace       affine pool: >= jf_prefill_workspace_bytes() (an int32
 *                   status word); TQ4 pool: >= jf_prefill_batch_workspace_bytes(
 *                   JF_FMT_TQ4, chunk_len, Hq, D, 1), 256-byte aligned.
 * Wave balance: the kernel runs one CTA per SM, two per pair.  A chunk over
 * a long prefix (q_start >= 4 chunk_len) whose CTA pairs would leave the last
 * wave partly empty runs, when the workspace holds
 * jf_prefill_chunk_workspace_bytes(...) bytes (256-byte aligned), as two
 * launches: its first query tiles as whole waves, then the rest with their
 * history split across pairs and merged (as jf_prefill_batch_attn with
 * num_splits > 1).  With a smaller workspace it runs as one launch.  Both
 * forms compute the same attention; the summation order, and so the last
 * bits, differ.
 * Numerics (affine pools): each 64-position K/V tile is rebuilt in shared
 * memory as fp16 code * scale + bias (one rounding) for the tensor cores, and
 * q * softmax_scale * log2(e) enters as fp16; accumulation and the softmax
 * run in fp32.  A K or V group whose reconstruction can leave the fp16 range
 * (|bias| + 15 scale >= 65504, or a non-finite scale/bias word) sets
 * JF_DEV_ERR_RANGE in the status word; outputs that attend such a group are
 * then not reliable.
 * TQ4 pools (Sec. 3.1: page lookup, unpacking, centroid lookup, inverse
 * rotation and norm restoration fused into the attention's operand path):
 * the queries are rotated once (q' = H S_K q / sqrt(D), fp32 in the
 * workspace), K and V tiles are built in shared memory as norm * centroid
 * (fp16) in the rotated basis, and each output row is rotated back
 * (S_V H / sqrt(D)) as the partials are merged.
 */
int jf_prefill_chunk_attn(const jf_kv_pool* pool, const int32_t* page_table_row,
                          const void* q, int32_t q_start, int32_t chunk_len, int32_t num_q_heads,
                          float softmax_scale, int32_t causal, void* out, void* workspace,
                          size_t workspace_bytes, void* stream);

/* Workspace bytes with which jf_prefill_chunk_attn runs this chunk in its
 * wave-balanced form on a GPU with num_sms SMs (0: the current device's);
 * the plain minimum when the chunk runs as one launch anyway.  Host only
 * (with num_sms > 0 it touches no device).  0 for invalid arguments. */
size_t jf_prefill_chunk_workspace_bytes(const jf_kv_pool* pool, int32_t q_start,
                                        int32_t chunk_len, int32_t num_q_heads, int32_t num_sms);

/*
 * Prefill chunks of several requests in one launch (Sec. 3.3: the scheduler
 * advances admitted prompts in bounded chunks between decode opportunities;
 * Sec. 3.1 / Eq. 5 for the attention).  Request b's chunk_len[b] queries at
 * absolute positions q_start[b] + i attend positions [0, q_start[b] + i]
 * (causal != 0) or [0, q_start[b] + chunk_len[b]) of its own cache, whose
 * pages are page_table[b * pt_stride ..]; every chunk's rows must already be
 * appended.  Each output equals jf_prefill_chunk_attn on that request alone.
 *   page_table   int32 [batch, pt_stride] (device)
 *   q_start, chunk_len  int32 [batch] on the HOST (scheduling metadata the
 *                caller already holds); q_start[b] + chunk_len[b] <=
 *                pt_stride * P; a zero chunk_len is skipped
 *   q, out       bf16 [sum_b chunk_len[b], Hq, D]; request b's rows start at
 *                row sum_{b' < b} chunk_len[b']
 *   batch        1 .. JF_PREFILL_MAX_BATCH (JF_ERR_UNSUPPORTED above)
 *   num_splits   >= 1: each query tile's history (its attended positions, in
 *                whole 64-position tiles) is cut into num_splits contiguous
 *                ranges, each its own pair of CTAs writing an unnormalized
 *                partial (max, sum, output); a second kernel merges them.
 *                Short chunks over long prefixes need it to fill the GPU;
 *                1 is a single pass (no partials, no merge).
 *   workspace    >= jf_prefill_batch_workspace_bytes(pool->format,
 *                sum_b chunk_len[b], Hq, D, num_splits) bytes, 256-byte
 *                aligned; its first int32 is the device status word.
 * The longest request's query tiles are scheduled first.  Either format.
 */
#define JF_PREFILL_MAX_BATCH 64

/* Workspace of a prefill launch over a pool of `format`: 256 bytes for an
 * affine pool with num_splits == 1; else 256 + roundup(8 R S, 256) + 4 R S D,
 * R = total_rows * Hq (the split partials), plus 4 R D for a TQ4 pool (its
 * rotated queries).  0 for invalid arguments. */
size_t jf_prefill_batch_workspace_bytes(int32_t format, int64_t total_rows, int32_t num_q_heads,
                                        int32_t head_dim, int32_t num_splits);

int jf_prefill_batch_attn(const jf_kv_pool* pool, const int32_t* page_table, int32_t pt_stride,
                          int32_t batch, const int32_t* q_start, const int32_t* chunk_len,
                          const void* q, int32_t num_q_heads, float softmax_scale, int32_t causal,
                          int32_t num_splits, void* out, void* workspace, size_t workspace_bytes,
                          void* stream);

/*
 * Page reservation of one unshared request (Eq. 7):
 *   R = ceil((prompt_len + min(output_len, g_out)) / page_size)
 * page equivalents, g_out the guaranteed output (8,192 in the paper, page
 * size 256).  Host only.  Returns -1 for a negative length or guarantee, a
 * page size below 1, or a sum that overflows int64.
 */
int64_t jf_reservation_pages(int64_t prompt_len, int64_t output_len, int64_t g_out,
                             int32_t page_size);

/*
 * Page-gather checkpoint (Sec. 3.4: read the request's page runs in place and
 * emit one packed stream).  Either format.  dst[k * page_bytes .. (k+1) * page_bytes) =
 * page record page_table_row[k] for k < num_pages, tail bytes included.
 *   dst        device buffer, >= num_pages * page_bytes bytes, 16-byte aligned
 *   err_flag   device int32 or NULL (JF_DEV_ERR_PAGE_ID for bad ids; the
 *              record is left untouched in dst).
 */
int jf_kv_checkpoint(const jf_kv_pool* pool, const int32_t* page_table_row, int32_t num_pages,
                     void* dst, size_t dst_bytes, int32_t* err_flag, void* stream);

/*
 * Restore (Sec. 3.4: restoration writes packed runs into the existing pool):
 * the inverse of jf_kv_checkpoint.  Page record page_table_row[k] of the pool
 * = src[k * page_bytes ..).  Page ids must be distinct.  Either format.
 */
int jf_kv_restore(const jf_kv_pool* pool, const int32_t* page_table_row, int32_t num_pages,
                  const void* src, size_t src_bytes, int32_t* err_flag, void* stream);

/*
 * Self-test of the bounded-wait give-up path (no paper counterpart; failure
 * detection).  Every wait of the library's kernels on a copy is bounded: it
 * polls a fixed number of times, then the kernel ORs JF_DEV_ERR_TIMEOUT into
 * its status word and returns, so a copy that never lands costs an error bit
 * instead of a hung GPU.  This call runs that path alone in one thread: it
 * waits on a shared-memory barrier that completes only if arrive != 0, so
 * with arrive == 0 the wait runs out (after 4,096 polls) and JF_DEV_ERR_TIMEOUT
 * is ORed into *status; with arrive != 0 *status is left unchanged.  No copy
 * or other CTA is involved and the CUDA context stays usable.
 *   status  device int32
 */
int jf_selftest_bounded_wait(int32_t* status, int32_t arrive, void* stream);

/*
 * Decode attention without a caller-supplied workspace.  The paper has no
 * counterpart; this entry point exists for callers that cannot allocate
 * device memory themselves -- for example a plug-in running inside a host
 * runtime that owns the whole device-memory budget and hands out no
 * allocator, or a plain C caller with no CUDA allocator of its own.
 *
 * Same arguments and result as jf_paged_decode_attn minus the workspace:
 * the split partials live in a file-scope device array of
 * JF_STATIC_WORKSPACE_BYTES bytes inside libjfkv.so, which every GPU that
 * loads the library holds until the process exits.  Nothing is allocated
 * or freed by this call.
 *   - Calls whose jf_attn_workspace_bytes(batch, Hq, Hkv, D, num_splits)
 *     exceeds JF_STATIC_WORKSPACE_BYTES return JF_ERR_WORKSPACE_TOO_SMALL
 *     (lower num_splits or the batch).
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current; make that first
 *     call before any stream capture.
 *   - All calls on a device share the one array and it keeps the last
 *     call's contents; the call clears the status word it needs to start
 *     at zero.  Calls that overlap on the GPU (different streams, or
 *     several host threads) race on the array: serialize them.
 *   - err_flag: device int32 or NULL; receives this call's device status
 *     word (JF_DEV_* bits) once the call completes on `stream`.
 */
#define JF_STATIC_WORKSPACE_BYTES ((size_t)8 << 20)

int jf_paged_decode_attn_noalloc(const jf_kv_pool* pool, const int32_t* page_table,
                                 int32_t pt_stride, const int32_t* context_lens, int32_t batch,
                                 const void* q, int32_t num_q_heads, float softmax_scale,
                                 void* out, int32_t num_splits, int32_t* err_flag, void* stream);

/* Human-readable name of a JF_* status code. */
const char* jf_status_string(int status);

/* Library version string. */
const char* jf_version(void);

#ifdef __cplusplus
}
#endif
#endif /* JFKV_H */
