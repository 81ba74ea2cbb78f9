/*
 * milo.h -- C ABI of libmilo: decode attention over a many-shot prefix whose
 * KV cache is stored block-wise in low-rank form (MILO, Sec. 4.2-4.4).
 *
 * The paper stores, per block i of the prefix and per KV head, the truncated
 * SVD factors of the block's keys and values (Eq. 3):
 *     K_i ~ A^k_i S^k_i (B^k_i)^T,   V_i ~ A^v_i S^v_i (B^v_i)^T,
 * with per-block ranks r^k_i, r^v_i chosen by the entropy-driven allocation
 * (Eq. 5-7).  At inference (Alg. 1, Stage 2) a query attends (Eq. 1) to the
 * selected blocks' reconstructed keys and values.  This library computes that
 * attention exactly (up to floating-point rounding) without reconstructing:
 *     q . K^_i^T = (q P^k_i^T) (C^k_i)^T,   p V^_i = (p C^v_i) P^v_i,
 * where C = A S (singular values folded into the coefficients, n_i x r) and
 * P = B^T (r x d, orthonormal rows in the paper's setting; not required).
 *
 * Conventions for every entry point:
 *  - Return a milo_status_t; no exceptions or aborts cross the ABI.
 *  - "device" pointers are CUDA global memory of the current device; "host"
 *    pointers are ordinary CPU memory.  The caller owns every buffer it passes.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *  - bf16 arrays hold IEEE bfloat16 values.
 */
#ifndef MILO_H
#define MILO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MILO_OK = 0,
    MILO_ERR_INVALID_ARG = 1,   /* null pointer, bad size, unsupported head dim ...  */
    MILO_ERR_BAD_TABLE = 2,     /* block table inconsistent (lengths, ranks, bounds)  */
    MILO_ERR_ALIGNMENT = 3,     /* an offset or pointer is not 16-byte aligned        */
    MILO_ERR_UNSUPPORTED = 4,   /* valid but outside what the kernels implement       */
    MILO_ERR_CUDA = 5,          /* a CUDA runtime call failed                         */
    MILO_ERR_TIMEOUT = 6,       /* device: a bounded wait gave up (sticky word)       */
    MILO_ERR_DEVICE_BOUNDS = 7, /* device: an index check failed (sticky word)        */
    MILO_ERR_WORKSPACE = 8      /* workspace missing or smaller than required         */
} milo_status_t;

/* Short English description of a status code (static string). */
const char *milo_status_string(int32_t status);

/* Library version as major*10000 + minor*100 + patch. */
int32_t milo_version(void);

/* Human-readable detail of the last error returned on the calling thread
 * (empty string if none).  Valid until the thread's next libmilo call. */
const char *milo_last_error_message(void);

/*
 * Block table of one decoder layer (the paper's low-rank cache LC, Alg. 1).
 * Entry e = b * num_kv_heads + g describes block b, KV head g.  The table's
 * block order is the attention order; passing a subset of blocks is the
 * paper's retrieval selection (Alg. 1, Stage 2).
 *
 *   num_blocks    >= 0 (0 = no prefix; only tails are attended).
 *   num_kv_heads  >= 1.
 *   head_dim      64 or 128.
 *   block_len     host [num_blocks]: tokens n_b of block b, 1 <= n_b <= 65536
 *                 (blocks may differ in length: a block holds m_i examples).
 *   rank_k/v      host [num_blocks * num_kv_heads]: 0 <= r <= head_dim.
 *                 A rank of 0 stores an all-zero key (or value) block.
 *   off_ck/pk/cv/pv host [num_blocks * num_kv_heads]: element offsets into
 *                 `arena` of C^K (n_b x r^k), P^K (r^k x d), C^V (n_b x r^v),
 *                 P^V (r^v x d), each row-major and dense; each offset a
 *                 multiple of 8 elements (16 bytes).  Regions must lie inside
 *                 [0, arena_elems) and must not overlap.
 *   arena         device bf16 [arena_elems], 16-byte aligned.  Read only by
 *                 milo_prefix_create; it may be freed after that call returns.
 *   arena_elems   size of `arena` in elements.
 */
typedef struct {
    int32_t num_blocks;
    int32_t num_kv_heads;
    int32_t head_dim;
    const int32_t *block_len;
    const int32_t *rank_k;
    const int32_t *rank_v;
    const int64_t *off_ck;
    const int64_t *off_pk;
    const int64_t *off_cv;
    const int64_t *off_pv;
    const void *arena;
    int64_t arena_elems;
} milo_block_table_t;

/* Opaque per-layer plan: packed factors, the work lists, accumulators. */
typedef struct milo_prefix milo_prefix_t;

/*
 * Check a block table on the host (no device access): lengths, ranks,
 * alignment, bounds, and pairwise overlap of the factor regions.
 * Returns MILO_OK, MILO_ERR_INVALID_ARG, MILO_ERR_BAD_TABLE or
 * MILO_ERR_ALIGNMENT.  milo_prefix_create runs the same checks.
 */
milo_status_t milo_validate_table(const milo_block_table_t *table);

/*
 * Packed ("kernel-native") layout of the factors, computed on the host.
 * Each factor is stored zero-padded to r8 = roundup(r, 8) ranks and, for the
 * coefficient matrices, n8 = roundup(n_b, 8) tokens, as 8x8 bf16 tiles of 128
 * contiguous bytes (one tile = 8 rows x 16 bytes):
 *   C (n_b x r): tile (token group tg, rank group rg) sits at
 *     (tg * r8/8 + rg) * 128 and holds row (t % 8), column (j % 8); tokens
 *     [t0, t1) with t0 % 8 == 0 are the contiguous bytes
 *     [t0 * r8 * 2, roundup(t1, 8) * r8 * 2).
 *   P (r x d): tile (rank group jg, column group cg) sits at
 *     (jg * d/8 + cg) * 128 and holds row (j % 8), column (c % 8).
 * packed_offsets: host [num_blocks * num_kv_heads * 4] byte offsets of
 * (C^K, P^K, C^V, P^V) for every entry (128-byte aligned); total_bytes: size
 * of the packed arena.  Either output may be NULL.
 */
milo_status_t milo_packed_layout(const milo_block_table_t *table,
                                 int64_t *packed_offsets, int64_t *total_bytes);

/*
 * Host-only: the static partition of the prefix over `num_shares` thread
 * blocks of the tensor-core grid (Alg. 1 Stage 2 split over token ranges,
 * merged by Eq. 1).  The prefix (every entry's tokens, KV-head-major, then
 * block order) is laid on a cost line in 32-token tiles, a tile of t8 tokens
 * (rounded up to 8) costing t8 x (64 + r16(r^k) + r16(r^v)) (r16 = rank
 * rounded up to 16: the softmax of a 128-row tile and the hi and lo score and
 * value products) and each entry's first tile 60000 more (its projection,
 * staging and back-projection); a tile goes to the share of the line,
 * (c T / num_shares, (c + 1) T / num_shares], that holds the midpoint of the
 * tile's cost, so no share costs more than T / num_shares plus one tile.
 * Consecutive tiles of one entry in one share form a segment; consecutive
 * segments of one share with the same KV head form a "run" whose partial
 * result occupies one slot (slots numbered in order, hence by KV head).
 *   seg_entry/seg_t0/seg_t1/seg_slot: host arrays of capacity `max_segments`
 *     (entry index b * num_kv_heads + g, token range [t0, t1), slot); all may
 *     be NULL to query the count.
 *   share_begin: host [num_shares + 1] first segment of each share; may be
 *     NULL.
 *   num_segments/num_slots: outputs (either may be NULL).
 * Returns the table's validation status, MILO_ERR_INVALID_ARG for
 * num_shares < 1, or (after setting the outputs) if max_segments is too small.
 */
milo_status_t milo_partition_prefix(const milo_block_table_t *table,
                                    int32_t num_shares, int32_t max_segments,
                                    int32_t *seg_entry, int32_t *seg_t0,
                                    int32_t *seg_t1, int32_t *seg_slot,
                                    int32_t *share_begin, int32_t *num_segments,
                                    int32_t *num_slots);

/*
 * Host-only: the work list of the chunk grid.  Every prefix entry, KV-head-major then in block
 * order, is cut into the fewest token ranges of at most 1024 tokens whose
 * coefficient rows (C^K and C^V at ranks rounded up to 8, tokens rounded up
 * to 8, bf16) fit 128 KB, of equal length in multiples of 32 tokens (the
 * last range takes the remainder; an entry of rank 0 in K and V, which has
 * no coefficient rows, is cut into 32-token ranges); each range is one thread block of the
 * decode grid per row group of 8 query rows (two row groups share a block
 * once a KV head has more than 8 rows).
 *   chunk_entry/chunk_t0/chunk_t1: host arrays of capacity `max_chunks`
 *     (entry index b * num_kv_heads + g, token range [t0, t1)); all may be
 *     NULL to query the count.
 *   num_chunks: output (may be NULL).
 * Returns MILO_ERR_INVALID_ARG (after setting num_chunks) if max_chunks is
 * too small, or the table's validation status.
 */
milo_status_t milo_chunk_prefix(const milo_block_table_t *table,
                                int32_t max_chunks, int32_t *chunk_entry,
                                int32_t *chunk_t0, int32_t *chunk_t1,
                                int32_t *num_chunks);

/*
 * Build a plan for one layer on the current device: validate the table,
 * allocate and fill the packed arena (a pack kernel on `stream`, then a
 * stream synchronisation), build the work lists and the device-side
 * accumulators.  The logical arena may be freed after this call returns.
 *   num_q_heads   multiple of num_kv_heads (query head h reads KV head
 *                 h / (num_q_heads / num_kv_heads)).
 *   max_batch     largest batch any decode call on this plan will use.
 *   out_plan      receives the plan; release with milo_prefix_destroy.
 * Errors: the table's validation status; MILO_ERR_INVALID_ARG for a bad
 * head count or max_batch < 1; MILO_ERR_UNSUPPORTED for
 * max_batch x (num_q_heads / num_kv_heads) above 2^30;
 * MILO_ERR_CUDA when an allocation, copy or the pack kernel fails.
 */
milo_status_t milo_prefix_create(const milo_block_table_t *table,
                                 int32_t num_q_heads, int32_t max_batch,
                                 void *stream, milo_prefix_t **out_plan);

/* Free a plan and its device memory (synchronises the device first). */
milo_status_t milo_prefix_destroy(milo_prefix_t *plan);

/* Plan facts for accounting and tests. */
typedef struct {
    int32_t num_blocks, num_kv_heads, num_q_heads, head_dim, max_batch;
    int64_t prefix_tokens;        /* sum of block lengths                     */
    int64_t logical_factor_bytes; /* bytes of C^K,P^K,C^V,P^V at true ranks   */
    int64_t packed_bytes;         /* bytes of the packed arena (with padding) */
    const void *packed_arena;     /* device pointer to the packed arena (an   */
                                  /* offloaded or INT8 plan: the staged copy, */
                                  /* or NULL)                                 */
} milo_prefix_info_t;

milo_status_t milo_prefix_get_info(const milo_prefix_t *plan,
                                   milo_prefix_info_t *info);

/*
 * Workspace a decode call needs (device memory the caller provides): the
 * split-softmax partial results (running max, sum and output per partition
 * of the tokens, Eq. 1 split over token ranges).  `bytes` receives the size,
 * enough for milo_attn_decode and milo_attn_decode_reconstruct alike.
 */
milo_status_t milo_workspace_size(const milo_prefix_t *plan, int32_t batch,
                                  int64_t max_tail_tokens, size_t *bytes);

/*
 * How a decode call of this shape runs (host only, no device access):
 *   path     MILO_PATH_CHUNKS (0): the chunk grid on warp-level MMA, one
 *            thread block per prefix chunk and row group of 8 query rows
 *            (fewer query rows per KV head than the tensor-core threshold,
 *            or no prefix: then the grid holds the tail items alone);
 *            MILO_PATH_TENSOR (1): the tensor-core grid (tcgen05, 128 query
 *            rows per product) for the prefix, with the dense tails on the
 *            chunk grid (at least the plan's threshold of query rows per KV
 *            head: milo_tensor_min_rows() unless set, see below).
 *   kernels  kernel launches of one call (each a grid).
 *   row_tiles  tensor-core path: tiles of 128 query rows per KV head (else 0).
 *   blocks   thread blocks of the call's main prefix grid.
 * Errors: MILO_ERR_INVALID_ARG for a null argument, batch outside
 * [1, max_batch] or max_tail_tokens < 0.
 */
typedef enum { MILO_PATH_CHUNKS = 0, MILO_PATH_TENSOR = 1 } milo_path_t;
typedef struct {
    int32_t path;
    int32_t kernels;
    int32_t row_tiles;
    int32_t blocks;
} milo_call_info_t;
milo_status_t milo_call_info(const milo_prefix_t *plan, int32_t batch,
                             int64_t max_tail_tokens, milo_call_info_t *info);

/* Query rows per KV head (batch x query heads per KV head) from which a
 * call takes the tensor-core path, by default. */
int32_t milo_tensor_min_rows(void);

/*
 * Set a plan's threshold (host only): its calls with at least `rows` query
 * rows per KV head take the tensor-core path, the others the chunk grid
 * (rows = 1: every call with a prefix on the tensor cores; a value above
 * max_batch x G: never).  Both paths compute the same attention; the
 * threshold only chooses the faster, so it is a tuning and testing knob.
 * It applies to calls enqueued after it returns, and milo_workspace_size
 * and milo_call_info follow it (the workspace a call needs depends on its
 * path).  An INT8 plan read directly always takes the chunk grid.
 * Errors: MILO_ERR_INVALID_ARG for a null plan or rows < 1.
 */
milo_status_t milo_prefix_set_tensor_min_rows(milo_prefix_t *plan, int32_t rows);

/*
 * One decode-attention call for one layer (Alg. 1 Stage 2 + Eq. 1):
 * for every query i and query head h (KV head g = h / G),
 *   out[i, h] = softmax(scale * q[i,h] . [K^_1 .. K^_N, Ktail_i[:, g]]) [V^ ...].
 *   q            device bf16 [batch, num_q_heads, head_dim].
 *   batch        1 <= batch <= plan's max_batch.
 *   tail_k/v     device bf16 [tail_rows, num_kv_heads, head_dim], 16-byte
 *                aligned; may be NULL when max_tail_tokens == 0.
 *   tail_offsets device int64 [batch + 1]: query i's tail is rows
 *                tail_offsets[i] .. tail_offsets[i+1]-1 (cu_seqlens style;
 *                nondecreasing, tail_offsets[batch] <= tail_rows).  May be NULL
 *                when max_tail_tokens == 0.
 *   tail_rows    rows allocated in tail_k / tail_v.
 *   max_tail_tokens  host upper bound on every query's tail length; it sets
 *                how the tails are split, a longer tail is an error recorded
 *                in the device status word (MILO_ERR_DEVICE_BOUNDS).
 *   softmax_scale  <= 0 selects 1 / sqrt(head_dim).
 *   out          device fp32 [batch, num_q_heads, head_dim].
 *   workspace    device, at least milo_workspace_size bytes, 16-byte aligned.
 * Asynchronous on `stream`: no host synchronisation and no allocation, so the
 * call can be captured in a CUDA graph.  A call is two or three kernels
 * (milo_call_info) launched with programmatic dependent launch: the prefix
 * grid may begin streaming the plan's factors before the preceding kernel on
 * `stream` finishes, and reads q, the tails and the workspace only after it
 * has; the last combines and writes `out`.  A plan holding pre-RoPE factors
 * (milo_prefix_set_rope) is refused with MILO_ERR_UNSUPPORTED: rank-space
 * scoring cannot apply a per-position rotation.  An offloaded plan must be
 * staged first (MILO_ERR_INVALID_ARG otherwise); an INT8 plan in device
 * memory that is not staged is read from its codes (milo_prefix_quantize_int8).
 * A plan must not be used by two calls that can run concurrently (it holds
 * per-call accumulators).  A query whose prefix and tail
 * are both empty yields NaN.  A call with more than 2^31 - 1 work items
 * (prefix chunks x row groups plus tail items) returns MILO_ERR_UNSUPPORTED
 * without launching anything.
 */
milo_status_t milo_attn_decode(const milo_prefix_t *plan, const void *q,
                               int32_t batch, const void *tail_k,
                               const void *tail_v, const int64_t *tail_offsets,
                               int64_t tail_rows, int64_t max_tail_tokens,
                               float softmax_scale, float *out, void *workspace,
                               size_t workspace_bytes, void *stream);

/*
 * milo_attn_decode without a workspace argument: the same computation, with
 * the partial results kept in a fixed scratch array built into the library
 * (8 MiB per GPU, held by every GPU that loads the library until the process
 * exits).  The paper has no counterpart; this exists for callers that cannot
 * allocate device memory on the decode path -- a plug-in that receives only
 * its inputs and outputs from a host runtime owning all device memory, or a
 * caller that must not call cudaMalloc there because it can synchronise the
 * device and stall other work.
 *   Arguments are those of milo_attn_decode minus workspace/workspace_bytes.
 *   Returns MILO_ERR_WORKSPACE if the call needs more scratch than the array
 *   holds (milo_workspace_size tells), without launching anything.
 *   The call allocates nothing.  Its first call on a device looks up the
 *   array's device address (once per device, with that device current); make
 *   that first call before any stream capture.  The scratch needs no
 *   clearing (every partial result is written before it is read in the same
 *   call) and keeps the last call's contents; all calls on a device share it,
 *   so calls that can overlap on the GPU (different streams) race.
 */
milo_status_t milo_attn_decode_static(const milo_prefix_t *plan, const void *q,
                                      int32_t batch, const void *tail_k,
                                      const void *tail_v,
                                      const int64_t *tail_offsets,
                                      int64_t tail_rows, int64_t max_tail_tokens,
                                      float softmax_scale, float *out,
                                      void *stream);

/*
 * The same decode call by reconstruct-then-attend, the paper's own inference
 * path (Alg. 1 Stage 2 with the fused reconstruction of Sec. 3.5): every
 * prefix token's key and value are rebuilt densely, K^ = C^K P^K and
 * V^ = C^V P^V, in fp16 tiles in shared memory (the paper's fp16 KV buffer)
 * and attended by flash decoding, instead of being scored in rank space.  It
 * is the comparison for the rank-space path and the path for pre-RoPE
 * factors.
 *   Arguments, layouts, ownership, workspace and errors are those of
 *   milo_attn_decode, and a plan's per-call state is shared between the two
 *   (calls on one plan must not overlap).  It needs a prefix and at most 8
 *   query heads per KV head (else MILO_ERR_UNSUPPORTED).  q, the
 *   reconstructed keys and values must lie inside the fp16 range (|x| < 65504).
 *   Three kernels at most: the tails' chunk grid (when there are tails), the
 *   reconstructing prefix grid (one block of 8 warps per chunk of up to 256
 *   tokens of one entry and group of up to 128 query rows), the finish grid.
 */
milo_status_t milo_attn_decode_reconstruct(const milo_prefix_t *plan, const void *q,
                                           int32_t batch, const void *tail_k,
                                           const void *tail_v,
                                           const int64_t *tail_offsets,
                                           int64_t tail_rows, int64_t max_tail_tokens,
                                           float softmax_scale, float *out,
                                           void *workspace, size_t workspace_bytes,
                                           void *stream);

/*
 * Declare the plan's factors to be those of pre-RoPE keys (Sec. 3: keys are
 * compressed before the rotary position embedding).  milo_attn_decode_reconstruct
 * then rotates every reconstructed prefix key to its position before scoring:
 * dimension i pairs with i + head_dim/2, and pair i turns counter-clockwise by
 * position * rope_theta^(-2i/head_dim); block b's token t sits at position
 * block_pos[b] + t.  q and the dense tails are taken as already rotated (as a
 * KV cache stores them); values are not rotated.
 *   rope_theta  > 0: the rotary base (e.g. 1e6 for the Qwen2.5 models);
 *               0 clears the setting (the factors are the keys as scored).
 *   block_pos   host int64 [num_blocks], each in [0, 2^40], read during the
 *               call only; NULL places the blocks at their starts in the
 *               concatenated prefix (0, n_0, n_0 + n_1, ...).  A retrieval
 *               subset of blocks passes their original positions.
 * Builds the rotation tables on the plan's device: allocates, synchronises
 * the device and copies, so it must not be called during stream capture or
 * while a call on the plan may be running.  Errors: MILO_ERR_INVALID_ARG
 * (null plan, rope_theta negative or not finite, a position out of range,
 * another device current), MILO_ERR_UNSUPPORTED (no prefix), MILO_ERR_CUDA.
 */
milo_status_t milo_prefix_set_rope(milo_prefix_t *plan, double rope_theta,
                                   const int64_t *block_pos);

/*
 * The offloaded prefix (the paper's throughput setting, Sec. 5.2: factors
 * held in CPU memory and brought to the GPU per step).  milo_prefix_offload moves the
 * plan's packed arena to pinned host memory (on GB300: Grace memory, read
 * over NVLink-C2C) and frees its device copy; it synchronises the device.
 * milo_prefix_stage then enqueues, on `stream`, the copy of that arena into a
 * caller-owned device buffer (at least milo_prefix_get_info's packed_bytes,
 * 128-byte aligned) and points the plan at it: the plan's decode calls from
 * then on read that buffer, which must hold the copy until they are done
 * (order them after the copy: the same stream, or an event).  Two buffers
 * let the copy of the next layer overlap the decode of this one.  A decode
 * call on an offloaded plan that was never staged returns
 * MILO_ERR_INVALID_ARG.  Staging is an ordinary asynchronous copy and can be
 * captured in a CUDA graph.  device_buffer NULL (bytes ignored): an INT8
 * plan in device memory stops reading a staged buffer and reads its codes
 * directly again (see milo_prefix_quantize_int8).  Errors:
 * MILO_ERR_INVALID_ARG (null plan, a plan not offloaded, a buffer too small,
 * a NULL buffer for any other plan, another device current),
 * MILO_ERR_ALIGNMENT, MILO_ERR_CUDA.
 */
milo_status_t milo_prefix_offload(milo_prefix_t *plan);
milo_status_t milo_prefix_stage(milo_prefix_t *plan, void *device_buffer, size_t bytes,
                                void *stream);

/*
 * INT8 storage of the factors (Sec. 5.3, Table 2, "MILO + INT8": asymmetric
 * INT8 quantisation on top of the low-rank cache).  The group is one 8x8
 * bf16 core of a packed arena (128 bytes: 8 tokens x 8 ranks of C, or 8
 * ranks x 8 columns of P).  Per group: m = the smallest value (+0 for a
 * zero), s = (largest - m) / 255 in fp32 rounded up to bf16, the 64 codes
 * c = rint((x - m) * (1 / s)) clamped to [0, 255] (0 when s = 0 or 1 / s
 * overflows fp32), and the
 * value read back bf16(m + s c) (fp32 arithmetic, one rounding to nearest
 * even for the sum, one to bf16).  Layout for an arena of `bytes` bytes
 * (a multiple of 128), group g at bytes [128 g, 128 g + 128):
 *   codes    bytes / 2 bytes; group g's 64 codes at [64 g, 64 g + 64), in
 *            the core's element order; 8-byte aligned.
 *   params   bytes / 32 bytes; one little-endian 32-bit word per group, the
 *            bf16 bits of m in its low half and of s in its high half;
 *            4-byte aligned.
 * Stored bytes: 68 per 128-byte core (1.88x fewer than bf16).  Values must
 * be finite with (largest - smallest) below the largest finite float.
 *
 * milo_quantize_int8 / milo_dequantize_int8: one stream-ordered kernel each
 * over any packed arena, group by group (padding included: a group's zero
 * padding takes part in its minimum and maximum, and reads back as m + s c).  The pointers are device pointers, or (dequantise's
 * codes and params) mapped pinned host memory.  Errors: MILO_ERR_INVALID_ARG
 * (null pointer, bytes negative or not a multiple of 128), MILO_ERR_ALIGNMENT
 * (packed not 16-byte aligned, codes not 8, params not 4), MILO_ERR_CUDA.
 */
milo_status_t milo_quantize_int8(const void *packed, int64_t bytes, void *codes, void *params,
                                 void *stream);
milo_status_t milo_dequantize_int8(const void *codes, const void *params, int64_t bytes,
                                   void *packed, void *stream);

/*
 * milo_prefix_quantize_int8 replaces a plan's resident bf16 arena with its
 * INT8 form (codes then params in one allocation: device memory when
 * to_host = 0, mapped pinned host memory when to_host = 1, the offloaded
 * INT8 prefix) and frees the bf16 arena; it synchronises the device.
 * With the codes in device memory, milo_attn_decode reads them directly:
 * the chunk grid (MILO_PATH_CHUNKS, whatever the batch) copies each piece's
 * codes and parameters and reads them back in shared memory, as the
 * staging kernel below would (milo_attn_decode_reconstruct needs a staged
 * plan).  Any INT8 plan can instead be staged with milo_prefix_stage: it
 * enqueues on `stream` one kernel that reads the codes (over NVLink-C2C for
 * host storage) and writes the bf16 values read back, with every factor's
 * padding (ranks past r, tokens past n_b) set to 0, into the caller's
 * buffer (as for an offloaded plan: at least packed_bytes, 128-byte
 * aligned, held until the decode calls that read it are done); decode
 * calls then compute attention over those values on any path.  Host-held
 * codes are read only by staging.  milo_prefix_storage_bytes
 * gives the bytes the plan's arena occupies at rest (bf16 or INT8, wherever
 * it is).  Errors: MILO_ERR_INVALID_ARG (null plan, the plan already
 * offloaded or quantised, another device current), MILO_ERR_CUDA.
 */
milo_status_t milo_prefix_quantize_int8(milo_prefix_t *plan, int32_t to_host);
milo_status_t milo_prefix_storage_bytes(const milo_prefix_t *plan, int64_t *bytes,
                                        int32_t *int8, int32_t *on_host);

/*
 * The compression stage (Alg. 1 Stage 1) on the GPU.  For every block b and
 * KV head g of a prefix, the SVD of its keys and of its values (Eq. 3; from
 * the eigen-decomposition of X^T X by Jacobi rotations, fp32), the ranks of
 * each (KV head, K) and (KV head, V) group by the greedy of Eq. 7 for the
 * budget problem of Eq. 6 (every block first gets min(r_min, n_b, d) units,
 * then the remaining budget goes one unit at a time to the block whose next
 * singular value has the largest gain log(1 + sigma^2 / eps^2), ties to the
 * lowest block index, never above min(r_max, n_b, d)), and the factors
 * C = A Sigma (n_b x r, row-major) and P = B^T (r x d, row-major) in bf16.
 *   num_blocks, num_kv_heads   the prefix's blocks and KV heads.
 *   head_dim                   64 or 128.
 *   block_len                  host [num_blocks], each in [1, 65536].
 *   r_min, r_max               0 <= r_min <= r_max.
 *   budget_k, budget_v         R_tot of every (KV head, K) and (KV head, V)
 *                              group; at least sum_b min(r_min, n_b, d).
 */
typedef struct {
    int32_t num_blocks;
    int32_t num_kv_heads;
    int32_t head_dim;
    const int32_t *block_len;
    int32_t r_min, r_max;
    int64_t budget_k, budget_v;
} milo_encode_params_t;

/*
 * The arena milo_encode fills: offsets, host [num_blocks * num_kv_heads * 4]
 * element offsets of C^K, P^K, C^V, P^V of entry b * num_kv_heads + g (each
 * region sized for min(r_max, n_b, d) ranks, 8-element aligned), and
 * *arena_elems the bf16 elements it spans.  With the ranks milo_encode
 * returns, these offsets form a milo_block_table_t.  Either output may be
 * NULL.  Errors: MILO_ERR_INVALID_ARG, MILO_ERR_BAD_TABLE (a block length),
 * MILO_ERR_UNSUPPORTED (head_dim).
 */
milo_status_t milo_encode_layout(const milo_encode_params_t *params, int64_t *offsets,
                                 int64_t *arena_elems);

/* Device workspace milo_encode needs (256-byte aligned): per key and value
 * matrix the singular values and the d x d eigenvectors (8 d^2 + O(d) bytes
 * per block and KV head). */
milo_status_t milo_encode_workspace_size(const milo_encode_params_t *params, size_t *bytes);

/*
 * Compress a prefix.
 *   k, v       device bf16 [sum n_b, num_kv_heads, head_dim] (token-major, as a
 *              KV cache holds them; block b is tokens n_0 + .. + n_{b-1} on),
 *              16-byte aligned.  For pre-RoPE factors pass the keys before
 *              the rotary embedding.
 *   arena      device bf16, at least milo_encode_layout's count, 16-byte
 *              aligned: receives the factors at its offsets.
 *   rank_k/v   device int32 [num_blocks * num_kv_heads]: the ranks.
 *   sigma      device fp32 [2 * num_blocks * num_kv_heads * head_dim] or NULL:
 *              the singular values (row 2e keys, 2e + 1 values of entry e),
 *              non-increasing.
 *   workspace  device, milo_encode_workspace_size bytes, 256-byte aligned.
 * It copies its small tables to the device and waits for that copy; the
 * three grids then run asynchronously on `stream` (not for stream capture).
 * Errors: those of milo_encode_layout, MILO_ERR_ALIGNMENT, MILO_ERR_WORKSPACE,
 * MILO_ERR_INVALID_ARG (a budget below the starting ranks, an arena too
 * small, a null pointer), MILO_ERR_CUDA.
 */
milo_status_t milo_encode(const milo_encode_params_t *params, const void *k, const void *v,
                          void *arena, int64_t arena_elems, int32_t *rank_k, int32_t *rank_v,
                          float *sigma, void *workspace, size_t workspace_bytes, void *stream);

/*
 * Check of the failure reporting: one warp waits, through the bounded
 * mbarrier wait every kernel of the library uses, on an mbarrier that nothing
 * completes (arrive = 0) or that the warp completes first (arrive != 0), with
 * a limit of limit_ns nanoseconds (in [1e6, 1e10]).  A wait that runs out sets
 * MILO_ERR_TIMEOUT in the plan's status word (milo_get_device_status reads
 * it) and the kernel returns: the failure is reported without faulting or
 * hanging the GPU, and the context stays usable.  Asynchronous on `stream`.
 * Errors: MILO_ERR_INVALID_ARG (null plan, limit out of range, another
 * device current), MILO_ERR_CUDA.
 */
milo_status_t milo_check_bounded_wait(const milo_prefix_t *plan, int64_t limit_ns,
                                      int32_t arrive, void *stream);

/*
 * Read (and optionally clear) the plan's sticky device status word, which the
 * kernels set on a timed-out wait (MILO_ERR_TIMEOUT) or a failed device-side
 * index check (MILO_ERR_DEVICE_BOUNDS).  Synchronises `stream`.
 */
milo_status_t milo_get_device_status(const milo_prefix_t *plan, void *stream,
                                     int32_t clear, int32_t *code);

#ifdef __cplusplus
}
#endif

#endif /* MILO_H */
