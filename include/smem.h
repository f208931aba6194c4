/*
 * smem.h -- C ABI of the SMem reader hot path on one GB300 (sm_103a).
 *
 * SMem (arXiv 2609.32395) keeps a context as a static memory: every block of
 * b tokens is encoded once, on its own, into b memory rows, and a reader
 * attends within the current block (block-local causal self-attention) and
 * then across the rows of all strictly earlier blocks (block-causal
 * cross-attention, with an optional learned null row); Sec. 2 "Model" and
 * App. A "Reader". This library serves that reader's attention over a
 * block-paged cache of the per-layer cross-attention K/V of the memory rows
 * (the "materialized cross-attention K/V" of Sec. 3.1):
 *
 *   - a pool of slots, one slot per memory block, each holding the block's
 *     K and V rows for every layer and head (bf16);
 *   - per sequence, a block table sorted by block index (the canonical order
 *     of Sec. 2) mapping block index -> slot, and one FIFO of free slots;
 *   - in-block self-attention K/V rows of the block being decoded.
 *
 * Deleting a block is a table edit plus a slot free (no row moves, O(b) as
 * in Theorem 1's editing cost); reads depend only on the block set, and the
 * kernels reduce in an order fixed by the number of blocks read, so the same
 * block set gives bitwise-identical outputs whatever the edit path.
 *
 * Conventions
 *   - Element type "bf16" is IEEE bfloat16 (passed as void pointers).
 *   - Device pointers are CUDA device addresses of the current device; every
 *     device pointer must be 16-byte aligned (SMEM_ERR_ALIGN otherwise).
 *   - `stream` is a cudaStream_t cast to void* (NULL = legacy default
 *     stream). All device work is enqueued on it; no call blocks except
 *     where stated. Host bookkeeping is updated synchronously, so calls on
 *     one cache must be issued from one thread and, when they touch device
 *     state, on one stream (or streams the caller orders).
 *   - Return value: SMEM_OK (0) or a negative SMEM_ERR_* code. A failing
 *     call leaves the cache's state (tables, free list, device contents)
 *     as it was. No C++ exception crosses this interface.
 *   - The library allocates no device memory: the caller passes one device
 *     buffer of smem_cache_required_bytes() bytes to smem_cache_create and
 *     owns it; it must outlive the cache. The reader-layer calls at the end
 *     take a caller-owned workspace as well.
 *   - Supported shapes: block_tokens == rows_per_block == 64,
 *     head_dim 32, 64 or 128 (SMEM_ERR_UNSUPPORTED otherwise).
 *   - At head_dim 64 the one-block prefill's split plan depends only on the
 *     readable block count and the head count (at most 15 splits); it runs
 *     one thread-block cluster of splits + 1 CTAs per head when the device
 *     can hold all of them at once (checked at cache creation), else on the
 *     cluster-free kernel with the same splits. The environment variable
 *     SMEM_PREFILL_CLUSTERS=0, read at creation, selects the cluster-free
 *     kernel. Both merge the same partials in the same order: the outputs
 *     are bitwise equal in either mode, on any device.
 */
#ifndef SMEM_H
#define SMEM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SMEM_ABI_VERSION 8

enum {
    SMEM_OK = 0,
    SMEM_ERR_INVALID_ARG = -1,     /* bad argument value, shape or id      */
    SMEM_ERR_ALIGN = -2,           /* pointer not 16-byte aligned          */
    SMEM_ERR_NO_SUCH_SEQ = -3,     /* sequence id out of range             */
    SMEM_ERR_DUPLICATE_BLOCK = -4, /* block index already in the table    */
    SMEM_ERR_NO_SUCH_BLOCK = -5,   /* block index not in the table         */
    SMEM_ERR_POOL_FULL = -6,       /* no free slot                         */
    SMEM_ERR_TABLE_FULL = -7,      /* sequence holds max_blocks_per_seq    */
    SMEM_ERR_CUDA = -8,            /* a CUDA runtime call failed           */
    SMEM_ERR_DEVICE_FAULT = -9,    /* a kernel recorded an error           */
    SMEM_ERR_UNSUPPORTED = -10,    /* shape outside the supported set      */
    SMEM_ERR_NO_DEVICE = -11,      /* bookkeeping-only cache: no device op */
    SMEM_ERR_SCRATCH_LIMIT = -12   /* request needs more than the library's
                                      fixed scratch (smem_decode_static_scratch) */
};

/* Cache geometry. Notation of the paper: L reader layers, H heads of
 * dimension d_h, blocks of b tokens, R memory rows per block (R = b). */
typedef struct smem_config {
    int32_t n_layers;           /* L >= 1                                      */
    int32_t n_heads;            /* H >= 1                                      */
    int32_t head_dim;           /* d_h: 32, 64 or 128                          */
    int32_t block_tokens;       /* b: 64                                       */
    int32_t rows_per_block;     /* R: 64                                       */
    int32_t max_seqs;           /* sequence ids are 0 .. max_seqs-1            */
    int32_t max_blocks_per_seq; /* table capacity per sequence                 */
    int32_t capacity_slots;     /* C: pool slots (memory blocks held at once)  */
    int32_t has_null_row;       /* 1: prepend a per-layer learned null row     */
    int32_t max_decode_batch;   /* largest nb of smem_decode, <= max_seqs      */
    const int32_t *free_order;  /* host, C entries: initial FIFO order, a
                                   permutation of 0..C-1; NULL = ascending.
                                   Copied at create time.                      */
    int32_t recompute_kv;       /* 0: a slot holds the block's projected K/V
                                   for every layer (materialized, Sec. 3.1).
                                   1: a slot holds only the block's memory
                                   rows mu [R][d] (d = H*d_h, shared by all
                                   layers; stored as d/64 contiguous chunks
                                   of [R][64]); the reader-layer calls re-derive
                                   each layer's keys and values from them
                                   (the recompute regime, App. "Serving").
                                   The pool is then 2L times smaller.          */
    int32_t rope_window;        /* 0: no rotary phases. W in 1..63: the
                                   SMem+RoPE composite (Sec. 4, App. "Training
                                   recipes"): self-attention queries/keys turn
                                   by their in-block offset, a cross-attention
                                   query by its block index i and a memory
                                   row's key by max(j, i - W) (the null row's
                                   by max(0, i - W); App. "Needle", saturating
                                   offsets, W = 15 in the paper); values never
                                   turn. Pairs (2m, 2m+1) turn by
                                   phase * base^(-2m/d_h). All inputs are
                                   given UNROTATED; stored in-block keys are
                                   kept turned. Not with recompute_kv.          */
    float rope_base;            /* rotary base (10000 in the paper)           */
    int32_t n_kv_heads;         /* grouped-query attention (Sec. 3.1: it
                                   composes with the KV saving): key/value
                                   heads of the memory rows and the in-block
                                   rows, H % n_kv_heads == 0; query head h
                                   reads key/value head h / (H / n_kv_heads).
                                   Slots, in-block rows, null rows and every
                                   K/V argument then have n_kv_heads heads
                                   (and W_qkv is [d][d + 2 n_kv_heads d_h],
                                   W_kc/W_vc [d][n_kv_heads d_h]). 0: = H.
                                   Not with recompute_kv.                      */
} smem_config;

typedef struct smem_cache smem_cache;

/* Size in bytes of the device buffer a cache with this geometry needs
 * (pool, in-block K/V, null rows, device block tables, split-K workspace).
 * Returns 0 for an invalid or unsupported geometry. */
size_t smem_cache_required_bytes(const smem_config *cfg);

/* Creates a cache. dev_buf: device buffer of at least
 * smem_cache_required_bytes(cfg) bytes, 256-byte aligned, owned by the
 * caller; dev_buf == NULL with dev_bytes == 0 creates a bookkeeping-only
 * cache (tables and free list, no device state, no CUDA call; device
 * operations then return SMEM_ERR_NO_DEVICE). Device creation zeroes the
 * tables and the workspace counters on the legacy default stream and waits
 * for it. *out receives the handle. */
int smem_cache_create(const smem_config *cfg, void *dev_buf, size_t dev_bytes, smem_cache **out);

/* Frees the host state. The device buffer stays the caller's. The caller
 * must ensure no enqueued work on the cache is still pending. */
int smem_cache_destroy(smem_cache *c);

/* Sets the learned null row (App. A "Positions and memory": one d-vector
 * prepended to the memory, projected by each layer's key/value maps):
 * k_null, v_null: device bf16 [L][H][d_h]. Requires has_null_row. Until it
 * is set the null row's k and v are zero. */
int smem_set_null_row(smem_cache *c, const void *k_null, const void *v_null, void *stream);

/* Appends memory block `block_idx` of sequence `seq` (Sec. 2: a block's rows
 * are written once, at its frozen index, and never change): takes the slot
 * at the front of the free FIFO, copies K and V (device bf16
 * [L][H][R][d_h], the block's cross-attention keys/values for every layer)
 * into it and inserts (block_idx, slot) into the sorted table. block_idx
 * >= 0 and unique within the sequence. *slot_out (may be NULL) receives the
 * slot. On a bookkeeping-only cache K and V must be NULL. */
int smem_append_block(smem_cache *c, int32_t seq, int32_t block_idx, const void *K, const void *V,
                      void *stream, int32_t *slot_out);

/* Deletes block `block_idx` of `seq` (Theorem 1: the result is exactly the
 * memory in which the block was never encoded; other blocks keep their
 * indices): removes the table entry and puts the slot at the back of the
 * free FIFO (once no other table entry shares it). No memory row moves. */
int smem_delete_block(smem_cache *c, int32_t seq, int32_t block_idx, void *stream);

/* Shares a cached block (exact composition, Sec. 2: a block encoded once is
 * reusable under any surrounding content): the table of dst_seq gains an
 * entry (dst_idx -> the slot of src_seq's block src_idx); no row is copied.
 * Slots count the table entries naming them; smem_delete_block and
 * smem_release_seq drop one reference each, and a slot returns to the back of
 * the free FIFO when its last reference goes. Without rotary phases the
 * block keeps its index (dst_idx must equal src_idx, SMEM_ERR_INVALID_ARG
 * otherwise: moving a block needs a re-encode); on a rope_window cache its
 * rows carry no position and dst_idx is free. Errors, checked in this order:
 * SMEM_ERR_NO_SUCH_SEQ (either id), SMEM_ERR_INVALID_ARG (negative index),
 * SMEM_ERR_NO_SUCH_BLOCK, SMEM_ERR_INVALID_ARG (index rule),
 * SMEM_ERR_DUPLICATE_BLOCK, SMEM_ERR_TABLE_FULL. *slot_out (may be NULL)
 * receives the shared slot. */
int smem_share_block(smem_cache *c, int32_t src_seq, int32_t src_idx, int32_t dst_seq, int32_t dst_idx,
                     void *stream, int32_t *slot_out);

/* Number of table entries naming `slot` (0: free). */
int smem_slot_refs(const smem_cache *c, int32_t slot, int32_t *n_out);

/* Deletes every block of `seq`; slots go to the back of the free FIFO in
 * ascending block order. */
int smem_release_seq(smem_cache *c, int32_t seq, void *stream);

/* Writes in-block self-attention rows 0..n_rows-1 of (seq, layer) for a
 * later smem_decode (e.g. the K/V a one-block prefill computed for the first
 * n_rows tokens of the current block). K, V: device bf16 [n_rows][H][d_h],
 * 0 <= n_rows <= b. */
int smem_write_inblock(smem_cache *c, int32_t seq, int32_t layer, int32_t n_rows, const void *K,
                       const void *V, void *stream);

/* One-block reader attention for one layer (block-skip serving, Sec. 3.1):
 * the b query tokens of block `q_block_idx` of `seq`
 *   Osa[t] = softmax_{u<=t}(Qs[t].Ks[u] / sqrt(d_h)) Vs      (in-block causal)
 *   Oca[t] = softmax_r(Qc[t].k_r / sqrt(d_h)) v_r           (cross-attention)
 * where r runs over the null row (if any) and the rows of every table
 * block with index < q_block_idx, in ascending block index. An empty row
 * set gives Oca = 0. Qs, Ks, Vs, Qc, Osa, Oca: device bf16 [b][H][d_h];
 * fp32 accumulation, bf16 round-to-nearest-even outputs. */
int smem_prefill_block(smem_cache *c, int32_t seq, int32_t layer, int32_t q_block_idx, const void *Qs,
                       const void *Ks, const void *Vs, const void *Qc, void *Osa, void *Oca, void *stream);

/* One decode step of one layer for nb sequences (KV-cached decode,
 * Sec. 3.1): item i is sequence seq_ids[i] (distinct), whose new token sits
 * at in-block offset pos[i] in [0, b) of block q_block_idx[i]. The step
 * writes k_new[i], v_new[i] into in-block row pos[i] of (seq, layer), then
 *   osa[i] = softmax over in-block rows 0..pos[i] (the new one included)
 *   oca[i] = cross-attention over the null row (if any) and the rows of the
 *            table blocks with index < q_block_idx[i], ascending.
 * seq_ids, pos, q_block_idx: HOST arrays [nb]; qs, k_new, v_new, qc, osa,
 * oca: device bf16 [nb][H][d_h]. 1 <= nb <= max_decode_batch. */
int smem_decode(smem_cache *c, int32_t layer, int32_t nb, const int32_t *seq_ids, const int32_t *pos,
                const int32_t *q_block_idx, const void *qs, const void *k_new, const void *v_new,
                const void *qc, void *osa, void *oca, void *stream);

/* The decode step of smem_decode with HOST inputs and outputs (a serving
 * loop whose tokens live on the host): qs, k_new, v_new, qc are host bf16
 * arrays [nb][..][d_h] (k_new, v_new with n_kv_heads heads), osa, oca host
 * bf16 [nb][H][d_h] receiving the results. The call copies the inputs into
 * one half of the caller's device staging buffer `stage` (256-byte aligned,
 * at least smem_decode_host_stage_bytes(c, nb) bytes; consecutive calls
 * alternate between its two halves), runs the decode step on `stream`, and
 * copies the outputs back -- all asynchronous. With copy_stream NULL the
 * copies run on `stream`; with another stream the outputs come back on it
 * and the inputs go in on a stream of the library's own, all ordered by
 * events against the decode, so that one call's copies overlap the
 * neighbouring calls' decode steps and no call's inputs wait behind the
 * previous call's outputs (a half is reused only after its previous outputs
 * have left). The host arrays must stay valid until the stream(s) have
 * drained and should be pinned (pageable memory makes the copies
 * synchronous); the outputs are on the host, and every input has been
 * read, once copy_stream (or stream) has drained. The first such call
 * creates the cache's ordering events and input stream (destroyed with the
 * cache); no device memory is allocated.
 * The paper has no counterpart. */
size_t smem_decode_host_stage_bytes(const smem_cache *c, int32_t nb);
int smem_decode_host(smem_cache *c, int32_t layer, int32_t nb, const int32_t *seq_ids, const int32_t *pos,
                     const int32_t *q_block_idx, const void *qs, const void *k_new, const void *v_new,
                     const void *qc, void *osa, void *oca, void *stage, size_t stage_bytes, void *stream,
                     void *copy_stream);

/* Bytes of the library's fixed device scratch used by
 * smem_decode_static_scratch (16 MiB; held on every GPU that loads the
 * library, for the life of the process). */
#define SMEM_STATIC_SCRATCH_BYTES (16u << 20)

/* Same decode step, arguments and results as smem_decode, but its split-K
 * scratch (per-split partial softmax states, split tickets and the unit
 * scheduler's counters) lives in a fixed array inside the library instead
 * of in the cache's device buffer, and the call allocates nothing. It is for
 * callers that must not allocate device memory on the serving path: a plugin
 * inside an engine or graph runtime that owns every device allocation and
 * hands out only inputs and outputs, or a latency-critical loop where an
 * allocation's implicit device-wide synchronisation is not acceptable.
 * (The paper has no counterpart; this is an interface choice of this
 * library.)
 *   - Scratch needed: 256 + 4*H*min(nb, 512) rounded up to 256, plus
 *     4*H*(d_h + 4) per (item, split) pair of the largest 512-item chunk;
 *     a request above SMEM_STATIC_SCRATCH_BYTES returns
 *     SMEM_ERR_SCRATCH_LIMIT before anything is enqueued.
 *   - The first call on each device looks up the array's device address
 *     with that device current; make that first call before any stream
 *     capture on the device. The address belongs to the device's current
 *     context: a call made after that context changed (for instance after
 *     cudaDeviceReset) looks it up again, so it too should come before any
 *     capture.
 *   - It runs the same kernel instance and split plan as smem_decode (the
 *     grouped units of a grouped-query cache included), so its outputs are
 *     bitwise equal to smem_decode's on the same cache state.
 *   - Every call on every cache of the process shares the one array, and it
 *     keeps the last call's contents: each call first clears the counters it
 *     needs at zero. Calls whose work overlaps on the GPU (different streams
 *     without ordering) race on the array and give wrong results; order
 *     them. */
int smem_decode_static_scratch(smem_cache *c, int32_t layer, int32_t nb, const int32_t *seq_ids,
                               const int32_t *pos, const int32_t *q_block_idx, const void *qs,
                               const void *k_new, const void *v_new, const void *qc, void *osa,
                               void *oca, void *stream);

/* ------------------------------------------------------------------------
 * Full reader layer (arXiv 2609.32395, Sec. 2 "Model", App. A "Reader").
 * With d = H * d_h, one reader layer maps the residual stream x (fp32) by
 * three pre-LN residual branches:
 *   x1 = x  + SA(LN1(x) W_qkv) W_os        block-local causal self-attention
 *   x2 = x1 + CA(LN2(x1) W_qc) W_oc        cross-attention into memory rows
 *   x3 = x2 + GELU(LN3(x2) W_1) W_2        FFN of width 4d, GELU = x Phi(x)
 * LN(x) = (x - mean) / sqrt(biased variance + 1e-5) * g + b per token.
 * A memory row mu (d wide, the block-local encoder's output, shared by all
 * layers) has per-layer keys mu W_kc and values mu W_vc; the null row is one
 * d-vector nu projected the same way. The attentions are those of
 * smem_prefill_block / smem_decode on the same cache; projections are bf16
 * products with fp32 accumulation on the library's tensor-core kernels
 * (LayerNorm applied as the operand is loaded; residual add, GELU, rotary
 * phases and in-block rows applied as results are stored); intermediates LN
 * outputs, q/k/v, attention outputs and GELU outputs are rounded to bf16,
 * the residual stream stays fp32. Every projection reduces in an order fixed
 * by its shape and the device's SM count, so results are bitwise
 * reproducible. Layer calls are issued with programmatic dependent launch:
 * a projection may start loading its weights while the previous kernel on
 * the stream finishes.
 *
 * Workspace: every call below takes a device buffer `ws` of at least
 * smem_layer_workspace_bytes(c, n_rows) bytes (256-byte aligned, the
 * caller's), n_rows = b for a prefill, nb for a decode, 0 for the memory
 * projections. Calls that share a workspace must be ordered. */
typedef struct smem_layer_weights {
    const float *ln1_g, *ln1_b; /* [d] fp32                                     */
    const void *w_qkv;          /* bf16 [d][3d], columns Q | K | V, each [H][d_h] */
    const void *w_os;           /* bf16 [d][d]                                  */
    const float *ln2_g, *ln2_b; /* [d]                                          */
    const void *w_qc;           /* bf16 [d][d], cross-attention query map       */
    const void *w_oc;           /* bf16 [d][d]                                  */
    const void *w_kc, *w_vc;    /* bf16 [d][d], memory-row key / value maps     */
    const float *ln3_g, *ln3_b; /* [d]                                          */
    const void *w_1;            /* bf16 [d][4d]                                 */
    const void *w_2;            /* bf16 [4d][d]                                 */
} smem_layer_weights;

/* Workspace bytes of a layer call over n_rows tokens (0 <= n_rows <=
 * max(b, max_decode_batch)); 0 for a bad argument. */
size_t smem_layer_workspace_bytes(const smem_cache *c, int32_t n_rows);

/* Appends memory block `block_idx` of `seq` given its memory rows: mu is
 * device bf16 [R][d]; w points to L HOST structs (layer 0..L-1) of which
 * w_kc and w_vc are read. The slot receives, for every layer l and head h,
 * K = mu W_kc^l[:, h d_h : (h+1) d_h] and V likewise (bf16), then the table
 * insert follows as in smem_append_block (same validation, errors and
 * FIFO order). On a recompute_kv cache the slot receives mu itself (in
 * 64-column chunks, each [R][64] contiguous) and w is not read (may be
 * NULL). */
int smem_append_block_rows(smem_cache *c, int32_t seq, int32_t block_idx, const void *mu,
                           const smem_layer_weights *w, void *ws, size_t ws_bytes, void *stream,
                           int32_t *slot_out);

/* Sets the null row from the d-vector nu (device bf16 [d]): per layer,
 * k_null = nu W_kc^l, v_null = nu W_vc^l. w: L host structs. Requires
 * has_null_row. On a recompute_kv cache nu itself is kept (w may be NULL). */
int smem_set_null_vector(smem_cache *c, const void *nu, const smem_layer_weights *w, void *ws,
                         size_t ws_bytes, void *stream);

/* One reader layer on the b tokens of block `q_block_idx` of `seq`
 * (block-skip serving, Sec. 3.1): x is device fp32 [b][d], read and
 * overwritten with the layer's output; w is one host struct (this layer's
 * weights). The block's self-attention keys/values (LN1(x) W_qkv, K and V
 * parts) are also stored as in-block rows 0..b-1 of (seq, layer), as
 * smem_write_inblock would, for later decode steps. Cross-attention reads
 * the null row and the table blocks with index < q_block_idx. */
int smem_reader_layer_prefill(smem_cache *c, int32_t seq, int32_t layer, int32_t q_block_idx,
                              const smem_layer_weights *w, float *x, void *ws, size_t ws_bytes,
                              void *stream);

/* One reader layer for one decode step of nb sequences (arguments as in
 * smem_decode): x is device fp32 [nb][d], read and overwritten; the new
 * tokens' self-attention k, v become in-block rows pos[i].
 *
 * On a recompute_kv cache both layer calls compute the cross-attention from
 * the memory rows: with q'_h = W_kc[:, h] q_h (times the softmax scale),
 * scores q'_h . mu_r and output (sum_r p_r mu_r) W_vc[:, h] -- the same
 * keys mu W_kc and values mu W_vc, re-associated so that each row is read
 * once per layer for all heads. q' and sum_r p_r mu_r are rounded to bf16.
 * smem_append_block, smem_set_null_row, smem_prefill_block, smem_decode and
 * smem_decode_static_scratch return SMEM_ERR_UNSUPPORTED there (they take
 * projected keys and values). */
int smem_reader_layer_decode(smem_cache *c, int32_t layer, int32_t nb, const int32_t *seq_ids,
                             const int32_t *pos, const int32_t *q_block_idx,
                             const smem_layer_weights *w, float *x, void *ws, size_t ws_bytes,
                             void *stream);

/* The memory-row cross-attention of a recompute_kv cache on its own (the
 * step between the two per-head maps of the reader layer): for every query
 * vector q' (d wide, already multiplied by W_kc,h and by the softmax scale
 * log2(e)/sqrt(d_h) -- scores are base-2 exponents)
 *   O'[q] = sum_r softmax_r(q' . mu_r) mu_r
 * over the null row nu (if any) and the memory rows of the table blocks with
 * index < the query block index, ascending. bf16 in and out, fp32
 * accumulation. ws as for the layer calls (smem_layer_workspace_bytes with
 * n_rows = nb, or b for the prefill form).
 * smem_mu_decode: item i reads sequence seq_ids[i] (distinct) below block
 *   q_block_idx[i] (host arrays [nb]); qp, op device [nb][H][d].
 * smem_mu_prefill: the b queries of every head of block q_block_idx of seq;
 *   qp, op device [H][b][d].
 * SMEM_ERR_UNSUPPORTED on a cache without recompute_kv. */
int smem_mu_decode(smem_cache *c, int32_t nb, const int32_t *seq_ids, const int32_t *q_block_idx,
                   const void *qp, void *op, void *ws, size_t ws_bytes, void *stream);
int smem_mu_prefill(smem_cache *c, int32_t seq, int32_t q_block_idx, const void *qp, void *op, void *ws,
                    size_t ws_bytes, void *stream);

/* Decode kernel of a recompute_kv cache's memory-row attention, chosen at
 * create time from H, d and the device (host state, no CUDA): *nq queries
 * per CTA; *cluster > 0: the column-slice form, each cluster of *cluster
 * CTAs streaming one row set once with *slice_cols columns per CTA (taken
 * only when the environment variable SMEM_MU_CLUSTERS is "1" at create
 * time); *cluster = 0: the two-pass form (one CTA reads each tile twice,
 * the second time normally from L2).
 * Any out pointer may be NULL. SMEM_ERR_UNSUPPORTED without recompute_kv,
 * SMEM_ERR_NO_DEVICE on a bookkeeping-only cache. */
int smem_mu_decode_plan(const smem_cache *c, int32_t *nq, int32_t *cluster, int32_t *slice_cols);

/* Introspection for bit-exact bookkeeping checks (host state, no CUDA).
 * smem_get_table: the table of `seq` in ascending block index; up to `cap`
 * entries into idx_out / slot_out (either may be NULL); *n_out = length.
 * smem_get_free_fifo: the free FIFO front to back. */
int smem_get_table(const smem_cache *c, int32_t seq, int32_t *idx_out, int32_t *slot_out, int32_t cap,
                   int32_t *n_out);
int smem_get_free_fifo(const smem_cache *c, int32_t *slots_out, int32_t cap, int32_t *n_out);

/* Copies the device copy of `seq`'s slot table (host int32, up to `cap`
 * entries, *n_out = length) after the work enqueued on `stream`. Blocks
 * until that stream has drained. */
int smem_get_device_table(smem_cache *c, int32_t seq, int32_t *slot_out, int32_t cap, int32_t *n_out,
                          void *stream);

/* Reads the device error word after the work enqueued on `stream` (blocks
 * until it drains): SMEM_OK, or SMEM_ERR_DEVICE_FAULT if a kernel gave up a
 * bounded wait; the word is then cleared. */
int smem_check_device_error(smem_cache *c, void *stream);

/* Number of pool slots currently free. */
int smem_free_slots(const smem_cache *c, int32_t *n_out);

/* Text describing the last SMEM_ERR_CUDA / SMEM_ERR_DEVICE_FAULT of the
 * calling thread (static storage, overwritten by the next failure). */
const char *smem_last_error_detail(void);

/* Testing hook (failure injection on the host): the n-th next device launch
 * of this cache fails with SMEM_ERR_CUDA before anything is enqueued, so
 * callers can check that a failing call leaves the state unchanged.
 * n = 0 disables it. */
int smem_debug_fail_after(smem_cache *c, int32_t n);

/* Testing hook (failure detection without a GPU fault): stores `slot` into
 * entry `pos` of the DEVICE copy of seq's table (pos < the table's length)
 * without touching the host state. A value other than the host's slot
 * corrupts the device table on purpose: a decode or prefill that meets a
 * slot outside [0, capacity) skips that read and records the device error
 * (smem_check_device_error then returns SMEM_ERR_DEVICE_FAULT). Writing the
 * host's slot back (smem_get_table) restores the entry. */
int smem_debug_set_table_entry(smem_cache *c, int32_t seq, int32_t pos, int32_t slot, void *stream);

/* Testing hook: launches a kernel whose one wait (an mbarrier nothing ever
 * arrives on) must give up after limit_ns nanoseconds (1 .. 1e9) and record
 * the device error, exercising the bounded waits every kernel uses. The
 * context stays usable; smem_check_device_error returns
 * SMEM_ERR_DEVICE_FAULT and clears the word. */
int smem_debug_wait_probe(smem_cache *c, long long limit_ns, void *stream);

/* Testing hook: one projection on the reader layer's tensor-core kernel, as
 * the layer calls use it (no counterpart in the paper; for kernel tests).
 *   out[b][m][n] = epi(alpha * sum_k A[b][m][k] W_b[k][n]),  b < batch
 * A: bf16 [M][lda] (+ b * a_bs elements). W: bf16 [w_rows][w_cols] (row
 * pitch w_cols); b_kmajor = 0: W_b[k][n] = W[k][n + b * w_boff];
 * 1: W_b[k][n] = W[n][k + b * w_boff]. epi 0: bf16 store, 1: fp32 add into
 * out, 2: GELU then bf16. Output column n of row m goes to out + b * o_bs +
 * (n / col_group) * group_stride + m * ldo + n % col_group (col_group 0: N).
 * N and K multiples of 32; device pointers 16-byte aligned. Uses the cache's
 * device only for its error word. */
int smem_debug_gemm(smem_cache *c, const void *A, int32_t lda, long long a_bs, const void *W, int32_t w_rows,
                    int32_t w_cols, int32_t b_kmajor, int32_t w_boff, int32_t M, int32_t N, int32_t K,
                    int32_t batch, int32_t epi, float alpha, void *out, int32_t ldo, long long o_bs,
                    int32_t col_group, long long group_stride, void *stream);

/* Testing hook: the reader layer's LayerNorm kernel, h [n][d] bf16 =
 * (x - mean) / sqrt(biased variance + 1e-5) * gain + bias per row of the fp32
 * x [n][d] (d a multiple of 4); fp32 statistics, bf16 round-to-nearest-even. */
int smem_debug_layernorm(smem_cache *c, const float *x, int32_t n, int32_t d, const float *gain, const float *bias,
                         void *h, void *stream);

/* Static text of an error code. */
const char *smem_strerror(int code);

/* SMEM_ABI_VERSION of the loaded library. */
int smem_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* SMEM_H */
