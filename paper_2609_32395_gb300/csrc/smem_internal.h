// smem_internal.h -- launch parameters and launchers shared by the C ABI
// (smem_capi.cpp) and the kernels (*.cu). Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime_api.h>

#ifdef __CUDACC__
#define SMEM_HD __host__ __device__
#else
#define SMEM_HD
#endif

namespace smem {

constexpr int kRows = 64;     // R: memory rows per block (one K/V tile)
constexpr int kBlockTok = 64; // b: query tokens per block

// ---------------------------------------------------------------------------
// device-buffer geometry (all offsets in bytes from dev_buf)
// ---------------------------------------------------------------------------
struct Layout {
  int L, H, D, max_seqs, max_blocks, capacity, has_null, max_batch;
  int Hkv;             // key/value heads of the memory rows and in-block rows (H % Hkv == 0)
  int recompute;       // 1: slots hold memory rows mu ([d/64][R][64]) instead of per-layer K/V
  int rope_w;          // 0: no rotary phases; else the saturating window W of the RoPE composite
  float rope_base;
  int dec_max_splits;  // split-K partial slots per (decode item, head)
  int pf_max_splits;   // split-K partial slots per prefill head
  size_t slot_elems;   // bf16 elements per pool slot: L*Hkv*2*R*D, or R*d (recompute)
  size_t off_pool, off_inblock, off_null, off_table, off_bidx, off_rope, off_rope_scr, off_dec_part, off_dec_cnt,
      off_pf_part, off_pf_cnt, off_err, total;
};

// Split-K plan of the decode cross-attention: the number of memory blocks a
// split reads, a function of the sequence's block count alone (so the same
// block set always reduces in the same order). Below 512 blocks, 16 blocks:
// a unit's fixed costs (queries, partial, ticket, merge) stay small next to
// its rows in batched decode. From 512 blocks on, ceil(nblk/64) within
// [8, 32] -- 64 splits up to 2048 blocks, 128 at 4096 -- so that a long
// context alone still gives the warps of every SM work. (Grouped-query
// units use the same plan: splits qn times shorter, for more units per warp,
// measured slower -- 13.9k against 18.2k tok/s at 4 key/value heads -- their
// per-unit partials, tickets and merges cost more than the shorter tail.)
SMEM_HD inline int decode_split_blocks(int nblk) {
  if (nblk < 512) return 16;
  const int sb = (nblk + 63) / 64;
  return sb < 8 ? 8 : (sb > 32 ? 32 : sb);
}
SMEM_HD inline int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Split plan of the one-block prefill cross-attention at d_h = 32 and 128
// (d_h = 64: prefill_split_blocks_d64), a function of the block count and the
// cache's fixed head count and head dimension alone: the cross-attention CTAs
// fit one wave on a GB300 (152 SMs; two CTAs per SM at d_h = 32, one at 128),
// at most kPrefillMaxSplits splits per head, at least two blocks per split.
constexpr int kPrefillMaxSplits = 16;
SMEM_HD inline int prefill_split_blocks(int nblk, int H, int D) {
  const int target = D <= 64 ? 304 : 152;
  int ns = target / H;
  if (ns > kPrefillMaxSplits) ns = kPrefillMaxSplits;
  if (ns > (nblk + 1) / 2) ns = (nblk + 1) / 2;
  if (ns < 1) ns = 1;
  return (nblk + ns - 1) / ns;
}

// ---------------------------------------------------------------------------
// decode
// ---------------------------------------------------------------------------
constexpr int kMaxDecodeItems = 512;  // items per launch (kernel parameter space)

struct DecodeItem {
  int seq;         // sequence id (row of the device table)
  int nblk;        // memory blocks read (table prefix with index < q_block_idx)
  int pos;         // in-block offset p of the new token
  int pair_begin;  // first (item, split) pair of this item
  int qblk;        // the token's block index (rotary phase of its cross-attention query)
};

// Rotary phases of the SMem+RoPE composite: a table of (cos, sin) of
// phase * theta_m for phases 0 .. kRopePhases-1 and pairs m < D/2
// (theta_m = base^(-2m/D)); self-attention phases are in-block offsets,
// cross-attention phase differences are clamped to the window W < 64.
constexpr int kRopePhases = 64;

struct DecodeParams {
  CUtensorMap tmap;          // pool viewed as [C][L*H*2*R][D] bf16, 128-byte swizzle
  const uint16_t* pool;      // [C][L][H][2][R][D]
  uint16_t* inblock;         // [max_seqs][L][H][2][b][D]
  const int* table;          // [max_seqs][max_blocks] slots, ascending block index
  const uint16_t* null_kv;   // [L][H][2][D] or nullptr
  float* part;               // [pair][H][D + 4]: m, l, pad, pad, acc[D]
  unsigned* counters;        // [max_batch][H] split tickets, zero between launches
  unsigned long long* sched; // [3]: next CA unit, warps finished, next SA unit; zero between launches
  int* err;                  // device error word
  const uint16_t* qs;        // [nb][H][D]
  const uint16_t* k_new;
  const uint16_t* v_new;
  const uint16_t* qc;
  uint16_t* osa;
  uint16_t* oca;
  long long slot_elems;      // elements per pool slot
  int L, H, layer, max_blocks, capacity;
  int n_items, n_pairs;      // items and CA (item, split) pairs in this launch
  int mode;                  // bit 0: in-block self-attention, bit 1: cross-attention
  int s_stride, c_stride;    // elements between items of qs and of qc
  int Hkv, kv_stride;        // key/value heads; elements between items of k_new/v_new
  int qn;                    // query heads per cross-attention unit (grouped-query decode; 1: one)
  float scale_log2;          // log2(e) / sqrt(D)
  const float2* rope_tab;    // [kRopePhases][D/2] (cos, sin), or nullptr: no rotary phases
  const int* bidx;           // [max_seqs][max_blocks] block index of each table entry
  int rope_w;                // saturating window W
  int max_seqs;              // rows of the device tables (bounds checks)
  long long part_pairs;      // (item, split) pairs the partial buffer holds (bounds checks)
  DecodeItem items[kMaxDecodeItems];
};

cudaError_t launch_decode(const DecodeParams& p, int D, int grid, cudaStream_t st);
// Query heads a grouped decode unit scores together for a group of G query
// heads per key/value head (1: one unit per query head).
int decode_group_width(int D, int G, bool rope);
// Device address of the fixed scratch array of smem_decode_static_scratch on
// the current device (looked up once per device). Returns a cudaError_t.
int static_scratch_address(void** out);
int decode_max_grid(int D, int num_sms);
int decode_warps_per_cta();
// Encodes the tensor map of the pool for the decode kernel (rows of D bf16,
// boxes of 64 columns x rows_per_box rows).
int encode_pool_map(CUtensorMap* map, void* pool, int L, int H, int D, int capacity, int rows_per_box);
int decode_stage_rows(int D);

// ---------------------------------------------------------------------------
// copies and table edits
// ---------------------------------------------------------------------------
// Appends: copy K, V [L][H][R][D] into a pool slot and insert `slot` at
// table position `pos` of `seq` (n_old entries before the insert).
// The block index is inserted at the same position of the block-index row.
cudaError_t launch_append(uint16_t* slot_base, const uint16_t* K, const uint16_t* V, int L, int H, int D,
                          int* table_row, int* bidx_row, int pos, int n_old, int slot, int block_idx,
                          cudaStream_t st);
// Removes table position `pos` of a row (and of its block-index row) holding n_old entries.
cudaError_t launch_table_remove(int* table_row, int* bidx_row, int pos, int n_old, cudaStream_t st);
// In-block write: rows [n][H][D] (token stride `tok` elements, 0: H*D) ->
// inblock[seq][layer][h][2][b][D]; with a rotary table the keys are stored
// turned by their in-block offset.
cudaError_t launch_inblock_write(uint16_t* ib_layer_base, const uint16_t* K, const uint16_t* V, int n, int H,
                                 int D, cudaStream_t st, int tok = 0, const float2* rope_tab = nullptr);
// Rotary phases by in-block offset, for two row sets at once (queries and
// keys): row t of a set (n tokens x H heads x D, token stride src_tok) turned
// by phase t into dst (token stride dst_tok; dst may equal src).
cudaError_t launch_rope_rows(const uint16_t* src_a, uint16_t* dst_a, int src_tok_a, int dst_tok_a, int H_a,
                             const uint16_t* src_b, uint16_t* dst_b, int src_tok_b, int dst_tok_b, int H_b, int n,
                             int D, const float2* rope_tab, cudaStream_t st);
// Null row: k,v [L][H][D] -> null_kv [L][H][2][D].
cudaError_t launch_null_write(uint16_t* null_kv, const uint16_t* k, const uint16_t* v, int L, int H, int D,
                              cudaStream_t st);
cudaError_t launch_zero(void* p, size_t bytes, cudaStream_t st);
// Testing hooks: store one int; a bounded wait that nothing completes.
cudaError_t launch_store_int(int* p, int v, cudaStream_t st);
cudaError_t launch_wait_probe(int* err, unsigned long long limit_ns, cudaStream_t st);
// Memory rows of a recompute cache: mu [R][d] (d a multiple of 64) -> slot
// [d/64][R][64], each 64-column chunk of the block contiguous (8 KB).
cudaError_t launch_mu_tile(uint16_t* slot, const uint16_t* mu, int d, cudaStream_t st);

// Table insert alone (the slot's rows written by other kernels before it).
cudaError_t launch_table_insert(int* table_row, int* bidx_row, int pos, int n_old, int slot, int block_idx,
                                cudaStream_t st);

// ---------------------------------------------------------------------------
// dense parts of the reader layer
// ---------------------------------------------------------------------------
constexpr float kLayerNormEps = 1e-5f;

// ---------------------------------------------------------------------------
// projections on tcgen05 (smem_gemm.cu)
// ---------------------------------------------------------------------------
enum GemmEpilogue : int {
  kEpiBf16 = 0,      // out (bf16) = alpha * acc
  kEpiAddF32 = 1,    // out (fp32) += alpha * acc  (residual stream)
  kEpiGeluBf16 = 2,  // out (bf16) = GELU(alpha * acc)
};

// One projection out[b][m][n] = epi(alpha * sum_k A[b][m][k] W_b[k][n]) for
// b < batch (grid z). A: bf16 [M][lda] (+ b * a_bs). W: the bf16 matrix
// [w_rows][w_cols] (row pitch ldw elements); b_kmajor = 0: W is [K][N] (the
// batch's columns start at b * w_boff); 1: W is [N][K] (the batch's K
// columns start at b * w_boff). Output column n goes to out + b * o_bs +
// (n / col_group) * group_stride + m * ldo + n % col_group (col_group 0: N).
// N and K multiples of 32.
struct GemmCall {
  const void* a = nullptr;
  int lda = 0;
  long long a_bs = 0;
  const void* w = nullptr;
  int w_rows = 0, w_cols = 0, ldw = 0;
  int b_kmajor = 0;
  int w_boff = 0;
  int M = 0, N = 0, K = 0, batch = 1;
  int epi = kEpiBf16;
  float alpha = 1.f;
  void* out = nullptr;
  int ldo = 0;
  long long o_bs = 0;
  int col_group = 0;
  long long group_stride = 0;
  // q|k|v projection of a one-block prefill: columns [0, rope_cols) turned by
  // the token's in-block offset (heads of rope_D columns); columns
  // [ib_col0, ib_col0 + 2 ib_kvd) also stored as in-block rows [Hkv][2][b][ib_D]
  const float2* rope_tab = nullptr;
  int rope_cols = 0, rope_D = 0;
  uint16_t* ib = nullptr;
  int ib_col0 = 0, ib_kvd = 0, ib_D = 0;
  int* err = nullptr;
  bool pdl = false;  // programmatic dependent launch after the previous kernel
};

struct GemmParams {
  CUtensorMap wmap;
  CUtensorMap amap;  // bf16 A as [batch][M][K] (a_bmajor: [M][batch][K]), boxes of 64 columns x 128 rows
  void* out;
  const float2* rope_tab;
  uint16_t* ib;
  long long o_bs, group_stride;
  int ldo, M, N, K;
  int b_kmajor, w_boff, epi, col_group, ks, chunks, a_bmajor;
  int ns, ring_bytes;  // ring stages of this launch and their bytes (set by the launcher)
  int rope_cols, rope_D, ib_col0, ib_kvd, ib_D;
  float alpha;
  int* err;
};

// h [n][d] bf16 = LayerNorm(x [n][d] fp32) * g + b (programmatic dependent
// launch when `pdl`).
cudaError_t launch_layernorm(const float* x, int n, int d, const float* g, const float* b, uint16_t* h, bool pdl,
                             cudaStream_t st);

// Programmatic dependent launch for the layer path's projections and the
// one-block prefill: on unless the environment variable SMEM_PDL is "0"
// (read once per process).
bool pdl_enabled();

struct GemmPlan {
  int bn, ks, ctas;
};
GemmPlan gemm_plan(int M, int N, int K, int batch, int num_sms);
cudaError_t launch_gemm(const GemmCall& g, int num_sms, cudaStream_t st);

// ---------------------------------------------------------------------------
// cross-attention over memory rows (recompute-K/V caches)
// ---------------------------------------------------------------------------
constexpr int kMaxMuGroups = 512;   // groups (row set x query tile) per launch
constexpr int kMuMaxSplits = 16;    // splits of one group's blocks
constexpr int kMuSmemBudget = 220 * 1024;  // one CTA per SM
// One group: NQ queries (rows n0.. of query set qg) that read the same row
// set (the first nblk table blocks of `seq`), cut into nsplit units of
// split_blks blocks; units of a group are consecutive from unit_begin.
struct MuGroup {
  int seq, qg, n0, nblk, split_blks, nsplit, unit_begin, pad;
};
struct MuParams {
  CUtensorMap pool2;          // memory rows [C][d/64 chunks][R][64], box 64 x 2R x 1 (two chunks)
  CUtensorMap pool4;          // the same view, box 64 x 4R x 1 (four chunks; encoded when d/64 % 4 == 0)
  CUtensorMap q;              // Q' [n_qg][nrows][d], box 64 x NQ x 1 (set by the launcher)
  const int* table;           // [max_seqs][max_blocks]
  const uint16_t* qptr;       // Q' (bf16, softmax scale log2(e)/sqrt(d_h) folded in)
  const uint16_t* nu;         // null row [d] or nullptr
  uint16_t* out;              // O' [n_qg][nrows][d] bf16, normalized
  float* part;                // [unit][NQ][d + 4]: m, l, pad, pad, O'[d]
  int* err;
  int d, nrows, n_qg, max_blocks, capacity, n_groups, n_units;
  int ns, nsv, cpb, nsb, off_ring, off_v, off_p, off_bar, off_misc;  // plan (set by the launcher)
  int cl, wsl, off_x;  // column-slice kernel: cluster size, slice width, exchange offset
  MuGroup groups[kMaxMuGroups];
};
// Decode plan of a recompute cache: nq queries per CTA (a multiple of 16,
// covering ceil(H / nq) query tiles per item); cl > 0 selects the
// column-slice kernel on clusters of cl CTAs of wsl = d / cl columns, cl = 0
// the two-pass kernel. A function of H, d and the current device only.
struct MuDecodePlan {
  int nq, cl, wsl;
};
MuDecodePlan mu_decode_plan(int H, int d);
cudaError_t launch_mu_slice(MuParams& P, const MuDecodePlan& pl, cudaStream_t st);
// Widest query tile (16, 32 or 64) for nq_total queries per row set at width
// d whose accumulators fit tensor memory; 0 if none does.
int mu_query_tile(int nq_total, int d);
// Query tile of the one-block form for nblk readable blocks (a function of
// the block count and the geometry only).
int mu_prefill_query_tile(int nblk, int H, int d);
int encode_mu_pool_map(CUtensorMap* map, void* pool, int d, int capacity, int chunks_per_box);
cudaError_t launch_mu_attention(MuParams& P, int nq, cudaStream_t st);
// Split plans (functions of the block count and the cache geometry only).
// A split reads at least kMuMinSplitBlocks blocks: its partial (NQ x d fp32)
// and fixed costs stay small next to the rows it streams.
// A unit pays a fixed start (queries, pipeline fill) and end (its O'
// partial), so splits are at least 24 blocks long; the column-slice kernel
// streams a tile in a fraction of the time of one CTA, so its splits are
// longer still (kMuSliceMinSplitBlocks).
constexpr int kMuMinSplitBlocks = 24;
constexpr int kMuSliceMinSplitBlocks = 32;
SMEM_HD inline int mu_decode_split_blocks(int nblk, int cl) {
  const int s = (nblk + kMuMaxSplits - 1) / kMuMaxSplits;
  const int lo = cl > 0 ? kMuSliceMinSplitBlocks : kMuMinSplitBlocks;
  return s > lo ? s : lo;
}
SMEM_HD inline int mu_prefill_split_blocks(int nblk, int groups) {
  int ns = (304 + groups - 1) / groups;
  if (ns > kMuMaxSplits) ns = kMuMaxSplits;
  const int cap = (nblk + 3) / 4;  // at least 4 blocks per split
  if (ns > cap) ns = cap;
  if (ns < 1) ns = 1;
  return (nblk + ns - 1) / ns;
}

// ---------------------------------------------------------------------------
// prefill
// ---------------------------------------------------------------------------
struct PrefillArgs {
  const CUtensorMap* pool_map;  // pool viewed as [C][L*H*2*R][D], boxes of 64 columns x 64 rows
  const uint16_t* pool;
  const int* table_row;       // slots of this sequence, ascending block index
  const uint16_t* null_kv;    // [L][H][2][D] or nullptr
  const uint16_t *qs, *ks, *vs, *qc;  // [b][H][D]
  uint16_t *osa, *oca;
  float* part;                // [H][pf_max_splits][b][D + 4]: m, l, pad, pad, O[D]
  unsigned* counters;         // [H]
  int* err;
  long long slot_elems;
  int L, H, D, layer, nblk, split_blks, n_splits, capacity;
  int max_blocks;             // table capacity of a sequence (bounds checks)
  int cluster;                // 1: cluster mode (one cluster of n_splits + 1 CTAs per head)
  const float2* rope_tab;     // rotary table or nullptr (Qs/Ks then arrive already turned by offset)
  const int* bidx_row;        // block index of each table entry of this sequence
  int rope_w, q_blk;          // saturating window, the query block's index
  int mode;                   // bit 0: self-attention, bit 1: cross-attention (0: both)
  int tok_s, tok_c;           // elements between tokens of Qs and of Qc (0: H*D)
  int Hkv, tok_kv;            // key/value heads; elements between tokens of Ks/Vs (0: tok_s or Hkv*D)
  float scale_log2;
};
cudaError_t launch_prefill(const PrefillArgs& a, cudaStream_t st);
// Largest cluster size (<= 16) with one cluster per head resident at once on
// the current device for the d_h = 64 prefill; 0 if cluster mode is unavailable.
int prefill_cluster_max(int H, int D);
// Split plan of the d_h = 64 prefill, a function of the block count and the
// head count alone: at most 15 splits, at least two blocks per split, and a
// cluster of splits + 1 CTAs per head within one wave of two CTAs on each of
// a GB300's 152 SMs. The launch runs it as clusters where the device holds
// one such cluster per head and on the cluster-free kernel otherwise; both
// merge the same partials in the same order, so the bits do not depend on
// the device.
SMEM_HD inline int prefill_split_blocks_d64(int nblk, int H) {
  int ns = 304 / H - 1;
  if (ns > 15) ns = 15;
  if (ns > (nblk + 1) / 2) ns = (nblk + 1) / 2;
  if (ns < 1) ns = 1;
  return (nblk + ns - 1) / ns;
}

}  // namespace smem
