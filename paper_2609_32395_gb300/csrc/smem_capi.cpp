// smem_capi.cpp -- the C ABI of include/smem.h: cache geometry, host
// bookkeeping (sorted per-sequence block tables and the free-slot FIFO),
// argument validation and kernel launches.
//
// Bookkeeping follows the memory's definition in arXiv 2609.32395 (Sec. 2
// "Model": the memory is a multiset stored canonically ordered by block
// index; Theorem 1: deleting a block yields exactly the memory in which it
// was never encoded). Every mutating call validates everything first,
// enqueues its device work, and only then commits the host state, so a
// failing call changes nothing.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <deque>
#include <new>
#include <vector>

#include "../../include/smem.h"
#include "smem_internal.h"

using smem::Layout;

struct smem_cache {
  CUtensorMap pool_map{};     // decode kernel's view of the pool (device caches)
  CUtensorMap pool_map_pf{};  // prefill kernel's view (a block's K and V rows of 64 columns per box)
  CUtensorMap pool_map_mu2{};  // memory-row view [C][d/64][R][64], two-chunk boxes (recompute caches)
  CUtensorMap pool_map_mu4{};  // the same, four-chunk boxes (when d/64 is a multiple of 4)
  smem_config cfg{};
  Layout lay{};
  uint8_t* dev = nullptr;  // nullptr: bookkeeping-only
  int device = -1;
  int num_sms = 0;
  std::vector<std::vector<int32_t>> idx;   // per sequence, ascending block index
  std::vector<std::vector<int32_t>> slot;  // per sequence, same order
  std::deque<int32_t> fifo;                // free slots, front = next to use
  std::vector<int32_t> refs;               // table entries naming each slot (0: free)
  std::vector<uint32_t> seen;              // decode: duplicate-sequence check
  uint32_t seen_epoch = 0;
  int fail_after = 0;                      // test hook: n-th next launch fails
  int pf_cluster_max = 0;                  // prefill cluster limit on this device (0: no clusters)
  smem::MuDecodePlan mu_plan{};            // recompute caches: decode kernel and query tile on this device
  // smem_decode_host: which half of the caller's staging buffer the next
  // call uses, and per half the events ordering its copies and its decode
  unsigned host_calls = 0;
  cudaEvent_t ev_in[2]{}, ev_out[2]{}, ev_free[2]{};
  bool ev_made = false;
  // smem_decode_host's input copies (with a separate copy stream): on a
  // stream of their own, so a layer's inputs do not queue behind the
  // previous layer's outputs, which wait for its decode
  cudaStream_t in_stream = nullptr;
  ~smem_cache() {
    if (ev_made)
      for (int i = 0; i < 2; ++i) {
        cudaEventDestroy(ev_in[i]);
        cudaEventDestroy(ev_out[i]);
        cudaEventDestroy(ev_free[i]);
      }
    if (in_stream) cudaStreamDestroy(in_stream);
  }
};

namespace {

thread_local char g_detail[256] = "";

void set_detail(const char* what, cudaError_t e) {
  std::snprintf(g_detail, sizeof(g_detail), "%s: %s", what, cudaGetErrorString(e));
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Geometry of the device buffer; false for an invalid or unsupported config.
int make_layout(const smem_config* c, Layout* L) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (c->n_layers < 1 || c->n_heads < 1 || c->max_seqs < 1 || c->max_blocks_per_seq < 1 || c->capacity_slots < 1 ||
      c->max_decode_batch < 1 || c->max_decode_batch > c->max_seqs)
    return SMEM_ERR_INVALID_ARG;
  if (c->n_layers > 4096 || c->n_heads > 1024 || c->max_seqs > (1 << 20) || c->max_blocks_per_seq > (1 << 22) ||
      c->capacity_slots > (1 << 26))
    return SMEM_ERR_INVALID_ARG;
  if (c->head_dim != 32 && c->head_dim != 64 && c->head_dim != 128) return SMEM_ERR_UNSUPPORTED;
  if (c->block_tokens != smem::kBlockTok || c->rows_per_block != smem::kRows) return SMEM_ERR_UNSUPPORTED;
  if (c->has_null_row != 0 && c->has_null_row != 1) return SMEM_ERR_INVALID_ARG;
  if (c->recompute_kv != 0 && c->recompute_kv != 1) return SMEM_ERR_INVALID_ARG;
  const int hkv = c->n_kv_heads ? c->n_kv_heads : c->n_heads;
  if (hkv < 1 || hkv > c->n_heads || c->n_heads % hkv) return SMEM_ERR_INVALID_ARG;
  if (hkv != c->n_heads && c->recompute_kv) return SMEM_ERR_UNSUPPORTED;
  if (c->rope_window < 0 || c->rope_window >= smem::kRopePhases) return SMEM_ERR_INVALID_ARG;
  if (c->rope_window > 0 && !(c->rope_base > 1.0f && c->rope_base < 1e30f)) return SMEM_ERR_INVALID_ARG;
  if (c->rope_window > 0 && c->recompute_kv) return SMEM_ERR_UNSUPPORTED;
  // recompute caches: rows of d = H*d_h in 128-column pairs, at most 64 heads per query tile
  if (c->recompute_kv && ((c->n_heads * c->head_dim) % 128 != 0 || c->n_heads > 64 ||
                          smem::mu_query_tile(c->n_heads, c->n_heads * c->head_dim) == 0))
    return SMEM_ERR_UNSUPPORTED;
  L->L = c->n_layers;
  L->H = c->n_heads;
  L->D = c->head_dim;
  L->max_seqs = c->max_seqs;
  L->max_blocks = c->max_blocks_per_seq;
  L->capacity = c->capacity_slots;
  L->has_null = c->has_null_row;
  L->max_batch = c->max_decode_batch;
  L->recompute = c->recompute_kv;
  L->Hkv = hkv;
  L->rope_w = c->rope_window;
  L->rope_base = c->rope_base;
  int ms = 1;
  for (int n = 1; n <= c->max_blocks_per_seq; ++n)
    ms = std::max(ms, smem::ceil_div(n, smem::decode_split_blocks(n)));
  L->dec_max_splits = ms;
  L->pf_max_splits = smem::kPrefillMaxSplits;
  const size_t D = (size_t)L->D;
  L->slot_elems = L->recompute ? (size_t)smem::kRows * L->H * D : (size_t)L->L * L->Hkv * 2 * smem::kRows * D;
  size_t off = 0;
  const size_t A = 1024;
  L->off_pool = off;
  off = align_up(off + (size_t)L->capacity * L->slot_elems * 2, A);
  L->off_inblock = off;
  off = align_up(off + (size_t)L->max_seqs * L->L * L->Hkv * 2 * smem::kBlockTok * D * 2, A);
  L->off_null = off;
  off = align_up(off + (!L->has_null ? 0 : L->recompute ? (size_t)L->H * D * 2 : (size_t)L->L * L->Hkv * 2 * D * 2),
                 A);
  L->off_table = off;
  off = align_up(off + (size_t)L->max_seqs * L->max_blocks * 4, A);
  L->off_bidx = off;
  off = align_up(off + (size_t)L->max_seqs * L->max_blocks * 4, A);
  L->off_rope = off;
  off = align_up(off + (L->rope_w ? (size_t)smem::kRopePhases * (D / 2) * 8 : 0), A);
  L->off_rope_scr = off;  // rotated copies of Qs and Ks for smem_prefill_block
  off = align_up(off + (L->rope_w ? (size_t)2 * smem::kBlockTok * L->H * D * 2 : 0), A);
  L->off_dec_part = off;
  off = align_up(off + (size_t)L->max_batch * L->H * L->dec_max_splits * (D + 4) * 4, A);
  L->off_dec_cnt = off;
  off = align_up(off + (size_t)L->max_batch * L->H * 4 + 64, A);  // + unit scheduler words
  L->off_pf_part = off;
  off = align_up(off + (size_t)L->H * L->pf_max_splits * smem::kBlockTok * (D + 4) * 4, A);
  L->off_pf_cnt = off;
  off = align_up(off + (size_t)L->H * 4, A);
  L->off_err = off;
  off = align_up(off + 256, A);
  L->total = off;
  return SMEM_OK;
}

struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) { ok = false; return; }
    if (prev != dev && cudaSetDevice(dev) != cudaSuccess) ok = false;
  }
  ~DeviceGuard() {
    int cur;
    if (ok && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

// Test hook: an injected failure stands in for a failing launch.
bool injected_failure(smem_cache* c) {
  if (c->fail_after <= 0) return false;
  if (--c->fail_after == 0) {
    std::snprintf(g_detail, sizeof(g_detail), "injected launch failure");
    return true;
  }
  return false;
}

int check_launch(smem_cache* c, cudaError_t e, const char* what) {
  (void)c;
  if (e != cudaSuccess) {
    set_detail(what, e);
    return SMEM_ERR_CUDA;
  }
  return SMEM_OK;
}

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }
inline uint16_t* pool_slot(smem_cache* c, int slot) {
  return reinterpret_cast<uint16_t*>(c->dev + c->lay.off_pool) + (size_t)slot * c->lay.slot_elems;
}
inline int* table_row(smem_cache* c, int seq) {
  return reinterpret_cast<int*>(c->dev + c->lay.off_table) + (size_t)seq * c->lay.max_blocks;
}
inline uint16_t* inblock_layer(smem_cache* c, int seq, int layer) {
  const Layout& L = c->lay;
  return reinterpret_cast<uint16_t*>(c->dev + L.off_inblock) +
         ((size_t)seq * L.L + layer) * L.Hkv * 2 * smem::kBlockTok * L.D;
}
inline int* bidx_row(smem_cache* c, int seq) {
  return reinterpret_cast<int*>(c->dev + c->lay.off_bidx) + (size_t)seq * c->lay.max_blocks;
}
inline const float2* rope_tab(smem_cache* c) {
  return c->lay.rope_w ? reinterpret_cast<const float2*>(c->dev + c->lay.off_rope) : nullptr;
}
inline const uint16_t* null_kv(smem_cache* c) {
  return c->lay.has_null ? reinterpret_cast<const uint16_t*>(c->dev + c->lay.off_null) : nullptr;
}

// Workspace of a reader-layer call over n rows (offsets from the caller's
// 256-byte aligned buffer): bf16 h [n][d] (LayerNorm output), qkv [n][3d],
// att [n][d], qc [n][d], g [n][4d]; on a recompute cache also bf16 q' and O'
// [n][H][d] and the split partials of the memory-row attention.
struct LayerWs {
  size_t h, qkv, att, qc, g, qp, op, part, total;
};

LayerWs layer_ws(const Layout& L, int n) {
  const size_t d = (size_t)L.H * L.D;
  LayerWs w{};
  size_t off = 0;
  w.h = off;
  off = align_up(off + (size_t)n * d * 2, 256);
  w.qkv = off;
  off = align_up(off + (size_t)n * 3 * d * 2, 256);
  w.att = off;
  off = align_up(off + (size_t)n * d * 2, 256);
  w.qc = off;
  off = align_up(off + (size_t)n * d * 2, 256);
  w.g = off;
  off = align_up(off + (size_t)n * 4 * d * 2, 256);
  w.qp = w.op = w.part = off;
  if (L.recompute) {
    const int nqd = smem::mu_query_tile(L.H, (int)d);
    w.qp = off;
    off = align_up(off + (size_t)n * L.H * d * 2, 256);
    w.op = off;
    off = align_up(off + (size_t)n * L.H * d * 2, 256);
    w.part = off;
    // decode: at most kMaxMuGroups groups per launch, each item ceil(H / nq)
    // tiles of nq (two-pass) or one tile of H rounded up to 16 (column slices)
    const size_t per_item = std::max((size_t)smem::ceil_div(L.H, nqd) * nqd, (size_t)(L.H + 15) / 16 * 16);
    const size_t rows = std::max((size_t)std::min(n, smem::kMaxMuGroups) * per_item,
                                 n >= smem::kBlockTok ? (size_t)smem::kBlockTok * L.H : (size_t)0);
    off = align_up(off + rows * smem::kMuMaxSplits * (d + 4) * 4, 256);
  }
  w.total = std::max(off, (size_t)256);
  return w;
}

int layer_rows_max(const Layout& L) { return std::max(smem::kBlockTok, L.max_batch); }

// Checks the workspace of a layer call.
int layer_begin(smem_cache* c, void* ws, size_t ws_bytes, int n_rows) {
  if (!ws) return SMEM_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(ws) & 255u) return SMEM_ERR_ALIGN;
  if (ws_bytes < layer_ws(c->lay, n_rows).total) return SMEM_ERR_INVALID_ARG;
  return SMEM_OK;
}

bool ok16(const void* p) { return p && aligned16(p); }

// The fields of one layer's weights a call reads: all (full layer) or only
// the memory key/value maps.
int check_weights(const smem_layer_weights* w, bool full) {
  if (!w) return SMEM_ERR_INVALID_ARG;
  const void* kv[2] = {w->w_kc, w->w_vc};
  for (const void* p : kv)
    if (!p) return SMEM_ERR_INVALID_ARG;
  for (const void* p : kv)
    if (!aligned16(p)) return SMEM_ERR_ALIGN;
  if (!full) return SMEM_OK;
  const void* all[14] = {w->ln1_g, w->ln1_b, w->w_qkv, w->w_os, w->ln2_g, w->ln2_b, w->w_qc,
                         w->w_oc, w->ln3_g, w->ln3_b, w->w_1,  w->w_2,  w->w_kc, w->w_vc};
  for (const void* p : all)
    if (!p) return SMEM_ERR_INVALID_ARG;
  for (const void* p : all)
    if (!aligned16(p)) return SMEM_ERR_ALIGN;
  return SMEM_OK;
}

int cuda_rc(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return SMEM_OK;
  set_detail(what, e);
  return SMEM_ERR_CUDA;
}

// A projection on the library's tensor-core kernel (error word of the cache).
int gemm_rc(smem_cache* c, smem::GemmCall g, cudaStream_t st, const char* what) {
  g.err = reinterpret_cast<int*>(c->dev + c->lay.off_err);
  return cuda_rc(smem::launch_gemm(g, c->num_sms, st), what);
}

// Per-head projection of `rows` memory rows X [rows][d] by a key or value map
// W [d][Hkv*D]: head h of the result, [rows][D] bf16, goes to
// out + h * head_stride (the pool slot's or null row's layout).
int project_heads(smem_cache* c, int rows, const void* X, const void* W, uint16_t* out, long long head_stride,
                  cudaStream_t st) {
  const Layout& L = c->lay;
  const int d = L.H * L.D, kvd = L.Hkv * L.D;
  smem::GemmCall g;
  g.a = X;
  g.lda = d;
  g.w = W;
  g.w_rows = d;
  g.w_cols = kvd;
  g.ldw = kvd;
  g.M = rows;
  g.N = kvd;
  g.K = d;
  g.out = out;
  g.ldo = L.D;
  g.col_group = L.D;
  g.group_stride = head_stride;
  return gemm_rc(c, g, st, "memory-row projection");
}


// One-block attention of one layer (arguments validated by the caller).
// mode bit 0: self-attention, bit 1: cross-attention; tok_s, tok_c: token
// strides (elements) of Qs/Ks/Vs and of Qc, 0 for H*D.
int prefill_impl(smem_cache* c, int seq, int layer, int q_block_idx, const void* Qs, const void* Ks, const void* Vs,
                 const void* Qc, void* Osa, void* Oca, int mode, int tok_s, int tok_c, cudaStream_t st) {
  const std::vector<int32_t>& ix = c->idx[seq];
  const int nblk = (int)(std::lower_bound(ix.begin(), ix.end(), q_block_idx) - ix.begin());
  smem::PrefillArgs a{};
  a.pool_map = &c->pool_map_pf;
  a.pool = reinterpret_cast<const uint16_t*>(c->dev + c->lay.off_pool);
  a.table_row = table_row(c, seq);
  a.null_kv = null_kv(c);
  a.qs = static_cast<const uint16_t*>(Qs);
  a.ks = static_cast<const uint16_t*>(Ks);
  a.vs = static_cast<const uint16_t*>(Vs);
  a.qc = static_cast<const uint16_t*>(Qc);
  a.osa = static_cast<uint16_t*>(Osa);
  a.oca = static_cast<uint16_t*>(Oca);
  a.part = reinterpret_cast<float*>(c->dev + c->lay.off_pf_part);
  a.counters = reinterpret_cast<unsigned*>(c->dev + c->lay.off_pf_cnt);
  a.err = reinterpret_cast<int*>(c->dev + c->lay.off_err);
  a.slot_elems = (long long)c->lay.slot_elems;
  a.L = c->lay.L;
  a.H = c->lay.H;
  a.Hkv = c->lay.Hkv;
  a.D = c->lay.D;
  a.layer = layer;
  a.nblk = nblk;
  if (c->lay.D == 64) {
    // one split plan per (block count, head count), whatever the device; it
    // runs as clusters where the device holds one cluster of splits + 1 CTAs
    // per head, else on the cluster-free kernel with the same splits (same bits)
    a.split_blks = nblk ? smem::prefill_split_blocks_d64(nblk, c->lay.H) : 1;
    a.n_splits = nblk ? smem::ceil_div(nblk, a.split_blks) : 0;
    a.cluster = c->pf_cluster_max >= a.n_splits + 1 && a.n_splits >= 1 ? 1 : 0;
  } else {
    a.cluster = 0;
    a.split_blks = nblk ? smem::prefill_split_blocks(nblk, c->lay.H, c->lay.D) : 1;
    a.n_splits = nblk ? smem::ceil_div(nblk, a.split_blks) : 0;
  }
  a.capacity = c->lay.capacity;
  a.max_blocks = c->lay.max_blocks;
  a.mode = mode;
  a.tok_s = tok_s;
  a.tok_c = tok_c;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c->lay.D));
  a.rope_tab = rope_tab(c);
  a.bidx_row = bidx_row(c, seq);
  a.rope_w = c->lay.rope_w;
  a.q_blk = q_block_idx;
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  return check_launch(c, smem::launch_prefill(a, st), "prefill");
}

// Host-side checks of a decode step (shared by every decode entry point).
int check_decode_args(smem_cache* c, int layer, int nb, const int32_t* seq_ids, const int32_t* pos,
                      const int32_t* q_block_idx) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  const Layout& L = c->lay;
  if (layer < 0 || layer >= L.L || nb < 1 || nb > L.max_batch) return SMEM_ERR_INVALID_ARG;
  if (!seq_ids || !pos || !q_block_idx) return SMEM_ERR_INVALID_ARG;
  if (++c->seen_epoch == 0) {
    std::fill(c->seen.begin(), c->seen.end(), 0u);
    c->seen_epoch = 1;
  }
  for (int i = 0; i < nb; ++i) {
    const int s = seq_ids[i];
    if (s < 0 || s >= L.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
    if (c->seen[s] == c->seen_epoch) return SMEM_ERR_INVALID_ARG;  // one token per sequence per step
    c->seen[s] = c->seen_epoch;
    if (pos[i] < 0 || pos[i] >= smem::kBlockTok || q_block_idx[i] < 0) return SMEM_ERR_INVALID_ARG;
  }
  return SMEM_OK;
}

// One decode step of one layer (arguments validated by the caller). mode as
// in prefill_impl; s_stride, c_stride: elements between items of
// qs/k_new/v_new and of qc. Outputs are [nb][H][D].
int decode_impl(smem_cache* c, int layer, int nb, const int32_t* seq_ids, const int32_t* pos,
                const int32_t* q_block_idx, const void* qs, const void* k_new, const void* v_new, const void* qc,
                void* osa, void* oca, int mode, int s_stride, int c_stride, cudaStream_t st, int kv_stride) {
  const Layout& L = c->lay;
  const size_t tok = (size_t)L.H * L.D;  // output elements per item
  static thread_local smem::DecodeParams P;
  for (int i0 = 0; i0 < nb; i0 += smem::kMaxDecodeItems) {
    const int n = std::min(nb - i0, smem::kMaxDecodeItems);
    P.tmap = c->pool_map;
    P.pool = reinterpret_cast<const uint16_t*>(c->dev + L.off_pool);
    P.inblock = reinterpret_cast<uint16_t*>(c->dev + L.off_inblock);
    P.table = reinterpret_cast<const int*>(c->dev + L.off_table);
    P.null_kv = null_kv(c);
    P.part = reinterpret_cast<float*>(c->dev + L.off_dec_part);
    P.counters = reinterpret_cast<unsigned*>(c->dev + L.off_dec_cnt);
    P.sched = reinterpret_cast<unsigned long long*>(c->dev + L.off_dec_cnt +
                                                    ((size_t)L.max_batch * L.H * 4 + 15) / 16 * 16);
    P.err = reinterpret_cast<int*>(c->dev + L.off_err);
    P.qs = static_cast<const uint16_t*>(qs) + (size_t)i0 * s_stride;
    P.k_new = static_cast<const uint16_t*>(k_new) + (size_t)i0 * kv_stride;
    P.v_new = static_cast<const uint16_t*>(v_new) + (size_t)i0 * kv_stride;
    P.qc = static_cast<const uint16_t*>(qc) + (size_t)i0 * c_stride;
    P.osa = static_cast<uint16_t*>(osa) + i0 * tok;
    P.oca = static_cast<uint16_t*>(oca) + i0 * tok;
    P.slot_elems = (long long)L.slot_elems;
    P.L = L.L;
    P.H = L.H;
    P.layer = layer;
    P.max_blocks = L.max_blocks;
    P.capacity = L.capacity;
    P.n_items = n;
    P.mode = mode;
    P.s_stride = s_stride;
    P.c_stride = c_stride;
    P.Hkv = L.Hkv;
    P.kv_stride = kv_stride;
    P.qn = smem::decode_group_width(L.D, L.H / L.Hkv, L.rope_w != 0);
    P.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)L.D));
    P.rope_tab = rope_tab(c);
    P.bidx = reinterpret_cast<const int*>(c->dev + L.off_bidx);
    P.rope_w = L.rope_w;
    P.max_seqs = L.max_seqs;
    P.part_pairs = (long long)L.max_batch * L.dec_max_splits;
    int pairs = 0;
    for (int i = 0; i < n; ++i) {
      const int s = seq_ids[i0 + i];
      const std::vector<int32_t>& ix = c->idx[s];
      const int nblk = (int)(std::lower_bound(ix.begin(), ix.end(), q_block_idx[i0 + i]) - ix.begin());
      P.items[i].seq = s;
      P.items[i].nblk = nblk;
      P.items[i].pos = pos[i0 + i];
      P.items[i].pair_begin = pairs;
      P.items[i].qblk = q_block_idx[i0 + i];
      if (nblk && (mode & 2)) pairs += smem::ceil_div(nblk, smem::decode_split_blocks(nblk));
    }
    P.n_pairs = pairs;
    const long long units = (long long)pairs * (L.H / P.qn) + (long long)n * L.H;
    const long long wpc = smem::decode_warps_per_cta();
    const int grid = (int)std::min<long long>((units + wpc - 1) / wpc, smem::decode_max_grid(L.D, c->num_sms));
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    const int rc = check_launch(c, smem::launch_decode(P, L.D, grid, st), "decode");
    if (rc) return rc;
  }
  return SMEM_OK;
}

}  // namespace

extern "C" {

size_t smem_cache_required_bytes(const smem_config* cfg) {
  Layout L;
  return make_layout(cfg, &L) == SMEM_OK ? L.total : 0;
}

int smem_cache_create(const smem_config* cfg, void* dev_buf, size_t dev_bytes, smem_cache** out) {
  if (!out) return SMEM_ERR_INVALID_ARG;
  *out = nullptr;
  Layout L;
  int rc = make_layout(cfg, &L);
  if (rc) return rc;
  const bool device = dev_buf != nullptr;
  if (!device && dev_bytes != 0) return SMEM_ERR_INVALID_ARG;
  if (device && (reinterpret_cast<uintptr_t>(dev_buf) & 255u)) return SMEM_ERR_ALIGN;
  if (device && dev_bytes < L.total) return SMEM_ERR_INVALID_ARG;
  std::vector<int32_t> order(L.capacity);
  if (cfg->free_order) {
    std::vector<uint8_t> hit(L.capacity, 0);
    for (int i = 0; i < L.capacity; ++i) {
      const int s = cfg->free_order[i];
      if (s < 0 || s >= L.capacity || hit[s]) return SMEM_ERR_INVALID_ARG;
      hit[s] = 1;
      order[i] = s;
    }
  } else {
    for (int i = 0; i < L.capacity; ++i) order[i] = i;
  }
  smem_cache* c = new (std::nothrow) smem_cache();
  if (!c) return SMEM_ERR_INVALID_ARG;
  c->cfg = *cfg;
  c->cfg.free_order = nullptr;
  c->lay = L;
  c->idx.assign(L.max_seqs, {});
  c->slot.assign(L.max_seqs, {});
  c->fifo.assign(order.begin(), order.end());
  c->refs.assign(L.capacity, 0);
  c->seen.assign(L.max_seqs, 0);
  if (device) {
    c->dev = static_cast<uint8_t*>(dev_buf);
    cudaError_t e = cudaGetDevice(&c->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
    // zero everything but the pool: in-block rows, null rows, tables,
    // workspace, counters and the error word
    if (e == cudaSuccess) e = smem::launch_zero(c->dev + L.off_inblock, L.total - L.off_inblock, nullptr);
    if (e == cudaSuccess && L.rope_w) {
      // rotary table: (cos, sin) of phase * base^(-2m/D), phases 0..63, pairs m < D/2
      std::vector<float> tab((size_t)smem::kRopePhases * L.D);
      for (int ph = 0; ph < smem::kRopePhases; ++ph)
        for (int m = 0; m < L.D / 2; ++m) {
          const double ang = ph * std::pow((double)L.rope_base, -2.0 * m / L.D);
          tab[((size_t)ph * (L.D / 2) + m) * 2] = (float)std::cos(ang);
          tab[((size_t)ph * (L.D / 2) + m) * 2 + 1] = (float)std::sin(ang);
        }
      e = cudaMemcpy(c->dev + L.off_rope, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(nullptr);
    if (e != cudaSuccess) {
      set_detail("create", e);
      delete c;
      return SMEM_ERR_CUDA;
    }
    int er = 0;
    if (L.recompute) {
      er = smem::encode_mu_pool_map(&c->pool_map_mu2, c->dev + L.off_pool, L.H * L.D, L.capacity, 2);
      if (er == 0 && (L.H * L.D / 64) % 4 == 0)
        er = smem::encode_mu_pool_map(&c->pool_map_mu4, c->dev + L.off_pool, L.H * L.D, L.capacity, 4);
    } else {
      er = smem::encode_pool_map(&c->pool_map, c->dev + L.off_pool, L.L, L.Hkv, L.D, L.capacity,
                                 smem::decode_stage_rows(L.D));
      if (er == 0)
        er = smem::encode_pool_map(&c->pool_map_pf, c->dev + L.off_pool, L.L, L.Hkv, L.D, L.capacity,
                                 2 * smem::kRows);  // a block's K rows and V rows in one box
    }
    if (er != 0) {
      std::snprintf(g_detail, sizeof(g_detail), "tensor map encode failed (%d)", er);
      delete c;
      return SMEM_ERR_CUDA;
    }
    const char* knob = std::getenv("SMEM_PREFILL_CLUSTERS");
    c->pf_cluster_max = (knob && knob[0] == '0') ? 0 : smem::prefill_cluster_max(L.H, L.D);
    if (L.recompute) {
      // the column-slice decode kernel is opt-in (SMEM_MU_CLUSTERS=1): at the
      // model shapes its per-slice softmax and cluster exchange cost more
      // than the two-pass kernel's second read of each tile from L2
      const char* mk = std::getenv("SMEM_MU_CLUSTERS");
      c->mu_plan = (mk && mk[0] == '1') ? smem::mu_decode_plan(L.H, L.H * L.D)
                                        : smem::MuDecodePlan{smem::mu_query_tile(L.H, L.H * L.D), 0, 0};
    }
  }
  *out = c;
  return SMEM_OK;
}

int smem_cache_destroy(smem_cache* c) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  delete c;
  return SMEM_OK;
}

int smem_set_null_row(smem_cache* c, const void* k_null, const void* v_null, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
  if (!c->lay.has_null || !k_null || !v_null) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(k_null) || !aligned16(v_null)) return SMEM_ERR_ALIGN;
  DeviceGuard g(c->device);
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  return check_launch(c,
                      smem::launch_null_write(reinterpret_cast<uint16_t*>(c->dev + c->lay.off_null),
                                              static_cast<const uint16_t*>(k_null),
                                              static_cast<const uint16_t*>(v_null), c->lay.L, c->lay.Hkv, c->lay.D,
                                              as_stream(stream)),
                      "null row");
}

int smem_append_block(smem_cache* c, int32_t seq, int32_t block_idx, const void* K, const void* V, void* stream,
                      int32_t* slot_out) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (block_idx < 0) return SMEM_ERR_INVALID_ARG;
  if (c->dev) {
    if (c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
    if (!K || !V) return SMEM_ERR_INVALID_ARG;
    if (!aligned16(K) || !aligned16(V)) return SMEM_ERR_ALIGN;
  } else if (K || V) {
    return SMEM_ERR_NO_DEVICE;
  }
  std::vector<int32_t>& ix = c->idx[seq];
  const auto it = std::lower_bound(ix.begin(), ix.end(), block_idx);
  const int pos = (int)(it - ix.begin());
  if (it != ix.end() && *it == block_idx) return SMEM_ERR_DUPLICATE_BLOCK;
  if ((int)ix.size() >= c->lay.max_blocks) return SMEM_ERR_TABLE_FULL;
  if (c->fifo.empty()) return SMEM_ERR_POOL_FULL;
  const int32_t s = c->fifo.front();
  if (c->dev) {
    DeviceGuard g(c->device);
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    const int rc = check_launch(c,
                                smem::launch_append(pool_slot(c, s), static_cast<const uint16_t*>(K),
                                                    static_cast<const uint16_t*>(V), c->lay.L, c->lay.Hkv, c->lay.D,
                                                    table_row(c, seq), bidx_row(c, seq), pos, (int)ix.size(), s,
                                                    block_idx, as_stream(stream)),
                                "append");
    if (rc) return rc;
  }
  c->fifo.pop_front();
  c->refs[s] = 1;
  ix.insert(ix.begin() + pos, block_idx);
  c->slot[seq].insert(c->slot[seq].begin() + pos, s);
  if (slot_out) *slot_out = s;
  return SMEM_OK;
}

int smem_delete_block(smem_cache* c, int32_t seq, int32_t block_idx, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (block_idx < 0) return SMEM_ERR_INVALID_ARG;
  std::vector<int32_t>& ix = c->idx[seq];
  const auto it = std::lower_bound(ix.begin(), ix.end(), block_idx);
  if (it == ix.end() || *it != block_idx) return SMEM_ERR_NO_SUCH_BLOCK;
  const int pos = (int)(it - ix.begin());
  if (c->dev) {
    DeviceGuard g(c->device);
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    const int rc = check_launch(c, smem::launch_table_remove(table_row(c, seq), bidx_row(c, seq), pos, (int)ix.size(),
                                                              as_stream(stream)),
                                "delete");
    if (rc) return rc;
  }
  const int32_t s = c->slot[seq][pos];
  ix.erase(ix.begin() + pos);
  c->slot[seq].erase(c->slot[seq].begin() + pos);
  if (--c->refs[s] == 0) c->fifo.push_back(s);
  return SMEM_OK;
}

int smem_share_block(smem_cache* c, int32_t src_seq, int32_t src_idx, int32_t dst_seq, int32_t dst_idx,
                     void* stream, int32_t* slot_out) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (src_seq < 0 || src_seq >= c->lay.max_seqs || dst_seq < 0 || dst_seq >= c->lay.max_seqs)
    return SMEM_ERR_NO_SUCH_SEQ;
  if (src_idx < 0 || dst_idx < 0) return SMEM_ERR_INVALID_ARG;
  const std::vector<int32_t>& sx = c->idx[src_seq];
  const auto si = std::lower_bound(sx.begin(), sx.end(), src_idx);
  if (si == sx.end() || *si != src_idx) return SMEM_ERR_NO_SUCH_BLOCK;
  // rows that carry no block position (rotary phases) may be reused at any index
  if (!c->lay.rope_w && dst_idx != src_idx) return SMEM_ERR_INVALID_ARG;
  const int32_t s = c->slot[src_seq][si - sx.begin()];
  std::vector<int32_t>& dx = c->idx[dst_seq];
  const auto di = std::lower_bound(dx.begin(), dx.end(), dst_idx);
  const int pos = (int)(di - dx.begin());
  if (di != dx.end() && *di == dst_idx) return SMEM_ERR_DUPLICATE_BLOCK;
  if ((int)dx.size() >= c->lay.max_blocks) return SMEM_ERR_TABLE_FULL;
  if (c->dev) {
    DeviceGuard g(c->device);
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    const int rc = check_launch(c,
                                smem::launch_table_insert(table_row(c, dst_seq), bidx_row(c, dst_seq), pos,
                                                          (int)dx.size(), s, dst_idx, as_stream(stream)),
                                "share");
    if (rc) return rc;
  }
  dx.insert(dx.begin() + pos, dst_idx);
  c->slot[dst_seq].insert(c->slot[dst_seq].begin() + pos, s);
  ++c->refs[s];
  if (slot_out) *slot_out = s;
  return SMEM_OK;
}

int smem_slot_refs(const smem_cache* c, int32_t slot, int32_t* n_out) {
  if (!c || !n_out || slot < 0 || slot >= c->lay.capacity) return SMEM_ERR_INVALID_ARG;
  *n_out = c->refs[slot];
  return SMEM_OK;
}

int smem_release_seq(smem_cache* c, int32_t seq, void* stream) {
  (void)stream;  // the device row needs no edit: its length lives on the host
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  for (int32_t s : c->slot[seq])
    if (--c->refs[s] == 0) c->fifo.push_back(s);
  c->idx[seq].clear();
  c->slot[seq].clear();
  return SMEM_OK;
}

int smem_write_inblock(smem_cache* c, int32_t seq, int32_t layer, int32_t n_rows, const void* K, const void* V,
                       void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (layer < 0 || layer >= c->lay.L || n_rows < 0 || n_rows > smem::kBlockTok) return SMEM_ERR_INVALID_ARG;
  if (n_rows == 0) return SMEM_OK;
  if (!K || !V) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(V)) return SMEM_ERR_ALIGN;
  DeviceGuard g(c->device);
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  return check_launch(c,
                      smem::launch_inblock_write(inblock_layer(c, seq, layer), static_cast<const uint16_t*>(K),
                                                 static_cast<const uint16_t*>(V), n_rows, c->lay.Hkv, c->lay.D,
                                                 as_stream(stream), 0, rope_tab(c)),
                      "in-block write");
}

int smem_prefill_block(smem_cache* c, int32_t seq, int32_t layer, int32_t q_block_idx, const void* Qs,
                       const void* Ks, const void* Vs, const void* Qc, void* Osa, void* Oca, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (layer < 0 || layer >= c->lay.L || q_block_idx < 0) return SMEM_ERR_INVALID_ARG;
  if (c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
  const void* ptrs[6] = {Qs, Ks, Vs, Qc, Osa, Oca};
  for (const void* p : ptrs) {
    if (!p) return SMEM_ERR_INVALID_ARG;
    if (!aligned16(p)) return SMEM_ERR_ALIGN;
  }
  DeviceGuard g(c->device);
  const cudaStream_t st = as_stream(stream);
  if (c->lay.rope_w) {
    // self-attention queries and keys turn by their in-block offsets first
    const Layout& L = c->lay;
    uint16_t* qr = reinterpret_cast<uint16_t*>(c->dev + L.off_rope_scr);
    uint16_t* kr = qr + (size_t)smem::kBlockTok * L.H * L.D;
    const int tq = L.H * L.D, tk = L.Hkv * L.D;
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    const int rc = check_launch(c, smem::launch_rope_rows(static_cast<const uint16_t*>(Qs), qr, tq, tq, L.H,
                                                          static_cast<const uint16_t*>(Ks), kr, tk, tk, L.Hkv,
                                                          smem::kBlockTok, L.D, rope_tab(c), st),
                                "rotary");
    if (rc) return rc;
    return prefill_impl(c, seq, layer, q_block_idx, qr, kr, Vs, Qc, Osa, Oca, 3, 0, 0, st);
  }
  return prefill_impl(c, seq, layer, q_block_idx, Qs, Ks, Vs, Qc, Osa, Oca, 3, 0, 0, st);
}

int smem_decode(smem_cache* c, int32_t layer, int32_t nb, const int32_t* seq_ids, const int32_t* pos,
                const int32_t* q_block_idx, const void* qs, const void* k_new, const void* v_new, const void* qc,
                void* osa, void* oca, void* stream) {
  const int rc = check_decode_args(c, layer, nb, seq_ids, pos, q_block_idx);
  if (rc) return rc;
  if (c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
  const void* ptrs[6] = {qs, k_new, v_new, qc, osa, oca};
  for (const void* p : ptrs) {
    if (!p) return SMEM_ERR_INVALID_ARG;
    if (!aligned16(p)) return SMEM_ERR_ALIGN;
  }
  DeviceGuard g(c->device);
  const int tok = c->lay.H * c->lay.D;
  return decode_impl(c, layer, nb, seq_ids, pos, q_block_idx, qs, k_new, v_new, qc, osa, oca, 3, tok, tok,
                     as_stream(stream), c->lay.Hkv * c->lay.D);
}

namespace {
// Staging half of smem_decode_host for nb items: qs, k_new, v_new, qc, osa,
// oca, each 256-byte aligned.
struct HostStage {
  size_t qs, kn, vn, qc, osa, oca, half;
};
HostStage host_stage(const Layout& L, int nb) {
  HostStage h{};
  const size_t q = align_up((size_t)nb * L.H * L.D * 2, 256), kv = align_up((size_t)nb * L.Hkv * L.D * 2, 256);
  h.qs = 0;
  h.kn = q;
  h.vn = h.kn + kv;
  h.qc = h.vn + kv;
  h.osa = h.qc + q;
  h.oca = h.osa + q;
  h.half = h.oca + q;
  return h;
}
}  // namespace

size_t smem_decode_host_stage_bytes(const smem_cache* c, int32_t nb) {
  if (!c || nb < 1 || nb > c->lay.max_batch) return 0;
  return 2 * host_stage(c->lay, nb).half;
}

int smem_decode_host(smem_cache* c, int32_t layer, int32_t nb, const int32_t* seq_ids, const int32_t* pos,
                     const int32_t* q_block_idx, const void* qs, const void* k_new, const void* v_new, const void* qc,
                     void* osa, void* oca, void* stage, size_t stage_bytes, void* stream, void* copy_stream) {
  int rc = check_decode_args(c, layer, nb, seq_ids, pos, q_block_idx);
  if (rc) return rc;
  if (c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
  const void* ptrs[7] = {qs, k_new, v_new, qc, osa, oca, stage};
  for (const void* p : ptrs)
    if (!p) return SMEM_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(stage) & 255u) return SMEM_ERR_ALIGN;
  const Layout& L = c->lay;
  const HostStage hs = host_stage(L, nb);
  if (stage_bytes < 2 * hs.half) return SMEM_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  if (!c->ev_made) {
    for (int i = 0; i < 2 && !rc; ++i)
      rc = cuda_rc(cudaEventCreateWithFlags(&c->ev_in[i], cudaEventDisableTiming), "event") ||
           cuda_rc(cudaEventCreateWithFlags(&c->ev_out[i], cudaEventDisableTiming), "event") ||
           cuda_rc(cudaEventCreateWithFlags(&c->ev_free[i], cudaEventDisableTiming), "event");
    if (rc) return SMEM_ERR_CUDA;
    c->ev_made = true;
  }
  const cudaStream_t st = as_stream(stream);
  const cudaStream_t cs = copy_stream ? as_stream(copy_stream) : st;
  if (cs != st && !c->in_stream &&
      cuda_rc(cudaStreamCreateWithFlags(&c->in_stream, cudaStreamNonBlocking), "input stream"))
    return SMEM_ERR_CUDA;
  // inputs: on the library's input stream (outputs on the copy stream)
  const cudaStream_t is = cs != st ? c->in_stream : st;
  const int half = (int)(c->host_calls & 1u);
  uint8_t* b = static_cast<uint8_t*>(stage) + (size_t)half * hs.half;
  const size_t qb = (size_t)nb * L.H * L.D * 2, kvb = (size_t)nb * L.Hkv * L.D * 2;
  // inputs in once this half's previous outputs are out
  cudaError_t e = cudaSuccess;
  if (cs != st && c->host_calls >= 2) e = cudaStreamWaitEvent(is, c->ev_free[half], 0);
  if (e == cudaSuccess) e = cudaMemcpyAsync(b + hs.qs, qs, qb, cudaMemcpyHostToDevice, is);
  if (e == cudaSuccess) e = cudaMemcpyAsync(b + hs.kn, k_new, kvb, cudaMemcpyHostToDevice, is);
  if (e == cudaSuccess) e = cudaMemcpyAsync(b + hs.vn, v_new, kvb, cudaMemcpyHostToDevice, is);
  if (e == cudaSuccess) e = cudaMemcpyAsync(b + hs.qc, qc, qb, cudaMemcpyHostToDevice, is);
  if (e == cudaSuccess && cs != st) e = cudaEventRecord(c->ev_in[half], is);
  if (e == cudaSuccess && cs != st) e = cudaStreamWaitEvent(st, c->ev_in[half], 0);
  if (e != cudaSuccess) return cuda_rc(e, "host decode inputs");
  const int tok = L.H * L.D;
  rc = decode_impl(c, layer, nb, seq_ids, pos, q_block_idx, b + hs.qs, b + hs.kn, b + hs.vn, b + hs.qc, b + hs.osa,
                   b + hs.oca, 3, tok, tok, st, L.Hkv * L.D);
  if (rc) return rc;
  // outputs out on the copy stream after the decode
  if (cs != st) e = cudaEventRecord(c->ev_out[half], st);
  if (e == cudaSuccess && cs != st) e = cudaStreamWaitEvent(cs, c->ev_out[half], 0);
  if (e == cudaSuccess) e = cudaMemcpyAsync(osa, b + hs.osa, qb, cudaMemcpyDeviceToHost, cs);
  if (e == cudaSuccess) e = cudaMemcpyAsync(oca, b + hs.oca, qb, cudaMemcpyDeviceToHost, cs);
  if (e == cudaSuccess && cs != st) e = cudaEventRecord(c->ev_free[half], cs);
  if (e != cudaSuccess) return cuda_rc(e, "host decode outputs");
  ++c->host_calls;
  return SMEM_OK;
}

int smem_decode_static_scratch(smem_cache* c, int32_t layer, int32_t nb, const int32_t* seq_ids, const int32_t* pos,
                               const int32_t* q_block_idx, const void* qs, const void* k_new, const void* v_new,
                               const void* qc, void* osa, void* oca, void* stream) {
  // Same validation as smem_decode; the split-K scratch comes from the
  // library's fixed array instead of the cache's workspace.
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  const Layout& L = c->lay;
  if (L.recompute) return SMEM_ERR_UNSUPPORTED;
  if (layer < 0 || layer >= L.L || nb < 1 || nb > L.max_batch) return SMEM_ERR_INVALID_ARG;
  if (!seq_ids || !pos || !q_block_idx) return SMEM_ERR_INVALID_ARG;
  const void* ptrs[6] = {qs, k_new, v_new, qc, osa, oca};
  for (const void* p : ptrs) {
    if (!p) return SMEM_ERR_INVALID_ARG;
    if (!aligned16(p)) return SMEM_ERR_ALIGN;
  }
  if (++c->seen_epoch == 0) {
    std::fill(c->seen.begin(), c->seen.end(), 0u);
    c->seen_epoch = 1;
  }
  std::vector<int> nblk(nb);
  for (int i = 0; i < nb; ++i) {
    const int s = seq_ids[i];
    if (s < 0 || s >= L.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
    if (c->seen[s] == c->seen_epoch) return SMEM_ERR_INVALID_ARG;
    c->seen[s] = c->seen_epoch;
    if (pos[i] < 0 || pos[i] >= smem::kBlockTok || q_block_idx[i] < 0) return SMEM_ERR_INVALID_ARG;
    const std::vector<int32_t>& ix = c->idx[s];
    nblk[i] = (int)(std::lower_bound(ix.begin(), ix.end(), q_block_idx[i]) - ix.begin());
  }
  const int qn = smem::decode_group_width(L.D, L.H / L.Hkv, L.rope_w != 0);  // the units smem_decode runs
  // scratch layout per launch: [256 B scheduler words][tickets][partials]
  const size_t ticket_bytes = align_up((size_t)std::min(nb, smem::kMaxDecodeItems) * L.H * 4, 256);
  size_t need = 0;
  for (int i0 = 0; i0 < nb; i0 += smem::kMaxDecodeItems) {
    const int n = std::min(nb - i0, smem::kMaxDecodeItems);
    size_t pairs = 0;
    for (int i = 0; i < n; ++i)
      if (nblk[i0 + i]) pairs += smem::ceil_div(nblk[i0 + i], smem::decode_split_blocks(nblk[i0 + i]));
    need = std::max(need, 256 + ticket_bytes + pairs * L.H * (L.D + 4) * 4);
  }
  if (need > SMEM_STATIC_SCRATCH_BYTES) {
    std::snprintf(g_detail, sizeof(g_detail), "decode needs %zu bytes of scratch, the fixed array holds %u", need,
                  SMEM_STATIC_SCRATCH_BYTES);
    return SMEM_ERR_SCRATCH_LIMIT;
  }
  DeviceGuard g(c->device);
  void* scratch = nullptr;
  const int se = smem::static_scratch_address(&scratch);
  if (se != 0) return check_launch(c, (cudaError_t)se, "static scratch address");
  uint8_t* sb = static_cast<uint8_t*>(scratch);
  const size_t tok = (size_t)L.H * L.D;
  static thread_local smem::DecodeParams P;
  for (int i0 = 0; i0 < nb; i0 += smem::kMaxDecodeItems) {
    const int n = std::min(nb - i0, smem::kMaxDecodeItems);
    P.tmap = c->pool_map;
    P.pool = reinterpret_cast<const uint16_t*>(c->dev + L.off_pool);
    P.inblock = reinterpret_cast<uint16_t*>(c->dev + L.off_inblock);
    P.table = reinterpret_cast<const int*>(c->dev + L.off_table);
    P.null_kv = null_kv(c);
    P.sched = reinterpret_cast<unsigned long long*>(sb);
    P.counters = reinterpret_cast<unsigned*>(sb + 256);
    P.part = reinterpret_cast<float*>(sb + 256 + ticket_bytes);
    P.err = reinterpret_cast<int*>(c->dev + L.off_err);
    P.qs = static_cast<const uint16_t*>(qs) + i0 * tok;
    P.k_new = static_cast<const uint16_t*>(k_new) + (size_t)i0 * L.Hkv * L.D;
    P.v_new = static_cast<const uint16_t*>(v_new) + (size_t)i0 * L.Hkv * L.D;
    P.qc = static_cast<const uint16_t*>(qc) + i0 * tok;
    P.osa = static_cast<uint16_t*>(osa) + i0 * tok;
    P.oca = static_cast<uint16_t*>(oca) + i0 * tok;
    P.slot_elems = (long long)L.slot_elems;
    P.L = L.L;
    P.H = L.H;
    P.layer = layer;
    P.max_blocks = L.max_blocks;
    P.capacity = L.capacity;
    P.n_items = n;
    P.mode = 3;
    P.s_stride = P.c_stride = L.H * L.D;
    P.Hkv = L.Hkv;
    P.kv_stride = L.Hkv * L.D;
    P.qn = qn;
    P.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)L.D));
    P.rope_tab = rope_tab(c);
    P.bidx = reinterpret_cast<const int*>(c->dev + L.off_bidx);
    P.rope_w = L.rope_w;
    P.max_seqs = L.max_seqs;
    P.part_pairs = (long long)((SMEM_STATIC_SCRATCH_BYTES - 256 - ticket_bytes) / ((size_t)L.H * (L.D + 4) * 4));
    int pairs = 0;
    for (int i = 0; i < n; ++i) {
      P.items[i].seq = seq_ids[i0 + i];
      P.items[i].nblk = nblk[i0 + i];
      P.items[i].pos = pos[i0 + i];
      P.items[i].pair_begin = pairs;
      P.items[i].qblk = q_block_idx[i0 + i];
      if (nblk[i0 + i]) pairs += smem::ceil_div(nblk[i0 + i], smem::decode_split_blocks(nblk[i0 + i]));
    }
    P.n_pairs = pairs;
    const long long units = (long long)pairs * (L.H / P.qn) + (long long)n * L.H;
    const long long wpc = smem::decode_warps_per_cta();
    const int grid = (int)std::min<long long>((units + wpc - 1) / wpc, smem::decode_max_grid(L.D, c->num_sms));
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    // the array keeps the previous call's contents: clear the scheduler
    // words and tickets this launch needs at zero
    int rc = check_launch(c, smem::launch_zero(sb, 256 + ticket_bytes, as_stream(stream)), "static scratch clear");
    if (rc) return rc;
    rc = check_launch(c, smem::launch_decode(P, L.D, grid, as_stream(stream)), "decode (static scratch)");
    if (rc) return rc;
  }
  return SMEM_OK;
}

// ---------------------------------------------------------------------------
// reader layer
// ---------------------------------------------------------------------------
size_t smem_layer_workspace_bytes(const smem_cache* c, int32_t n_rows) {
  if (!c || n_rows < 0 || n_rows > layer_rows_max(c->lay)) return 0;
  return layer_ws(c->lay, n_rows).total;
}

int smem_append_block_rows(smem_cache* c, int32_t seq, int32_t block_idx, const void* mu,
                           const smem_layer_weights* w, void* ws, size_t ws_bytes, void* stream, int32_t* slot_out) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (block_idx < 0 || !mu || (!w && !c->lay.recompute)) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(mu)) return SMEM_ERR_ALIGN;
  const Layout& L = c->lay;
  for (int l = 0; l < L.L && !L.recompute; ++l) {
    const int rc = check_weights(&w[l], false);
    if (rc) return rc;
  }
  std::vector<int32_t>& ix = c->idx[seq];
  const auto it = std::lower_bound(ix.begin(), ix.end(), block_idx);
  const int pos = (int)(it - ix.begin());
  if (it != ix.end() && *it == block_idx) return SMEM_ERR_DUPLICATE_BLOCK;
  if ((int)ix.size() >= L.max_blocks) return SMEM_ERR_TABLE_FULL;
  if (c->fifo.empty()) return SMEM_ERR_POOL_FULL;
  DeviceGuard g(c->device);
  const cudaStream_t st = as_stream(stream);
  int rc = layer_begin(c, ws, ws_bytes, 0);
  if (rc) return rc;
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  const int32_t s = c->fifo.front();
  // the slot is still free: a failure below leaves only a free slot's rows written
  uint16_t* slot = pool_slot(c, s);
  const int d = L.H * L.D;
  const size_t head_stride = (size_t)2 * smem::kRows * L.D;
  if (L.recompute)  // the slot keeps the memory rows themselves, one 64-column chunk after another
    rc = cuda_rc(smem::launch_mu_tile(slot, static_cast<const uint16_t*>(mu), d, st), "append rows");
  for (int l = 0; l < L.L && !rc && !L.recompute; ++l)
    for (int kv = 0; kv < 2 && !rc; ++kv)
      rc = project_heads(c, smem::kRows, mu, kv ? w[l].w_vc : w[l].w_kc,
                         slot + ((size_t)l * L.Hkv * 2 + kv) * smem::kRows * L.D, (long long)head_stride, st);
  if (!rc) rc = cuda_rc(smem::launch_table_insert(table_row(c, seq), bidx_row(c, seq), pos, (int)ix.size(), s,
                                                          block_idx, st), "append rows");
  if (rc) return rc;
  c->fifo.pop_front();
  c->refs[s] = 1;
  ix.insert(ix.begin() + pos, block_idx);
  c->slot[seq].insert(c->slot[seq].begin() + pos, s);
  if (slot_out) *slot_out = s;
  return SMEM_OK;
}

int smem_set_null_vector(smem_cache* c, const void* nu, const smem_layer_weights* w, void* ws, size_t ws_bytes,
                         void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  const Layout& L = c->lay;
  if (!L.has_null || !nu || (!w && !L.recompute)) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(nu)) return SMEM_ERR_ALIGN;
  for (int l = 0; l < L.L && !L.recompute; ++l) {
    const int rc = check_weights(&w[l], false);
    if (rc) return rc;
  }
  DeviceGuard g(c->device);
  int rc = layer_begin(c, ws, ws_bytes, 0);
  if (rc) return rc;
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  uint16_t* nk = reinterpret_cast<uint16_t*>(c->dev + L.off_null);
  const int d = L.H * L.D;
  if (L.recompute)
    return cuda_rc(cudaMemcpyAsync(nk, nu, (size_t)d * 2, cudaMemcpyDeviceToDevice, as_stream(stream)), "null vector");
  for (int l = 0; l < L.L && !rc; ++l)
    for (int kv = 0; kv < 2 && !rc; ++kv)
      rc = project_heads(c, 1, nu, kv ? w[l].w_vc : w[l].w_kc, nk + ((size_t)l * L.Hkv * 2 + kv) * L.D,
                         (long long)2 * L.D, as_stream(stream));
  return rc;
}

namespace {

// The dense tail shared by prefill and decode layers: after the attention
// outputs are in place, x += att W_o etc. Steps are issued in the layer's
// order on one stream.
struct LayerRun {
  smem_cache* c;
  const smem_layer_weights* w;
  float* x;
  uint8_t* ws;
  LayerWs o;
  int n, d;
  cudaStream_t st;
  int kvd() const { return c->lay.Hkv * c->lay.D; }  // key (or value) width of a token
  int w3() const { return d + 2 * kvd(); }            // q|k|v width of a token
  uint16_t* h() const { return reinterpret_cast<uint16_t*>(ws + o.h); }
  uint16_t* qkv() const { return reinterpret_cast<uint16_t*>(ws + o.qkv); }
  uint16_t* att() const { return reinterpret_cast<uint16_t*>(ws + o.att); }
  uint16_t* qc() const { return reinterpret_cast<uint16_t*>(ws + o.qc); }
  uint16_t* g() const { return reinterpret_cast<uint16_t*>(ws + o.g); }
  // h = LN(x) with this gain and bias (bf16)
  int ln(const float* gain, const float* bias) {
    return cuda_rc(smem::launch_layernorm(x, n, d, gain, bias, h(), true, st), "layernorm");
  }
  // out = A W over this call's n tokens (A bf16 [n][k])
  smem::GemmCall proj(const void* A, const void* W, int cols, int k, void* out, int epi) const {
    smem::GemmCall g;
    g.a = A;
    g.lda = k;
    g.w = W;
    g.w_rows = k;
    g.w_cols = cols;
    g.ldw = cols;
    g.M = n;
    g.N = cols;
    g.K = k;
    g.epi = epi;
    g.out = out;
    g.ldo = cols;
    g.pdl = true;
    return g;
  }
  // qkv = LN1(x) W_qkv; for a one-block prefill (ib set) the key/value
  // columns also become the block's in-block rows, and with rotary phases
  // the query and key columns turn by the token's offset first
  int qkv_proj(uint16_t* ib) {
    int rc = ln(w->ln1_g, w->ln1_b);
    if (rc) return rc;
    smem::GemmCall g = proj(h(), w->w_qkv, w3(), d, qkv(), smem::kEpiBf16);
    if (ib) {
      g.ib = ib;
      g.ib_col0 = d;
      g.ib_kvd = kvd();
      g.ib_D = c->lay.D;
      if (c->lay.rope_w) {
        g.rope_tab = rope_tab(c);
        g.rope_cols = d + kvd();
        g.rope_D = c->lay.D;
      }
    }
    return gemm_rc(c, g, st, "qkv projection");
  }
  // x += att W_os; qc = LN2(x) W_qc
  int after_sa() {
    int rc = gemm_rc(c, proj(att(), w->w_os, d, d, x, smem::kEpiAddF32), st, "output projection");
    if (!rc) rc = ln(w->ln2_g, w->ln2_b);
    return rc ? rc : gemm_rc(c, proj(h(), w->w_qc, d, d, qc(), smem::kEpiBf16), st, "cross-attention query projection");
  }
  // x += att W_oc; x += GELU(LN3(x) W_1) W_2
  int after_ca() {
    int rc = gemm_rc(c, proj(att(), w->w_oc, d, d, x, smem::kEpiAddF32), st, "output projection");
    if (!rc) rc = ln(w->ln3_g, w->ln3_b);
    if (!rc) rc = gemm_rc(c, proj(h(), w->w_1, 4 * d, d, g(), smem::kEpiGeluBf16), st, "FFN");
    return rc ? rc : gemm_rc(c, proj(g(), w->w_2, d, 4 * d, x, smem::kEpiAddF32), st, "FFN");
  }
};

// The memory-row attention launch(es): O' of every query in qp (prefill:
// [H][b][d], one row set; decode: [nb][H][d], one row set per item).
int mu_attend(smem_cache* c, uint8_t* ws, const LayerWs& o, bool prefill, int nb, const int32_t* seq_ids,
              const int32_t* q_block_idx, int seq, int q_idx, const uint16_t* qp, uint16_t* op, cudaStream_t st) {
  const Layout& L = c->lay;
  const int d = L.H * L.D, H = L.H;
  int rc = SMEM_OK;
  static thread_local smem::MuParams P;
  P.pool2 = c->pool_map_mu2;
  P.pool4 = c->pool_map_mu4;
  P.table = reinterpret_cast<const int*>(c->dev + L.off_table);
  P.nu = L.has_null ? reinterpret_cast<const uint16_t*>(c->dev + L.off_null) : nullptr;
  P.part = reinterpret_cast<float*>(ws + o.part);
  P.err = reinterpret_cast<int*>(c->dev + L.off_err);
  P.d = d;
  P.max_blocks = L.max_blocks;
  P.capacity = L.capacity;
  if (prefill) {
    const std::vector<int32_t>& ix = c->idx[seq];
    const int nblk = (int)(std::lower_bound(ix.begin(), ix.end(), q_idx) - ix.begin());
    const int nqt = smem::mu_prefill_query_tile(nblk, H, d);
    const int tiles = smem::kBlockTok / nqt;
    const int groups = H * tiles;
    const int sb = nblk ? smem::mu_prefill_split_blocks(nblk, groups) : 1;
    const int nsplit = nblk ? smem::ceil_div(nblk, sb) : 1;
    P.qptr = qp;
    P.out = op;
    P.nrows = smem::kBlockTok;
    P.n_qg = H;
    P.n_groups = groups;
    int u = 0;
    for (int h = 0; h < H; ++h)
      for (int t = 0; t < tiles; ++t) {
        smem::MuGroup& G = P.groups[h * tiles + t];
        G = {seq, h, t * nqt, nblk, sb, nsplit, u, 0};
        u += nsplit;
      }
    P.n_units = u;
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    rc = cuda_rc(smem::launch_mu_attention(P, nqt, st), "memory-row attention");
  } else {
    // one group per (item, tile of nq heads); the column-slice kernel when planned
    const smem::MuDecodePlan& pl = c->mu_plan;
    const int nqt = pl.nq;
    const int qtiles = smem::ceil_div(H, nqt);
    const int per_launch = smem::kMaxMuGroups / qtiles;
    for (int i0 = 0; i0 < nb && !rc; i0 += per_launch) {
      const int n = std::min(nb - i0, per_launch);
      P.qptr = qp + (size_t)i0 * H * d;
      P.out = op + (size_t)i0 * H * d;
      P.nrows = H;
      P.n_qg = n;
      P.n_groups = n * qtiles;
      int u = 0;
      for (int i = 0; i < n; ++i) {
        const std::vector<int32_t>& ix = c->idx[seq_ids[i0 + i]];
        const int nblk = (int)(std::lower_bound(ix.begin(), ix.end(), q_block_idx[i0 + i]) - ix.begin());
        const int sb = nblk ? smem::mu_decode_split_blocks(nblk, pl.cl) : 1;
        const int nsplit = nblk ? smem::ceil_div(nblk, sb) : 1;
        for (int q = 0; q < qtiles; ++q) {
          P.groups[i * qtiles + q] = {seq_ids[i0 + i], i, q * nqt, nblk, sb, nsplit, u, 0};
          u += nsplit;
        }
      }
      P.n_units = u;
      if (injected_failure(c)) return SMEM_ERR_CUDA;
      rc = cuda_rc(pl.cl > 0 ? smem::launch_mu_slice(P, pl, st) : smem::launch_mu_attention(P, nqt, st),
                   "memory-row attention");
    }
  }
  return rc;
}

// Cross-attention of a layer call on a recompute cache (the memory rows mu
// in the pool): q'_h = scale W_kc,h q_h, O'_h = attention of q'_h over the
// rows, att_h = O'_h W_vc,h. Prefill: one row set, groups (head, query
// tile); decode: one group per sequence holding all its heads.
int mu_cross_attention(LayerRun& r, int layer, int nb, const int32_t* seq_ids, const int32_t* q_block_idx,
                       bool prefill, int seq, int q_idx) {
  smem_cache* c = r.c;
  const Layout& L = c->lay;
  const int d = r.d, H = L.H, D = L.D;
  const float scale = (float)(1.4426950408889634 / std::sqrt((double)D));
  const uint16_t* wkc = static_cast<const uint16_t*>(r.w->w_kc);
  const uint16_t* wvc = static_cast<const uint16_t*>(r.w->w_vc);
  uint16_t* qp = reinterpret_cast<uint16_t*>(r.ws + r.o.qp);
  uint16_t* op = reinterpret_cast<uint16_t*>(r.ws + r.o.op);
  const int nq = prefill ? smem::kBlockTok : nb;  // queries per head
  // q'[.][h][i] = scale sum_j qc[.][h][j] W_kc[i][h D + j]; prefill stores [h][q][d], decode [s][h][d]
  smem::GemmCall g;
  g.a = r.qc();
  g.lda = d;
  g.a_bs = D;
  g.w = wkc;
  g.w_rows = d;
  g.w_cols = d;
  g.ldw = d;
  g.b_kmajor = 1;
  g.w_boff = D;
  g.M = nq;
  g.N = d;
  g.K = D;
  g.batch = H;
  g.alpha = scale;
  g.out = qp;
  g.ldo = prefill ? d : H * d;
  g.o_bs = prefill ? (long long)smem::kBlockTok * d : d;
  g.pdl = true;
  int rc = gemm_rc(c, g, r.st, "memory-row query map");
  if (rc) return rc;
  rc = mu_attend(c, r.ws, r.o, prefill, nb, seq_ids, q_block_idx, seq, q_idx, qp, op, r.st);
  if (rc) return rc;
  // att[.][h][e] = sum_i O'[h-row][i] W_vc[i][h D + e]
  smem::GemmCall v;
  v.a = op;
  v.lda = prefill ? d : H * d;
  v.a_bs = prefill ? (long long)smem::kBlockTok * d : d;
  v.w = wvc;
  v.w_rows = d;
  v.w_cols = d;
  v.ldw = d;
  v.w_boff = D;
  v.M = nq;
  v.N = D;
  v.K = d;
  v.batch = H;
  v.out = r.att();
  v.ldo = d;
  v.o_bs = D;
  v.pdl = true;
  return gemm_rc(c, v, r.st, "memory-row value map");
}

}  // namespace

int smem_reader_layer_prefill(smem_cache* c, int32_t seq, int32_t layer, int32_t q_block_idx,
                              const smem_layer_weights* w, float* x, void* ws, size_t ws_bytes, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (layer < 0 || layer >= c->lay.L || q_block_idx < 0 || !x) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(x)) return SMEM_ERR_ALIGN;
  int rc = check_weights(w, true);
  if (rc) return rc;
  DeviceGuard g(c->device);
  const cudaStream_t st = as_stream(stream);
  const int n = smem::kBlockTok;
  rc = layer_begin(c, ws, ws_bytes, n);
  if (rc) return rc;
  const Layout& L = c->lay;
  LayerRun r{c, w, x, static_cast<uint8_t*>(ws), layer_ws(L, n), n, L.H * L.D, st};
  const int d = r.d, kvd = r.kvd(), w3 = r.w3();
  // q|k|v of the block; its self-attention keys/values also become its
  // in-block rows, queries and keys turned by their offsets with rotary phases
  rc = r.qkv_proj(inblock_layer(c, seq, layer));
  if (!rc)
    rc = prefill_impl(c, seq, layer, q_block_idx, r.qkv(), r.qkv() + d, r.qkv() + d + kvd, r.qkv(), r.att(), r.att(),
                      1, w3, w3, st);
  if (!rc) rc = r.after_sa();
  if (!rc) {
    if (L.recompute)
      rc = mu_cross_attention(r, layer, 0, nullptr, nullptr, true, seq, q_block_idx);
    else
      rc = prefill_impl(c, seq, layer, q_block_idx, r.qc(), r.qc(), r.qc(), r.qc(), r.att(), r.att(), 2, d, d, st);
  }
  if (!rc) rc = r.after_ca();
  return rc;
}

int smem_reader_layer_decode(smem_cache* c, int32_t layer, int32_t nb, const int32_t* seq_ids, const int32_t* pos,
                             const int32_t* q_block_idx, const smem_layer_weights* w, float* x, void* ws,
                             size_t ws_bytes, void* stream) {
  int rc = check_decode_args(c, layer, nb, seq_ids, pos, q_block_idx);
  if (rc) return rc;
  if (!x) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(x)) return SMEM_ERR_ALIGN;
  rc = check_weights(w, true);
  if (rc) return rc;
  DeviceGuard g(c->device);
  const cudaStream_t st = as_stream(stream);
  rc = layer_begin(c, ws, ws_bytes, nb);
  if (rc) return rc;
  const Layout& L = c->lay;
  LayerRun r{c, w, x, static_cast<uint8_t*>(ws), layer_ws(L, nb), nb, L.H * L.D, st};
  const int d = r.d, kvd = r.kvd(), w3 = r.w3();
  rc = r.qkv_proj(nullptr);
  if (!rc)
    rc = decode_impl(c, layer, nb, seq_ids, pos, q_block_idx, r.qkv(), r.qkv() + d, r.qkv() + d + kvd, r.qkv(),
                     r.att(), r.att(), 1, w3, w3, st, w3);
  if (!rc) rc = r.after_sa();
  if (!rc) {
    if (L.recompute)
      rc = mu_cross_attention(r, layer, nb, seq_ids, q_block_idx, false, 0, 0);
    else
      rc = decode_impl(c, layer, nb, seq_ids, pos, q_block_idx, r.qc(), r.qc(), r.qc(), r.qc(), r.att(), r.att(), 2,
                       d, d, st, d);
  }
  if (!rc) rc = r.after_ca();
  return rc;
}

int smem_mu_decode(smem_cache* c, int32_t nb, const int32_t* seq_ids, const int32_t* q_block_idx, const void* qp,
                   void* op, void* ws, size_t ws_bytes, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (!c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
  if (nb < 1 || nb > c->lay.max_batch || !seq_ids || !q_block_idx || !qp || !op) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(qp) || !aligned16(op)) return SMEM_ERR_ALIGN;
  if (++c->seen_epoch == 0) {
    std::fill(c->seen.begin(), c->seen.end(), 0u);
    c->seen_epoch = 1;
  }
  for (int i = 0; i < nb; ++i) {
    const int s = seq_ids[i];
    if (s < 0 || s >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
    if (c->seen[s] == c->seen_epoch || q_block_idx[i] < 0) return SMEM_ERR_INVALID_ARG;
    c->seen[s] = c->seen_epoch;
  }
  DeviceGuard g(c->device);
  const cudaStream_t st = as_stream(stream);
  const int rc = layer_begin(c, ws, ws_bytes, nb);
  if (rc) return rc;
  return mu_attend(c, static_cast<uint8_t*>(ws), layer_ws(c->lay, nb), false, nb, seq_ids, q_block_idx, 0, 0,
                   static_cast<const uint16_t*>(qp), static_cast<uint16_t*>(op), st);
}

int smem_mu_prefill(smem_cache* c, int32_t seq, int32_t q_block_idx, const void* qp, void* op, void* ws,
                    size_t ws_bytes, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (!c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (q_block_idx < 0 || !qp || !op) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(qp) || !aligned16(op)) return SMEM_ERR_ALIGN;
  DeviceGuard g(c->device);
  const cudaStream_t st = as_stream(stream);
  const int rc = layer_begin(c, ws, ws_bytes, smem::kBlockTok);
  if (rc) return rc;
  return mu_attend(c, static_cast<uint8_t*>(ws), layer_ws(c->lay, smem::kBlockTok), true, 0, nullptr, nullptr, seq,
                   q_block_idx, static_cast<const uint16_t*>(qp), static_cast<uint16_t*>(op), st);
}

int smem_get_table(const smem_cache* c, int32_t seq, int32_t* idx_out, int32_t* slot_out, int32_t cap,
                   int32_t* n_out) {
  if (!c || !n_out || cap < 0) return SMEM_ERR_INVALID_ARG;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  const int n = (int)c->idx[seq].size();
  *n_out = n;
  const int m = std::min(n, (int)cap);
  for (int i = 0; i < m; ++i) {
    if (idx_out) idx_out[i] = c->idx[seq][i];
    if (slot_out) slot_out[i] = c->slot[seq][i];
  }
  return SMEM_OK;
}

int smem_get_free_fifo(const smem_cache* c, int32_t* slots_out, int32_t cap, int32_t* n_out) {
  if (!c || !n_out || cap < 0) return SMEM_ERR_INVALID_ARG;
  const int n = (int)c->fifo.size();
  *n_out = n;
  const int m = std::min(n, (int)cap);
  for (int i = 0; i < m && slots_out; ++i) slots_out[i] = c->fifo[i];
  return SMEM_OK;
}

int smem_get_device_table(smem_cache* c, int32_t seq, int32_t* slot_out, int32_t cap, int32_t* n_out, void* stream) {
  if (!c || !n_out || cap < 0) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  const int n = (int)c->idx[seq].size();
  *n_out = n;
  const int m = std::min(n, (int)cap);
  if (m == 0 || !slot_out) return SMEM_OK;
  DeviceGuard g(c->device);
  cudaError_t e = cudaMemcpyAsync(slot_out, table_row(c, seq), (size_t)m * 4, cudaMemcpyDeviceToHost, as_stream(stream));
  if (e == cudaSuccess) e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) {
    set_detail("device table read", e);
    return SMEM_ERR_CUDA;
  }
  return SMEM_OK;
}

int smem_check_device_error(smem_cache* c, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  DeviceGuard g(c->device);
  int word = 0;
  int* dev_err = reinterpret_cast<int*>(c->dev + c->lay.off_err);
  cudaError_t e = cudaMemcpyAsync(&word, dev_err, sizeof(int), cudaMemcpyDeviceToHost, as_stream(stream));
  if (e == cudaSuccess) e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) {
    set_detail("error word read", e);
    return SMEM_ERR_CUDA;
  }
  if (word == 0) return SMEM_OK;
  std::snprintf(g_detail, sizeof(g_detail), "device error code %d", word);
  // clear the word and the split counters an aborted launch may have left
  const Layout& L = c->lay;
  e = smem::launch_zero(c->dev + L.off_dec_cnt, L.off_pf_part - L.off_dec_cnt, as_stream(stream));
  if (e == cudaSuccess) e = smem::launch_zero(c->dev + L.off_pf_cnt, L.total - L.off_pf_cnt, as_stream(stream));
  if (e == cudaSuccess) e = cudaStreamSynchronize(as_stream(stream));
  return SMEM_ERR_DEVICE_FAULT;
}

int smem_free_slots(const smem_cache* c, int32_t* n_out) {
  if (!c || !n_out) return SMEM_ERR_INVALID_ARG;
  *n_out = (int32_t)c->fifo.size();
  return SMEM_OK;
}

int smem_debug_fail_after(smem_cache* c, int32_t n) {
  if (!c || n < 0) return SMEM_ERR_INVALID_ARG;
  c->fail_after = n;
  return SMEM_OK;
}

const char* smem_last_error_detail(void) { return g_detail; }

const char* smem_strerror(int code) {
  switch (code) {
    case SMEM_OK: return "ok";
    case SMEM_ERR_INVALID_ARG: return "invalid argument";
    case SMEM_ERR_ALIGN: return "pointer not 16-byte aligned";
    case SMEM_ERR_NO_SUCH_SEQ: return "no such sequence";
    case SMEM_ERR_DUPLICATE_BLOCK: return "block index already present";
    case SMEM_ERR_NO_SUCH_BLOCK: return "no such block";
    case SMEM_ERR_POOL_FULL: return "pool full";
    case SMEM_ERR_TABLE_FULL: return "block table full";
    case SMEM_ERR_CUDA: return "CUDA error";
    case SMEM_ERR_DEVICE_FAULT: return "device error recorded";
    case SMEM_ERR_UNSUPPORTED: return "unsupported shape";
    case SMEM_ERR_NO_DEVICE: return "bookkeeping-only cache";
    case SMEM_ERR_SCRATCH_LIMIT: return "request exceeds the fixed scratch array";
    default: return "unknown error";
  }
}

int smem_mu_decode_plan(const smem_cache* c, int32_t* nq, int32_t* cluster, int32_t* slice_cols) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->lay.recompute) return SMEM_ERR_UNSUPPORTED;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (nq) *nq = c->mu_plan.nq;
  if (cluster) *cluster = c->mu_plan.cl;
  if (slice_cols) *slice_cols = c->mu_plan.wsl;
  return SMEM_OK;
}

int smem_debug_set_table_entry(smem_cache* c, int32_t seq, int32_t pos, int32_t slot, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (pos < 0 || pos >= (int)c->idx[seq].size()) return SMEM_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  return cuda_rc(smem::launch_store_int(table_row(c, seq) + pos, slot, as_stream(stream)), "table entry");
}

int smem_debug_wait_probe(smem_cache* c, long long limit_ns, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (limit_ns < 1 || limit_ns > 1000000000LL) return SMEM_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  return cuda_rc(smem::launch_wait_probe(reinterpret_cast<int*>(c->dev + c->lay.off_err),
                                         (unsigned long long)limit_ns, as_stream(stream)),
                 "wait probe");
}

int smem_debug_gemm(smem_cache* c, const void* A, int32_t lda, long long a_bs, const void* W, int32_t w_rows,
                    int32_t w_cols, int32_t b_kmajor, int32_t w_boff, int32_t M, int32_t N, int32_t K, int32_t batch,
                    int32_t epi, float alpha, void* out, int32_t ldo, long long o_bs, int32_t col_group,
                    long long group_stride, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (!A || !W || !out || M < 1 || N < 32 || K < 32 || N % 32 || K % 32 || batch < 1 || epi < 0 || epi > 2 ||
      lda < K || w_rows < 1 || w_cols < 1 || (b_kmajor != 0 && b_kmajor != 1) || w_boff < 0 || col_group < 0 ||
      (col_group && col_group % 32) || lda % 8 || ldo % 8 || a_bs % 8 || o_bs % 8 || w_cols % 8 ||
      (batch > 1 && a_bs < 1))
    return SMEM_ERR_INVALID_ARG;
  if (!aligned16(A) || !aligned16(W) || !aligned16(out)) return SMEM_ERR_ALIGN;
  DeviceGuard g(c->device);
  smem::GemmCall gc;
  gc.a = A;
  gc.lda = lda;
  gc.a_bs = a_bs;
  gc.w = W;
  gc.w_rows = w_rows;
  gc.w_cols = w_cols;
  gc.ldw = w_cols;
  gc.b_kmajor = b_kmajor;
  gc.w_boff = w_boff;
  gc.M = M;
  gc.N = N;
  gc.K = K;
  gc.batch = batch;
  gc.epi = epi;
  gc.alpha = alpha;
  gc.out = out;
  gc.ldo = ldo;
  gc.o_bs = o_bs;
  gc.col_group = col_group;
  gc.group_stride = group_stride;
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  return gemm_rc(c, gc, as_stream(stream), "projection");
}

int smem_debug_layernorm(smem_cache* c, const float* x, int32_t n, int32_t d, const float* gain, const float* bias,
                         void* h, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (!x || !gain || !bias || !h || n < 1 || d < 4 || d % 4) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(gain) || !aligned16(bias) || !aligned16(h)) return SMEM_ERR_ALIGN;
  DeviceGuard g(c->device);
  return cuda_rc(smem::launch_layernorm(x, n, d, gain, bias, static_cast<uint16_t*>(h), false, as_stream(stream)),
                 "layernorm");
}

int smem_abi_version(void) { return SMEM_ABI_VERSION; }

}  // extern "C"
