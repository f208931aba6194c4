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
  CUtensorMap pool_map_pf{};  // prefill kernel's view (whole 64-row tiles)
  smem_config cfg{};
  Layout lay{};
  uint8_t* dev = nullptr;  // nullptr: bookkeeping-only
  int device = -1;
  int num_sms = 0;
  std::vector<std::vector<int32_t>> idx;   // per sequence, ascending block index
  std::vector<std::vector<int32_t>> slot;  // per sequence, same order
  std::deque<int32_t> fifo;                // free slots, front = next to use
  std::vector<uint32_t> seen;              // decode: duplicate-sequence check
  uint32_t seen_epoch = 0;
  int fail_after = 0;                      // test hook: n-th next launch fails
  int pf_cluster_max = 0;                  // prefill cluster limit on this device (0: no clusters)
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
  if (c->head_dim != 64 && c->head_dim != 128) return SMEM_ERR_UNSUPPORTED;
  if (c->block_tokens != smem::kBlockTok || c->rows_per_block != smem::kRows) return SMEM_ERR_UNSUPPORTED;
  if (c->has_null_row != 0 && c->has_null_row != 1) return SMEM_ERR_INVALID_ARG;
  L->L = c->n_layers;
  L->H = c->n_heads;
  L->D = c->head_dim;
  L->max_seqs = c->max_seqs;
  L->max_blocks = c->max_blocks_per_seq;
  L->capacity = c->capacity_slots;
  L->has_null = c->has_null_row;
  L->max_batch = c->max_decode_batch;
  int ms = 1;
  for (int n = 1; n <= c->max_blocks_per_seq; ++n)
    ms = std::max(ms, smem::ceil_div(n, smem::decode_split_blocks(n)));
  L->dec_max_splits = ms;
  L->pf_max_splits = smem::kPrefillMaxSplits;
  const size_t D = (size_t)L->D;
  L->slot_elems = (size_t)L->L * L->H * 2 * smem::kRows * D;
  size_t off = 0;
  const size_t A = 1024;
  L->off_pool = off;
  off = align_up(off + (size_t)L->capacity * L->slot_elems * 2, A);
  L->off_inblock = off;
  off = align_up(off + (size_t)L->max_seqs * L->L * L->H * 2 * smem::kBlockTok * D * 2, A);
  L->off_null = off;
  off = align_up(off + (L->has_null ? (size_t)L->L * L->H * 2 * D * 2 : 0), A);
  L->off_table = off;
  off = align_up(off + (size_t)L->max_seqs * L->max_blocks * 4, A);
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
         ((size_t)seq * L.L + layer) * L.H * 2 * smem::kBlockTok * L.D;
}
inline const uint16_t* null_kv(smem_cache* c) {
  return c->lay.has_null ? reinterpret_cast<const uint16_t*>(c->dev + c->lay.off_null) : nullptr;
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
  c->seen.assign(L.max_seqs, 0);
  if (device) {
    c->dev = static_cast<uint8_t*>(dev_buf);
    cudaError_t e = cudaGetDevice(&c->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
    // zero everything but the pool: in-block rows, null rows, tables,
    // workspace, counters and the error word
    if (e == cudaSuccess) e = smem::launch_zero(c->dev + L.off_inblock, L.total - L.off_inblock, nullptr);
    if (e == cudaSuccess) e = cudaStreamSynchronize(nullptr);
    if (e != cudaSuccess) {
      set_detail("create", e);
      delete c;
      return SMEM_ERR_CUDA;
    }
    int er = smem::encode_pool_map(&c->pool_map, c->dev + L.off_pool, L.L, L.H, L.D, L.capacity,
                                   smem::decode_stage_rows(L.D));
    if (er == 0)
      er = smem::encode_pool_map(&c->pool_map_pf, c->dev + L.off_pool, L.L, L.H, L.D, L.capacity, smem::kRows);
    if (er != 0) {
      std::snprintf(g_detail, sizeof(g_detail), "tensor map encode failed (%d)", er);
      delete c;
      return SMEM_ERR_CUDA;
    }
    const char* knob = std::getenv("SMEM_PREFILL_CLUSTERS");
    c->pf_cluster_max = (knob && knob[0] == '0') ? 0 : smem::prefill_cluster_max(L.H, L.D);
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
  if (!c->lay.has_null || !k_null || !v_null) return SMEM_ERR_INVALID_ARG;
  if (!aligned16(k_null) || !aligned16(v_null)) return SMEM_ERR_ALIGN;
  DeviceGuard g(c->device);
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  return check_launch(c,
                      smem::launch_null_write(reinterpret_cast<uint16_t*>(c->dev + c->lay.off_null),
                                              static_cast<const uint16_t*>(k_null),
                                              static_cast<const uint16_t*>(v_null), c->lay.L, c->lay.H, c->lay.D,
                                              as_stream(stream)),
                      "null row");
}

int smem_append_block(smem_cache* c, int32_t seq, int32_t block_idx, const void* K, const void* V, void* stream,
                      int32_t* slot_out) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (block_idx < 0) return SMEM_ERR_INVALID_ARG;
  if (c->dev) {
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
                                                    static_cast<const uint16_t*>(V), c->lay.L, c->lay.H, c->lay.D,
                                                    table_row(c, seq), pos, (int)ix.size(), s, as_stream(stream)),
                                "append");
    if (rc) return rc;
  }
  c->fifo.pop_front();
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
    const int rc = check_launch(c, smem::launch_table_remove(table_row(c, seq), pos, (int)ix.size(), as_stream(stream)),
                                "delete");
    if (rc) return rc;
  }
  const int32_t s = c->slot[seq][pos];
  ix.erase(ix.begin() + pos);
  c->slot[seq].erase(c->slot[seq].begin() + pos);
  c->fifo.push_back(s);
  return SMEM_OK;
}

int smem_release_seq(smem_cache* c, int32_t seq, void* stream) {
  (void)stream;  // the device row needs no edit: its length lives on the host
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  for (int32_t s : c->slot[seq]) c->fifo.push_back(s);
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
                                                 static_cast<const uint16_t*>(V), n_rows, c->lay.H, c->lay.D,
                                                 as_stream(stream)),
                      "in-block write");
}

int smem_prefill_block(smem_cache* c, int32_t seq, int32_t layer, int32_t q_block_idx, const void* Qs,
                       const void* Ks, const void* Vs, const void* Qc, void* Osa, void* Oca, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  if (seq < 0 || seq >= c->lay.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
  if (layer < 0 || layer >= c->lay.L || q_block_idx < 0) return SMEM_ERR_INVALID_ARG;
  const void* ptrs[6] = {Qs, Ks, Vs, Qc, Osa, Oca};
  for (const void* p : ptrs) {
    if (!p) return SMEM_ERR_INVALID_ARG;
    if (!aligned16(p)) return SMEM_ERR_ALIGN;
  }
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
  a.D = c->lay.D;
  a.layer = layer;
  a.nblk = nblk;
  a.cluster = smem::prefill_use_clusters(nblk, c->pf_cluster_max) ? 1 : 0;
  if (a.cluster)
    a.split_blks = nblk ? smem::prefill_cluster_split_blocks(nblk, c->pf_cluster_max) : 1;
  else
    a.split_blks = nblk ? smem::prefill_split_blocks(nblk, c->lay.H, c->lay.D) : 1;
  a.n_splits = nblk ? smem::ceil_div(nblk, a.split_blks) : 0;
  a.capacity = c->lay.capacity;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c->lay.D));
  DeviceGuard g(c->device);
  if (injected_failure(c)) return SMEM_ERR_CUDA;
  return check_launch(c, smem::launch_prefill(a, as_stream(stream)), "prefill");
}

int smem_decode(smem_cache* c, int32_t layer, int32_t nb, const int32_t* seq_ids, const int32_t* pos,
                const int32_t* q_block_idx, const void* qs, const void* k_new, const void* v_new, const void* qc,
                void* osa, void* oca, void* stream) {
  if (!c) return SMEM_ERR_INVALID_ARG;
  if (!c->dev) return SMEM_ERR_NO_DEVICE;
  const Layout& L = c->lay;
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
  for (int i = 0; i < nb; ++i) {
    const int s = seq_ids[i];
    if (s < 0 || s >= L.max_seqs) return SMEM_ERR_NO_SUCH_SEQ;
    if (c->seen[s] == c->seen_epoch) return SMEM_ERR_INVALID_ARG;  // one token per sequence per step
    c->seen[s] = c->seen_epoch;
    if (pos[i] < 0 || pos[i] >= smem::kBlockTok || q_block_idx[i] < 0) return SMEM_ERR_INVALID_ARG;
  }
  DeviceGuard g(c->device);
  const size_t tok = (size_t)L.H * L.D;  // elements per item
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
    P.qs = static_cast<const uint16_t*>(qs) + i0 * tok;
    P.k_new = static_cast<const uint16_t*>(k_new) + i0 * tok;
    P.v_new = static_cast<const uint16_t*>(v_new) + i0 * tok;
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
    P.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)L.D));
    int pairs = 0;
    for (int i = 0; i < n; ++i) {
      const int s = seq_ids[i0 + i];
      const std::vector<int32_t>& ix = c->idx[s];
      const int nblk = (int)(std::lower_bound(ix.begin(), ix.end(), q_block_idx[i0 + i]) - ix.begin());
      P.items[i].seq = s;
      P.items[i].nblk = nblk;
      P.items[i].pos = pos[i0 + i];
      P.items[i].pair_begin = pairs;
      if (nblk) pairs += smem::ceil_div(nblk, smem::decode_split_blocks(nblk));
    }
    P.n_pairs = pairs;
    const long long units = (long long)(pairs + n) * L.H;
    const long long wpc = smem::decode_warps_per_cta();
    const int grid = (int)std::min<long long>((units + wpc - 1) / wpc, smem::decode_max_grid(L.D, c->num_sms));
    if (injected_failure(c)) return SMEM_ERR_CUDA;
    const int rc = check_launch(c, smem::launch_decode(P, L.D, grid, as_stream(stream)), "decode");
    if (rc) return rc;
  }
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
    P.k_new = static_cast<const uint16_t*>(k_new) + i0 * tok;
    P.v_new = static_cast<const uint16_t*>(v_new) + i0 * tok;
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
    P.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)L.D));
    int pairs = 0;
    for (int i = 0; i < n; ++i) {
      P.items[i].seq = seq_ids[i0 + i];
      P.items[i].nblk = nblk[i0 + i];
      P.items[i].pos = pos[i0 + i];
      P.items[i].pair_begin = pairs;
      if (nblk[i0 + i]) pairs += smem::ceil_div(nblk[i0 + i], smem::decode_split_blocks(nblk[i0 + i]));
    }
    P.n_pairs = pairs;
    const long long units = (long long)(pairs + n) * L.H;
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

int smem_abi_version(void) { return SMEM_ABI_VERSION; }

}  // extern "C"
