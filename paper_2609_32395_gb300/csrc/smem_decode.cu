// smem_decode.cu -- batched decode step of the SMem reader (one layer).
//
// Per decode item (one sequence, one new token at in-block offset p) and
// head, the reader computes (arXiv 2609.32395, Sec. 2 "Model", Sec. 3.1):
//   osa = softmax over the in-block rows 0..p   (block-local causal SA)
//   oca = softmax over the null row and the memory rows of the blocks with
//         index < the token's block index, in ascending block index
//         (block-causal CA over the materialised cross-attention K/V).
//
// Work decomposition. A work unit is (item, split, head) for CA -- a split is
// a run of consecutive table blocks whose length depends only on the block
// count -- or (item, head) for SA. CA units are handed out by a launch-wide
// atomic counter; every warp of a CTA is an independent worker with its own ring of
// shared-memory stages. A stage holds 32 rows (d_h = 64) or 16 rows
// (d_h = 128) of K and of V of one head -- 8 KB -- loaded by tensor TMA with
// the 128-byte swizzle, so that a lane can read a whole K row without bank
// conflicts. Lane 0 keeps the ring three stages ahead of the warp, across
// unit boundaries. Scores are lane-per-row fp32 dot products (no shuffles),
// the online softmax runs in base 2 with one warp maximum per stage, and P.V
// accumulates in fp32 with each lane owning 8 columns of a quarter of the
// rows. A CA unit writes its split partial (m, l, acc[d_h]); the warp that
// completes the last split of an (item, head) merges all splits in split
// order (null row first). With grouped-query attention a CA unit serves the
// 2 or 4 query heads that share a key/value head: the warp scores each stage
// against all of them with warp-level tensor-core MMAs (the stage's keys as
// the 16 rows, the group's queries as the columns), transposes P in
// registers (movmatrix) into the operand of O^T += V^T P^T, so the rows
// stream once per group at 16 MMAs per stage. SA units read their <= 64
// in-block rows straight from global memory (every load of a unit in flight
// at once) and come from a second counter once a warp's CA stream has ended,
// so they fill the launch's tail. No warp ever waits for another warp; every reduction
// order is fixed by the block count, so the same block set gives the same
// bits whatever the slots or the edit history.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cudaTypedefs.h>
#include <mutex>

#include "../../include/smem.h"

#include "smem_device.cuh"
#include "smem_internal.h"

namespace smem {

constexpr int kUnitQueue = 8;  // fetched-but-unconsumed units of a warp (<= NS + 1 used)

template <int D, int QN = 1>
struct Dec {
  static constexpr int R = kRows;
  static constexpr int SROWS = D == 32 ? 64 : (D == 64 ? 32 : 16);  // rows per stage
  static constexpr int CHUNKS = R / SROWS;         // stages per memory block
  static constexpr int HALF = SROWS * D * 2;       // K (or V) bytes of a stage
  static constexpr int STAGE = 2 * HALF;           // 8 KB
  static constexpr int BOXES = D < 64 ? 1 : D / 64;  // TMA boxes per row (64 or 128 bytes wide)
  static constexpr int ROWB = D < 64 ? D * 2 : 128;  // bytes of a row within a box
  static constexpr int BOX_BYTES = SROWS * ROWB;
  static constexpr int QW = D < 64 ? D : 64;       // query columns a lane holds
  static constexpr int RPL = D == 32 ? 2 : 1;      // K rows a lane scores per stage
  static constexpr int NW = 8;                     // worker warps per CTA
  static constexpr int NS = 3;                     // stages per warp
  static constexpr int THREADS = NW * 32;
  static constexpr int LPR = D < 64 ? 1 : D / 64;  // lanes per row in the score phase
  static constexpr int OFF_BAR = NW * NS * STAGE;
  static constexpr int OFF_P = OFF_BAR + NW * NS * 8;               // per warp: P of 64 rows (fp32)
  static constexpr int OFF_Q = OFF_P + NW * 64 * 4;                 // per stage: the unit's queries
  static constexpr int OFF_UQ = OFF_Q + NW * NS * QN * D * 2;       // per warp: unit queue
  static constexpr int OFF_END = OFF_UQ + NW * kUnitQueue * 4;
  static constexpr int SMEM = OFF_END + 1024;      // + slack to align the base to 1 KB
};

// Byte offset of 16-byte chunk c of row r in a stage half: 128-byte swizzle
// over boxes of 64 columns, or the 64-byte swizzle of 32-column rows.
template <int D>
__device__ __forceinline__ int chunk_off(int r, int c) {
  if constexpr (D == 32) return r * 64 + ((c ^ ((r >> 1) & 3)) << 4);
  else return (c >> 3) * Dec<D>::BOX_BYTES + r * 128 + (((c & 7) ^ (r & 7)) << 4);
}

struct Unit {
  int sa;     // 1: self-attention unit
  int item;
  int h;
  int split;  // CA only
  int b0;     // first table position (CA)
  int nt;     // memory blocks (CA)
};

__device__ __forceinline__ Unit unit_of(const DecodeParams& p, int u) {
  Unit U;
  const int upp = p.H / p.qn;  // CA units per (item, split): one per group of qn query heads
  const int nca = p.n_pairs * upp;
  if (u < nca) {
    const int pair = u / upp;
    U.sa = 0;
    U.h = (u - pair * upp) * p.qn;  // first query head of the unit
    int lo = 0, hi = p.n_items - 1;  // last item with pair_begin <= pair
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (p.items[mid].pair_begin <= pair) lo = mid; else hi = mid - 1;
    }
    U.item = lo;
    U.split = pair - p.items[lo].pair_begin;
    const int sb = decode_split_blocks(p.items[lo].nblk);
    U.b0 = U.split * sb;
    const int rem = p.items[lo].nblk - U.b0;
    U.nt = rem < sb ? rem : sb;
  } else {
    const int v = u - nca;
    U.sa = 1;
    U.item = v / p.H;
    U.h = v - U.item * p.H;
    U.split = 0;
    U.b0 = 0;
    U.nt = 0;
  }
  return U;
}

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ uint4 ld_nc16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Warp-level tensor-core helpers of the grouped decode (PTX mma.sync /
// ldmatrix). mma_16816: D[16x8] += A[16x16] B[16x8], bf16 in, fp32 out, the
// A rows 8..15 zero (a1 = a3 = 0): a0/a2 = columns 2t.. / 2t+8.. of row g.
__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a2, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1));
}
// The same keeping only row g of D (the rows 8..15 of a zero A are zero).
__device__ __forceinline__ void mma_16816_acc2(float (&d)[2], uint32_t a0, uint32_t a2, uint32_t b0, uint32_t b1) {
  float z0 = 0.f, z1 = 0.f;
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(z0), "+f"(z1)
      : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1));
}
// D[16x8] += A[16x16] B[16x8] with every A row used (keys as rows).
__device__ __forceinline__ void mma_16816_full(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// Transpose of an 8x8 b16 matrix held as (row lane/4, columns 2(lane%4) ..+1).
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
// Four 8x8 b16 matrices; lane l gives the 16-byte row address of row l%8 of
// matrix l/8. Plain: thread (g, t) gets row g, columns 2t, 2t+1 of each
// matrix; trans: rows 2t, 2t+1 of column g.
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t saddr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(saddr));
}
__device__ __forceinline__ void ldsm_x4_trans(uint32_t (&r)[4], uint32_t saddr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(saddr));
}

__device__ __forceinline__ void store_bf16x8(uint16_t* dst, const float* v, float scale) {
  uint4 o;
  o.x = pack_bf16x2(v[0] * scale, v[1] * scale);
  o.y = pack_bf16x2(v[2] * scale, v[3] * scale);
  o.z = pack_bf16x2(v[4] * scale, v[5] * scale);
  o.w = pack_bf16x2(v[6] * scale, v[7] * scale);
  *reinterpret_cast<uint4*>(dst) = o;
}

// Rotary phase: the 8 values t (pairs (0,1) .. (6,7)) turned by the angles
// of pairs cs[0..3] of a table row.
__device__ __forceinline__ void rot8f(float* t, const float2* cs) {
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 c = cs[e];
    const float x0 = t[2 * e], x1 = t[2 * e + 1];
    t[2 * e] = x0 * c.x - x1 * c.y;
    t[2 * e + 1] = x0 * c.y + x1 * c.x;
  }
}

// Issue side of one warp's chunk stream over dynamically fetched CA units.
// Lane 0 only. Units come from a launch-wide atomic counter; the next unit is
// fetched when the issue side reaches the end of the current one (still NS
// chunks ahead of the warp's math), so a warp never holds a unit it will not
// start soon -- with about one unit per warp, an early fetch let some warps
// take two units while others had none. Each fetched unit is pushed on the
// warp's unit queue together with the stage that holds its first chunk.
struct Issue {
  int u;       // unit being issued (< 0: exhausted)
  int c;       // next chunk of that unit
  int nc;      // chunks of that unit
  int item, h, b0;
  int ybase;   // pool-map row of the unit's (layer, key/value head) K tile
  int pushed;  // queue entries pushed
  int slot;    // pool slot of the block being issued
  int slot_next;  // the unit's next block's slot, loaded a block ahead (-1: none or out of range)
};

// Table entry `blk` of a stream's item, or -1 when the index is out of range
// (recorded in the bounds-checking build). The load is issued here and its
// value is used a block later, so its latency stays off the warp's path.
__device__ __forceinline__ int table_slot(const DecodeParams& p, int item, int blk) {
  const DecodeItem& itm = p.items[item];
  const bool in_range = SMEM_DCHECK(item < p.n_items && itm.seq >= 0 && itm.seq < p.max_seqs && blk >= 0 &&
                                        blk < itm.nblk && itm.nblk <= p.max_blocks,
                                    p.err);
  return in_range ? p.table[(size_t)itm.seq * p.max_blocks + blk] : -1;
}

__device__ __forceinline__ int fetch_unit(const DecodeParams& p) {
  const unsigned long long u = atomicAdd(p.sched, 1ull);
  const int nca = p.n_pairs * (p.H / p.qn);
  return u < (unsigned long long)nca ? (int)u : -1;
}

template <int D>
__device__ __forceinline__ void issue_begin_unit(const DecodeParams& p, Issue& is, int u, int* uq) {
  is.u = u;
  is.c = 0;
  if (u >= 0) {
    const Unit U = unit_of(p, u);
    is.nc = U.nt * Dec<D>::CHUNKS;
    is.item = U.item;
    is.h = U.h;
    is.b0 = U.b0;
    is.ybase = ((p.layer * p.Hkv + U.h / (p.H / p.Hkv)) * 2) * Dec<D>::R;
    is.slot_next = table_slot(p, U.item, U.b0);  // used when the unit's first chunk is issued
  } else {
    is.nc = 0;
  }
  uq[is.pushed % kUnitQueue] = u;  // -1 marks the end of the stream
  ++is.pushed;
}

// Loads the next chunk of the stream into `stage` (and the unit's query into
// `qslot` with its first chunk); returns false when the stream is exhausted.
template <int D>
__device__ __forceinline__ bool issue_next(const DecodeParams& p, Issue& is, uint8_t* stage, uint16_t* qslot,
                                           uint64_t* bar, int* uq) {
  using C = Dec<D>;
  if (is.u < 0) return false;
  const int row0 = (is.c % C::CHUNKS) * C::SROWS;
  if (is.c % C::CHUNKS == 0) {
    // a new block: its slot was loaded a block ago; load the next block's now
    is.slot = is.slot_next;
    const int nxt = is.c / C::CHUNKS + 1;  // the unit's next block (relative)
    is.slot_next = nxt * C::CHUNKS < is.nc ? table_slot(p, is.item, is.b0 + nxt) : -1;
  }
  const int slot = is.slot;
  const uint32_t qbytes = is.c == 0 ? p.qn * D * 2 : 0;  // the unit's qn query heads (contiguous)
  if (slot < 0 || slot >= p.capacity) {
    record_error(p.err, kDevErrBounds);
    mbar_arrive(bar);  // the stage keeps stale rows; the error is flagged
  } else {
    const int y = is.ybase + row0;
    mbar_arrive_expect_tx(bar, C::STAGE + qbytes);
#pragma unroll
    for (int bx = 0; bx < C::BOXES; ++bx) {
      tma_load_3d(stage + bx * C::BOX_BYTES, &p.tmap, bx * 64, y, slot, bar);
      tma_load_3d(stage + C::HALF + bx * C::BOX_BYTES, &p.tmap, bx * 64, y + C::R, slot, bar);
    }
    if (qbytes) bulk_g2s(qslot, p.qc + (size_t)is.item * p.c_stride + (size_t)is.h * D, qbytes, bar);
  }
  if (++is.c == is.nc) issue_begin_unit<D>(p, is, fetch_unit(p), uq);
  return true;
}

// Self-attention unit: in-block rows 0..p-1 and the new token's row, read
// directly from global memory. Writes osa, stores the new row, and writes
// oca for a sequence that has no readable memory block.
template <int D, bool ROPE>
__device__ void sa_unit(const DecodeParams& p, const Unit& U, float* pbuf, int lane) {
  constexpr int LPR = Dec<D>::LPR;
  constexpr int RPP = 32 / LPR;  // rows per pass
  const DecodeItem& it = p.items[U.item];
  if (!SMEM_DCHECK(U.item < p.n_items && it.seq >= 0 && it.seq < p.max_seqs && it.pos >= 0 && it.pos < kBlockTok &&
                       it.nblk <= p.max_blocks,
                   p.err))
    return;
  const int n = it.pos + 1;
  const int grp = p.H / p.Hkv;  // query heads per key/value head (grouped-query attention)
  const int kvh = U.h / grp;
  const size_t qoff = ((size_t)U.item * p.H + U.h) * D;               // outputs
  const size_t soff = (size_t)U.item * p.s_stride + (size_t)U.h * D;   // qs
  const size_t koff = (size_t)U.item * p.kv_stride + (size_t)kvh * D;  // k_new, v_new
  const uint16_t* ib = p.inblock + (((size_t)it.seq * p.L + p.layer) * p.Hkv + kvh) * (size_t)2 * kBlockTok * D;
  constexpr int QW = Dec<D>::QW;  // columns of a row per lane
  const int hh = lane % LPR;  // which QW columns of the row
  // with rotary phases the new token's query and key turn by its offset p
  const float2* rp = ROPE ? p.rope_tab + (size_t)it.pos * (D / 2) + hh * (QW / 2) : nullptr;
  if (p.mode & 1) {
    constexpr int NP = kBlockTok / RPP;  // score passes
    constexpr int NJ = QW / 8;           // 16-byte loads per row slice
    constexpr int KB = NP * NJ <= 16 ? NP : 1;  // passes whose key rows load in one batch
    // P.V: lane (g, c) owns column chunk c of rows g*RG .. g*RG+RG-1
    constexpr int CPL = D / 8;        // column chunks
    constexpr int G = 32 / CPL;       // row groups
    constexpr int RG = kBlockTok / G; // rows per group
    constexpr int VB = RG < 16 ? RG : 16;  // value rows per batch of loads
    const int g = lane / CPL, c = lane % CPL;
    // None of the unit's loads depends on another: the query slice, the first
    // batch of key rows and (without rotary phases, whose tables need the
    // registers) the first batch of value rows all go out before the first
    // product, so the unit pays one memory round trip, not three.
    uint4 qw[NJ], kw[KB][NJ], vw[VB];
    auto load_keys = [&](int k0) {
#pragma unroll
      for (int kb = 0; kb < KB; ++kb) {
        const int r = (k0 + kb) * RPP + lane / LPR;
        const uint16_t* row = r == it.pos ? p.k_new + koff : ib + (size_t)r * D;
#pragma unroll
        for (int j = 0; j < NJ; ++j) kw[kb][j] = r < n ? ld_nc16(row + hh * QW + j * 8) : make_uint4(0u, 0u, 0u, 0u);
      }
    };
    auto load_values = [&](int i0) {
#pragma unroll
      for (int i = 0; i < VB; ++i) {
        const int r = g * RG + i0 + i;
        const uint16_t* row = r == it.pos ? p.v_new + koff : ib + (size_t)kBlockTok * D + (size_t)r * D;
        vw[i] = r < n ? ld_nc16(row + c * 8) : make_uint4(0u, 0u, 0u, 0u);
      }
    };
#pragma unroll
    for (int j = 0; j < NJ; ++j) qw[j] = ld_nc16(p.qs + soff + hh * QW + j * 8);
    load_keys(0);
    if (!ROPE) load_values(0);
    float q[QW];
#pragma unroll
    for (int j = 0; j < NJ; ++j) {
      float t[8];
      unpack8(qw[j], t);
      if (ROPE) rot8f(t, rp + j * 4);
#pragma unroll
      for (int e = 0; e < 8; ++e) q[j * 8 + e] = t[e] * p.scale_log2;
    }
    // scores of rows lane/LPR + k*RPP
    float s[NP];
    float mx = -INFINITY;
#pragma unroll
    for (int k0 = 0; k0 < NP; k0 += KB) {
      if (k0 > 0) load_keys(k0);
#pragma unroll
      for (int kb = 0; kb < KB; ++kb) {
        const int k = k0 + kb;
        const int r = k * RPP + lane / LPR;
        float dot = 0.f;
        if (r < n) {
#pragma unroll
          for (int j = 0; j < NJ; ++j) {
            float t[8];
            unpack8(kw[kb][j], t);
            if (ROPE && r == it.pos) rot8f(t, rp + j * 4);  // stored rows are already turned
#pragma unroll
            for (int e = 0; e < 8; ++e) dot = fmaf(q[j * 8 + e], t[e], dot);
          }
        }
        if (LPR == 2) dot += __shfl_xor_sync(0xffffffffu, dot, 1);
        s[k] = r < n ? dot : -INFINITY;
        mx = fmaxf(mx, s[k]);
      }
    }
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float l = 0.f;
#pragma unroll
    for (int k = 0; k < NP; ++k) {
      const int r = k * RPP + lane / LPR;
      const float pr = r < n ? exp2f(s[k] - mx) : 0.f;
      if (hh == 0) {
        l += pr;
        pbuf[r] = pr;
      }
    }
    __syncwarp();
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    float acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.f;
    // products in row order, VB value rows per batch of loads
#pragma unroll
    for (int i0 = 0; i0 < RG; i0 += VB) {
      if (i0 > 0 || ROPE) load_values(i0);
#pragma unroll
      for (int i = 0; i < VB; ++i) {
        const int r = g * RG + i0 + i;
        if (r < n) {
          const float pr = pbuf[r];
          float t[8];
          unpack8(vw[i], t);
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[e] = fmaf(pr, t[e], acc[e]);
        }
      }
    }
#pragma unroll
    for (int o = CPL; o < 32; o <<= 1)
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
    if (g == 0) store_bf16x8(p.osa + qoff + c * 8, acc, 1.f / l);
    // the new token's k and v become in-block row p for later steps (one
    // query head of the group writes the shared row)
    if (U.h % grp == 0 && lane < 2 * CPL) {
      const int kv = lane / CPL, cc = lane % CPL;
      uint16_t* dst = (uint16_t*)ib + (size_t)kv * kBlockTok * D + (size_t)it.pos * D + cc * 8;
      uint4 w = ld_nc16((kv ? p.v_new : p.k_new) + koff + cc * 8);
      if (ROPE && !kv) {
        float t[8];
        unpack8(w, t);
        rot8f(t, p.rope_tab + (size_t)it.pos * (D / 2) + cc * 4);
        w = make_uint4(pack_bf16x2(t[0], t[1]), pack_bf16x2(t[2], t[3]), pack_bf16x2(t[4], t[5]),
                       pack_bf16x2(t[6], t[7]));
      }
      *reinterpret_cast<uint4*>(dst) = w;
    }
  }  // self-attention half
  // no readable memory block: oca is the null row's value or zero
  if ((p.mode & 2) && it.nblk == 0 && lane < D / 8) {
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = 0.f;
    if (p.null_kv) unpack8(ld_nc16(p.null_kv + ((size_t)p.layer * p.Hkv + kvh) * 2 * D + D + lane * 8), v);
    store_bf16x8(p.oca + qoff + lane * 8, v, 1.f);
  }
  __syncwarp();
}

// Split partials a warp has written but not yet announced (pend1), or
// announced with a ticket still in flight (pend2): the fence and the atomic of
// a unit are issued one unit later and their result read two units later,
// so neither stalls the warp while the ring keeps streaming.
struct Pending {
  int valid, item, h, nsplit, pair_begin;
  unsigned ticket;  // lane 0
};

template <int D, bool ROPE>
__device__ void merge_splits(const DecodeParams& p, const Pending& pd, int lane) {
  if (!SMEM_DCHECK(pd.item < p.n_items && pd.h < p.H && (long long)pd.pair_begin + pd.nsplit <= p.part_pairs, p.err))
    return;
  constexpr int CPT = D / 32;  // columns per lane
  const size_t qoff = ((size_t)pd.item * p.H + pd.h) * D;
  const size_t qcoff = (size_t)pd.item * p.c_stride + (size_t)pd.h * D;
  float nscore = -INFINITY;
  if (p.null_kv) {
    // null-row score with the same scaled-query dot product as the rows
    const uint16_t* kn = p.null_kv + ((size_t)p.layer * p.Hkv + pd.h / (p.H / p.Hkv)) * 2 * D;
    float qv[CPT];
#pragma unroll
    for (int e = 0; e < CPT; ++e) qv[e] = bf16lo(p.qc[qcoff + lane * CPT + e]);
    if (ROPE) {
      // the null row's key phase is max(0, i - W): the query turns by min(i, W)
      const int qb = p.items[pd.item].qblk;
      const float2* tab = p.rope_tab + (size_t)min(qb, p.rope_w) * (D / 2);
      if constexpr (CPT == 1) {
        // one column per lane: the pair (2m, 2m+1) spans lanes 2m and 2m+1
        const float xe = __shfl_sync(0xffffffffu, qv[0], lane & ~1);
        const float xo = __shfl_sync(0xffffffffu, qv[0], lane | 1);
        const float2 c = tab[lane >> 1];
        qv[0] = (lane & 1) ? xe * c.y + xo * c.x : xe * c.x - xo * c.y;
      } else {
        const float2* cs = tab + lane * (CPT / 2);
#pragma unroll
        for (int e = 0; e < CPT; e += 2) {
          const float2 c = cs[e / 2];
          const float x0 = qv[e], x1 = qv[e + 1];
          qv[e] = x0 * c.x - x1 * c.y;
          qv[e + 1] = x0 * c.y + x1 * c.x;
        }
      }
    }
    float dot = 0.f;
#pragma unroll
    for (int e = 0; e < CPT; ++e) dot = fmaf(qv[e] * p.scale_log2, bf16lo(kn[lane * CPT + e]), dot);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    nscore = dot;
  }
  const float* pb = p.part + ((size_t)pd.pair_begin * p.H + pd.h) * (D + 4);
  const size_t ps = (size_t)p.H * (D + 4);
  constexpr int G = 16;  // splits whose loads are in flight together
  // pass 1: the maximum over the null row and every split -- lane i reads
  // splits i, i + 32, ... and the warp reduces (a maximum is order-free)
  float M = nscore;
  for (int s2 = lane; s2 < pd.nsplit; s2 += 32) M = fmaxf(M, __ldcg(pb + s2 * ps));
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float Lsum = 0.f, A[CPT];
#pragma unroll
  for (int e = 0; e < CPT; ++e) A[e] = 0.f;
  if (p.null_kv) {
    const float f = exp2f(nscore - M);
    Lsum = f;
    const uint16_t* vn = p.null_kv + ((size_t)p.layer * p.Hkv + pd.h / (p.H / p.Hkv)) * 2 * D + D;
#pragma unroll
    for (int e = 0; e < CPT; ++e) A[e] = f * bf16lo(vn[lane * CPT + e]);
  }
  // pass 2: weighted sums in split order, G splits' loads issued first
  for (int s0 = 0; s0 < pd.nsplit; s0 += G) {
    float ml[G][2], av[G][CPT];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const bool in = s0 + g < pd.nsplit;
      const float* ps2 = pb + (s0 + g) * ps;
      const float2 v = in ? __ldcg(reinterpret_cast<const float2*>(ps2)) : make_float2(-INFINITY, 0.f);
      ml[g][0] = v.x;
      ml[g][1] = v.y;
#pragma unroll
      for (int e = 0; e < CPT; ++e) av[g][e] = in ? __ldcg(ps2 + 4 + lane * CPT + e) : 0.f;
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      if (s0 + g >= pd.nsplit) break;
      const float f = exp2f(ml[g][0] - M);
      Lsum = fmaf(f, ml[g][1], Lsum);
#pragma unroll
      for (int e = 0; e < CPT; ++e) A[e] = fmaf(f, av[g][e], A[e]);
    }
  }
  const float inv = 1.f / Lsum;
  if constexpr (CPT == 1) {
    const __nv_bfloat16 b = __float2bfloat16_rn(A[0] * inv);
    p.oca[qoff + lane] = *reinterpret_cast<const uint16_t*>(&b);
  } else {
    uint32_t* o32 = reinterpret_cast<uint32_t*>(p.oca + qoff) + lane * (CPT / 2);
#pragma unroll
    for (int e = 0; e < CPT; e += 2) o32[e / 2] = pack_bf16x2(A[e] * inv, A[e + 1] * inv);
  }
  if (lane == 0) p.counters[pd.item * p.H + pd.h] = 0u;
}

// The merges of a grouped unit's query heads h0 + j (bit j of `heads`: the
// heads whose last ticket this warp holds), all at once: lanes
// j*LPH .. j*LPH+LPH-1 serve head h0 + j with CPL columns each, so every
// head's loads go out together instead of one head's after another's. Per
// head the arithmetic is merge_splits' (the null-row score, the maximum over
// it and the splits, then the weighted sums with the null row first and the
// splits in split order).
template <int D, bool ROPE, int QN>
__device__ void merge_group(const DecodeParams& p, int item, int h0, unsigned heads, int nsplit, int pair_begin,
                            int lane) {
  constexpr int LPH = 32 / QN;  // lanes per query head
  constexpr int CPL = D / LPH;  // columns per lane (4 or 8)
  constexpr int GB = 8;         // splits whose loads are in flight together
  static_assert(CPL % 4 == 0, "whole float4 column groups per lane");
  const int j = lane / LPH, li = lane % LPH, c0 = li * CPL;
  const bool act = ((heads >> j) & 1u) &&
                   SMEM_DCHECK(item < p.n_items && h0 + j < p.H && (long long)pair_begin + nsplit <= p.part_pairs,
                               p.err);
  const int h = act ? h0 + j : h0;  // idle lanes address a valid head and load nothing
  const uint16_t* kn = p.null_kv ? p.null_kv + ((size_t)p.layer * p.Hkv + h / (p.H / p.Hkv)) * 2 * D : nullptr;
  float nscore = -INFINITY;
  if (kn) {
    float qv[CPL];
#pragma unroll
    for (int e = 0; e < CPL; ++e) qv[e] = act ? bf16lo(p.qc[(size_t)item * p.c_stride + (size_t)h * D + c0 + e]) : 0.f;
    if (ROPE) {
      // the null row's key phase is max(0, i - W): the query turns by min(i, W)
      const float2* cs = p.rope_tab + (size_t)min(p.items[item].qblk, p.rope_w) * (D / 2) + c0 / 2;
#pragma unroll
      for (int e = 0; e < CPL; e += 2) {
        const float2 c = cs[e / 2];
        const float x0 = qv[e], x1 = qv[e + 1];
        qv[e] = x0 * c.x - x1 * c.y;
        qv[e + 1] = x0 * c.y + x1 * c.x;
      }
    }
    float dot = 0.f;
#pragma unroll
    for (int e = 0; e < CPL; ++e) dot = fmaf(qv[e] * p.scale_log2, act ? bf16lo(kn[c0 + e]) : 0.f, dot);
#pragma unroll
    for (int o = 1; o < LPH; o <<= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    nscore = dot;
  }
  const float* pb = p.part + ((size_t)pair_begin * p.H + h) * (D + 4);
  const size_t ps = (size_t)p.H * (D + 4);
  float M = nscore;
  if (act)
    for (int s2 = li; s2 < nsplit; s2 += LPH) M = fmaxf(M, __ldcg(pb + s2 * ps));
#pragma unroll
  for (int o = 1; o < LPH; o <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  float Lsum = 0.f, A[CPL];
#pragma unroll
  for (int e = 0; e < CPL; ++e) A[e] = 0.f;
  if (kn && act) {
    const float f = exp2f(nscore - M);
    Lsum = f;
#pragma unroll
    for (int e = 0; e < CPL; ++e) A[e] = f * bf16lo(kn[D + c0 + e]);
  }
  for (int s0 = 0; s0 < nsplit; s0 += GB) {
    float2 ml[GB];
    float4 av[GB][CPL / 4];
#pragma unroll
    for (int g = 0; g < GB; ++g) {
      const bool in = act && s0 + g < nsplit;
      const float* ps2 = pb + (size_t)(s0 + g) * ps;
      ml[g] = in ? __ldcg(reinterpret_cast<const float2*>(ps2)) : make_float2(-INFINITY, 0.f);
#pragma unroll
      for (int e = 0; e < CPL / 4; ++e)
        av[g][e] = in ? __ldcg(reinterpret_cast<const float4*>(ps2 + 4 + c0) + e) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int g = 0; g < GB; ++g) {
      if (s0 + g >= nsplit) break;
      const float f = exp2f(ml[g].x - M);
      Lsum = fmaf(f, ml[g].y, Lsum);
#pragma unroll
      for (int e = 0; e < CPL / 4; ++e) {
        A[4 * e] = fmaf(f, av[g][e].x, A[4 * e]);
        A[4 * e + 1] = fmaf(f, av[g][e].y, A[4 * e + 1]);
        A[4 * e + 2] = fmaf(f, av[g][e].z, A[4 * e + 2]);
        A[4 * e + 3] = fmaf(f, av[g][e].w, A[4 * e + 3]);
      }
    }
  }
  if (act) {
    const float inv = 1.f / Lsum;
    uint32_t* o32 = reinterpret_cast<uint32_t*>(p.oca + ((size_t)item * p.H + h) * D + c0);
#pragma unroll
    for (int e = 0; e < CPL; e += 2) o32[e / 2] = pack_bf16x2(A[e] * inv, A[e + 1] * inv);
    if (li == 0) p.counters[item * p.H + h] = 0u;
  }
}

// pend2: read its ticket; the warp that completed the last split merges.
template <int D, bool ROPE>
__device__ __forceinline__ void settle(const DecodeParams& p, Pending& pd, int lane) {
  if (!pd.valid) return;
  const unsigned t = __shfl_sync(0xffffffffu, pd.ticket, 0);
  if (t == (unsigned)(pd.nsplit - 1)) {
    __threadfence();
    merge_splits<D, ROPE>(p, pd, lane);
  }
  pd.valid = 0;
}

// pend1 -> pend2: make its partial visible, then take a ticket.
__device__ __forceinline__ void announce(const DecodeParams& p, Pending& from, Pending& to, int lane) {
  if (!from.valid) return;
  __threadfence();
  if (lane == 0) from.ticket = atomicAdd(&p.counters[from.item * p.H + from.h], 1u);
  to = from;
  from.valid = 0;
}

template <int D, bool ROPE, int QN>
__global__ void __launch_bounds__(Dec<D>::THREADS, 1) decode_kernel(const __grid_constant__ DecodeParams p) {
  using C = Dec<D, QN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint8_t* ring = base + warp * C::NS * C::STAGE;
  uint64_t* full = reinterpret_cast<uint64_t*>(base + C::OFF_BAR) + warp * C::NS;
  float* pbuf = reinterpret_cast<float*>(base + C::OFF_P) + warp * 64;
  uint16_t* qarea = reinterpret_cast<uint16_t*>(base + C::OFF_Q) + warp * C::NS * QN * D;
  int* uq = reinterpret_cast<int*>(base + C::OFF_UQ) + warp * kUnitQueue;

  if (lane == 0) {
    for (int s = 0; s < C::NS; ++s) mbar_init(&full[s], 1);
    fence_mbar_init();
  }
  __syncthreads();


  // prologue: start streaming the first CA units. Every warp begins with
  // cross-attention; the self-attention units come after a warp's stream has
  // ended (below).
  Issue is;
  int issued = 0;
  if (lane == 0) {
    is.pushed = 0;
    issue_begin_unit<D>(p, is, fetch_unit(p), uq);
    for (int s = 0; s < C::NS; ++s)
      if (issue_next<D>(p, is, ring + s * C::STAGE, qarea + s * QN * D, &full[s], uq)) ++issued;
  }
  __syncwarp();

  constexpr int CPL = D / 8;             // P.V column chunks
  constexpr int G = 32 / CPL;            // P.V row groups per stage
  constexpr int RG = C::SROWS / G;       // rows per group per stage (8)
  const int g = lane / CPL, c = lane % CPL;
  const int hh = lane % C::LPR;          // score phase: which 64 columns
  const int rr = lane / C::LPR;          // score phase: row within the stage
  int k = 0;                             // chunks consumed
  int popped = 0;
  bool failed = false;
  Pending pend1, pend2;
  pend1.valid = pend2.valid = 0;

  while (!failed) {
    const int u = uq[popped % kUnitQueue];
    ++popped;
    if (u < 0) break;
    const Unit U = unit_of(p, u);
    const DecodeItem& it = p.items[U.item];
    if constexpr (QN > 1) {
      // ---- grouped unit: the p.qn query heads U.h .. U.h+qn-1 read one
      // key/value head; the warp scores every stage against all of them on
      // the tensor cores (mma.sync m16n8k16, bf16 in, fp32 accumulate) with
      // the stage's keys as the 16 rows and the group's queries as the 8
      // columns (query columns >= qn are zero):
      //   S^T[key][q] = K[key][:] . Q[q][:]     (A = K by ldmatrix, B = Q)
      //   O^T[c][q]  += V^T[c][key] P^T[key][q] (A = V^T by ldmatrix.trans)
      // P^T's fragments come from the score accumulators by one movmatrix
      // transpose per 8x8 tile. Thread (g = lane/4, t = lane%4) holds keys g,
      // g+8 of every 16-key tile and columns c = g, g+8 of every 16-column
      // tile, for queries 2t, 2t+1. A stage costs 16 MMAs at every head
      // width; the rows stream once per group.
      constexpr int MT = C::SROWS / 16;  // 16-key tiles of a stage
      constexpr int KS = D / 16;         // k-steps of the score MMAs
      constexpr int DT = D / 16;         // 16-column tiles of O^T
      const int ng = p.qn;
      const int gq = lane >> 2, tq = lane & 3;
      uint32_t qb[KS][2];  // B fragments: query gq, columns 16ks + 2tq (+8)
      float o[DT][4];      // O^T: columns 16dt + gq (+8) x queries 2tq, 2tq+1
      float gm[2] = {-INFINITY, -INFINITY}, gl[2] = {0.f, 0.f};  // per query column 2tq + e
#pragma unroll
      for (int dt = 0; dt < DT; ++dt) o[dt][0] = o[dt][1] = o[dt][2] = o[dt][3] = 0.f;
      const int nch = U.nt * C::CHUNKS;
      for (int ch = 0; ch < nch; ++ch, ++k) {
        const int s = k % C::NS;
        const uint32_t par = (k / C::NS) & 1;
        if (!__all_sync(0xffffffffu, mbar_wait_bounded(&full[s], par, nullptr))) {
          if (lane == 0) record_error(p.err, kDevErrWaitFull);
          failed = true;
          break;
        }
        if (ch == 0) {
          const bool real = gq < ng;
          const uint16_t* qs = qarea + s * QN * D + (real ? gq : 0) * D;
#pragma unroll
          for (int ks = 0; ks < KS; ++ks) {
            qb[ks][0] = real ? *reinterpret_cast<const uint32_t*>(qs + 16 * ks + 2 * tq) : 0u;
            qb[ks][1] = real ? *reinterpret_cast<const uint32_t*>(qs + 16 * ks + 8 + 2 * tq) : 0u;
          }
        }
        const uint8_t* kb = ring + s * C::STAGE;
        const uint8_t* vb = kb + C::HALF;
        // S^T per 16-key tile: keys as A rows (lane l addresses key 16mt +
        // l%8 + 8((l/8)%2), columns 16ks + 8(l/16) ..)
        float sacc[MT][4];
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          sacc[mt][0] = sacc[mt][1] = sacc[mt][2] = sacc[mt][3] = 0.f;
#pragma unroll
          for (int ks = 0; ks < KS; ++ks) {
            uint32_t a[4];
            ldsm_x4(a, smem_u32(kb + chunk_off<D>(16 * mt + (lane & 7) + 8 * ((lane >> 3) & 1), 2 * ks + (lane >> 4))));
            mma_16816_full(sacc[mt], a, qb[ks][0], qb[ks][1]);
          }
        }
        // online softmax per query column (2tq + e): maximum over the keys of
        // this thread, then over the 8 threads of the column (lanes tq + 4j)
        float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            sacc[mt][e] *= p.scale_log2;
            mx[e & 1] = fmaxf(mx[e & 1], sacc[mt][e]);
          }
        float alpha[2], mn[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
#pragma unroll
          for (int off = 4; off < 32; off <<= 1) mx[e] = fmaxf(mx[e], __shfl_xor_sync(0xffffffffu, mx[e], off));
          mn[e] = fmaxf(gm[e], mx[e]);
          alpha[e] = exp2f(gm[e] - mn[e]);
          gm[e] = mn[e];
        }
        // P (bf16) and its transpose into the B fragments of P^T
        uint32_t pb[MT][2];
        float ps[2] = {0.f, 0.f};
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          const uint32_t top = pack_bf16x2(exp2f(sacc[mt][0] - mn[0]), exp2f(sacc[mt][1] - mn[1]));  // key gq
          const uint32_t bot = pack_bf16x2(exp2f(sacc[mt][2] - mn[0]), exp2f(sacc[mt][3] - mn[1]));  // key gq + 8
          ps[0] += bf16lo(top) + bf16lo(bot);  // the sums of the P the MMAs use
          ps[1] += bf16hi(top) + bf16hi(bot);
          pb[mt][0] = movmatrix_trans(top);
          pb[mt][1] = movmatrix_trans(bot);
        }
#pragma unroll
        for (int e = 0; e < 2; ++e) gl[e] = gl[e] * alpha[e] + ps[e];
#pragma unroll
        for (int dt = 0; dt < DT; ++dt) {
          o[dt][0] *= alpha[0];
          o[dt][1] *= alpha[1];
          o[dt][2] *= alpha[0];
          o[dt][3] *= alpha[1];
        }
        // O^T += V^T P^T: A = V^T tiles by ldmatrix.trans (lane l addresses
        // key 16kk + l%8 + 8(l/16), columns 16dt + 8((l/8)%2) ..)
#pragma unroll
        for (int dt = 0; dt < DT; ++dt)
#pragma unroll
          for (int kk = 0; kk < MT; ++kk) {
            uint32_t a[4];
            ldsm_x4_trans(a, smem_u32(vb + chunk_off<D>(16 * kk + (lane & 7) + 8 * (lane >> 4), 2 * dt + ((lane >> 3) & 1))));
            mma_16816_full(o[dt], a, pb[kk][0], pb[kk][1]);
          }
        __syncwarp();
        if (lane == 0) {
          fence_proxy_async_smem();
          if (issue_next<D>(p, is, ring + s * C::STAGE, qarea + s * QN * D, &full[s], uq)) ++issued;
        }
        __syncwarp();
      }
      if (failed) break;
      // column sums over the 8 threads of each query column
#pragma unroll
      for (int e = 0; e < 2; ++e)
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) gl[e] += __shfl_xor_sync(0xffffffffu, gl[e], off);
      const int nsplit = ceil_div(it.nblk, decode_split_blocks(it.nblk));
      const bool direct = nsplit == 1 && !p.null_kv;
      const bool part_in = direct || SMEM_DCHECK((long long)it.pair_begin + U.split < p.part_pairs, p.err);
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int q = 2 * tq + e;
        if (q >= ng || !part_in) continue;
        if (direct) {
          const float inv = 1.f / gl[e];
          uint16_t* dst = p.oca + ((size_t)U.item * p.H + U.h + q) * D + gq;
#pragma unroll
          for (int dt = 0; dt < DT; ++dt) {
            const __nv_bfloat16 b0 = __float2bfloat16_rn(o[dt][e] * inv);
            const __nv_bfloat16 b1 = __float2bfloat16_rn(o[dt][2 + e] * inv);
            dst[16 * dt] = *reinterpret_cast<const uint16_t*>(&b0);
            dst[16 * dt + 8] = *reinterpret_cast<const uint16_t*>(&b1);
          }
        } else {
          float* pp = p.part + ((size_t)(it.pair_begin + U.split) * p.H + U.h + q) * (D + 4);
#pragma unroll
          for (int dt = 0; dt < DT; ++dt) {
            pp[4 + 16 * dt + gq] = o[dt][e];
            pp[4 + 16 * dt + 8 + gq] = o[dt][2 + e];
          }
          if (gq == 0) {
            pp[0] = gm[e];
            pp[1] = gl[e];
          }
        }
      }
      if (direct) continue;
      __threadfence();
      // one ticket per query head, taken by lanes 0 .. ng-1 at once
      const bool mine = lane < ng && atomicAdd(&p.counters[U.item * p.H + U.h + lane], 1u) == (unsigned)(nsplit - 1);
      const unsigned last = __ballot_sync(0xffffffffu, mine);
      if (last) {
        __threadfence();
        merge_group<D, ROPE, QN>(p, U.item, U.h, last, nsplit, it.pair_begin, lane);
      }
      continue;
    }
    const size_t qoff = ((size_t)U.item * p.H + U.h) * D;
    float q[C::QW];
    float m = -INFINITY, l = 0.f, acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.f;
    // Rotary phases (CA): the query turns by W once; a block j read from query
    // block i needs the relative phase min(i - j, W), so only the last W table
    // entries can differ from W -- their keys turn by W - (i - j) on the fly.
    // Their block indices are fetched here, while the first chunk is in flight.
    int near0 = 0x7fffffff, jv0 = 0, jv1 = 0;
    if (ROPE) {
      near0 = max(U.b0, it.nblk - p.rope_w);
      const int* brow = p.bidx + (size_t)it.seq * p.max_blocks;
      if (near0 + lane < U.b0 + U.nt) jv0 = brow[near0 + lane];
      if (near0 + 32 + lane < U.b0 + U.nt) jv1 = brow[near0 + 32 + lane];
    }

    const int nch = U.nt * C::CHUNKS;
    for (int ch = 0; ch < nch; ++ch, ++k) {
      const int s = k % C::NS;
      const uint32_t par = (k / C::NS) & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(&full[s], par, nullptr));
      if (!ok) {
        if (lane == 0) record_error(p.err, kDevErrWaitFull);
        failed = true;
        break;
      }
      if (ch == 0) {
        const uint16_t* qs = qarea + s * QN * D + hh * C::QW;
#pragma unroll
        for (int j = 0; j < C::QW / 8; ++j) {
          float t[8];
          unpack8(*reinterpret_cast<const uint4*>(qs + j * 8), t);
          if (ROPE) rot8f(t, p.rope_tab + (size_t)p.rope_w * (D / 2) + hh * (C::QW / 2) + j * 4);
#pragma unroll
          for (int e = 0; e < 8; ++e) q[j * 8 + e] = t[e] * p.scale_log2;
        }
      }
      int dk = 0;  // extra key phase of this chunk's block (0: none)
      if (ROPE) {
        const int bp = U.b0 + ch / C::CHUNKS;
        if (bp >= near0) {
          const int o = bp - near0;
          const int j = __shfl_sync(0xffffffffu, o < 32 ? jv0 : jv1, o & 31);
          dk = max(0, p.rope_w - (it.qblk - j));
        }
      }
      const uint8_t* kb = ring + s * C::STAGE;
      const uint8_t* vb = kb + C::HALF;
      if constexpr (D == 32) {
        // scores: two rows per lane (rows lane and lane + 32), 64-byte rows
        float sc2[2];
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const int r = lane + 32 * h2;
          float dot = 0.f;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            float t[8];
            unpack8(*reinterpret_cast<const uint4*>(kb + chunk_off<D>(r, j)), t);
            if (ROPE && dk > 0) rot8f(t, p.rope_tab + (size_t)dk * (D / 2) + j * 4);
#pragma unroll
            for (int e = 0; e < 8; ++e) dot = fmaf(q[j * 8 + e], t[e], dot);
          }
          sc2[h2] = dot;
        }
        float mx = fmaxf(sc2[0], sc2[1]);
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_new = fmaxf(m, mx);
        const float alpha = exp2f(m - m_new);
        const float p0 = exp2f(sc2[0] - m_new), p1 = exp2f(sc2[1] - m_new);
        l = l * alpha + p0 + p1;
        pbuf[lane] = p0;
        pbuf[lane + 32] = p1;
        m = m_new;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] *= alpha;
      } else {
        // scores: lane-per-row (two lanes per row at d_h = 128)
        float dot0 = 0.f, dot1 = 0.f;
        const uint8_t* krow = kb + hh * C::BOX_BYTES + rr * 128;
        if (ROPE && dk > 0) {
          const float2* cs = p.rope_tab + (size_t)dk * (D / 2) + hh * 32;
  #pragma unroll
          for (int j = 0; j < 8; j += 2) {
            float t0[8], t1[8];
            unpack8(*reinterpret_cast<const uint4*>(krow + ((j ^ (rr & 7)) << 4)), t0);
            unpack8(*reinterpret_cast<const uint4*>(krow + (((j + 1) ^ (rr & 7)) << 4)), t1);
            rot8f(t0, cs + j * 4);
            rot8f(t1, cs + j * 4 + 4);
  #pragma unroll
            for (int e = 0; e < 8; ++e) {
              dot0 = fmaf(q[j * 8 + e], t0[e], dot0);
              dot1 = fmaf(q[j * 8 + 8 + e], t1[e], dot1);
            }
          }
        } else {
  #pragma unroll
          for (int j = 0; j < 8; j += 2) {
            float t0[8], t1[8];
            unpack8(*reinterpret_cast<const uint4*>(krow + ((j ^ (rr & 7)) << 4)), t0);
            unpack8(*reinterpret_cast<const uint4*>(krow + (((j + 1) ^ (rr & 7)) << 4)), t1);
  #pragma unroll
            for (int e = 0; e < 8; ++e) {
              dot0 = fmaf(q[j * 8 + e], t0[e], dot0);
              dot1 = fmaf(q[j * 8 + 8 + e], t1[e], dot1);
            }
          }
        }
        float sc = dot0 + dot1;
        if (C::LPR == 2) sc += __shfl_xor_sync(0xffffffffu, sc, 1);
        float mx = sc;
  #pragma unroll
        for (int o = C::LPR; o < 32; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_new = fmaxf(m, mx);
        const float alpha = exp2f(m - m_new);
        const float pr = exp2f(sc - m_new);
        l = l * alpha + (hh == 0 ? pr : 0.f);
        if (hh == 0) pbuf[rr] = pr;
        m = m_new;
  #pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] *= alpha;
      }
      __syncwarp();
      // P.V: lane (g, c), rows g*RG .. g*RG+RG-1, columns c*8 .. c*8+7
      const float4 p0 = *reinterpret_cast<const float4*>(pbuf + g * RG);
      const float4 p1 = *reinterpret_cast<const float4*>(pbuf + g * RG + 4);
      const float pv[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
      const uint8_t* vcol = vb + (D == 32 ? 0 : (c >> 3) * C::BOX_BYTES);
      const int cc = D == 32 ? c : (c & 7);
#pragma unroll
      for (int i = 0; i < RG; ++i) {
        const int r = g * RG + i;
        float t[8];
        const int off = D == 32 ? r * 64 + ((cc ^ ((r >> 1) & 3)) << 4) : r * 128 + ((cc ^ (r & 7)) << 4);
        unpack8(*reinterpret_cast<const uint4*>(vcol + off), t);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = fmaf(pv[i], t[e], acc[e]);
      }
      __syncwarp();
      // refill this stage with the chunk NS ahead
      if (lane == 0) {
        fence_proxy_async_smem();
        if (issue_next<D>(p, is, ring + s * C::STAGE, qarea + s * QN * D, &full[s], uq)) ++issued;
      }
      __syncwarp();
    }
    if (failed) break;

    // merge the row groups and the lanes of the warp (fixed butterflies)
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
#pragma unroll
    for (int o = CPL; o < 32; o <<= 1)
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);

    const int nsplit = ceil_div(it.nblk, decode_split_blocks(it.nblk));
    if (nsplit == 1 && !p.null_kv) {
      if (g == 0) store_bf16x8(p.oca + qoff + c * 8, acc, 1.f / l);
      continue;
    }
    settle<D, ROPE>(p, pend2, lane);
    announce(p, pend1, pend2, lane);
    const bool part_in = SMEM_DCHECK((long long)it.pair_begin + U.split < p.part_pairs, p.err);
    float* pp = p.part + ((size_t)(it.pair_begin + U.split) * p.H + U.h) * (D + 4);
    if (g == 0 && part_in) {
      *reinterpret_cast<float4*>(pp + 4 + c * 8) = make_float4(acc[0], acc[1], acc[2], acc[3]);
      *reinterpret_cast<float4*>(pp + 8 + c * 8) = make_float4(acc[4], acc[5], acc[6], acc[7]);
    }
    if (lane == 0 && part_in) {
      pp[0] = m;
      pp[1] = l;
    }
    pend1.valid = 1;
    pend1.item = U.item;
    pend1.h = U.h;
    pend1.nsplit = nsplit;
    pend1.pair_begin = it.pair_begin;
  }

  if (!failed) {
    settle<D, ROPE>(p, pend2, lane);
    announce(p, pend1, pend2, lane);
    settle<D, ROPE>(p, pend2, lane);
    // Self-attention units (in-block rows, read from global memory), fetched
    // from their own counter once the warp's cross-attention stream has
    // ended: they fill the launch's tail instead of holding every warp's
    // first stage behind a memory system still busy with the ring
    // prologues. They read no row and write no output that a cross-attention
    // unit of the launch uses.
    const int n_sa = p.n_items * p.H;
    while (true) {
      int v = 0;
      if (lane == 0) v = (int)min(atomicAdd(p.sched + 2, 1ull), (unsigned long long)n_sa);
      v = __shfl_sync(0xffffffffu, v, 0);
      if (v >= n_sa) break;
      Unit U;
      U.sa = 1;
      U.item = v / p.H;
      U.h = v - U.item * p.H;
      U.split = U.b0 = U.nt = 0;
      sa_unit<D, ROPE>(p, U, pbuf, lane);
    }
  }
  if (lane == 0) {
    if (failed) {
      // let copies already in flight land (bounded) before the warp exits
      for (int j = k; j < issued; ++j) mbar_wait_bounded(&full[j % C::NS], (j / C::NS) & 1, nullptr);
    }
    // the last warp out resets the unit counter for the next launch
    const unsigned long long done = atomicAdd(p.sched + 1, 1ull);
    if (done == (unsigned long long)gridDim.x * C::NW - 1) {
      p.sched[0] = 0ull;
      p.sched[1] = 0ull;
      p.sched[2] = 0ull;  // next self-attention unit
    }
  }
}

// Fixed scratch of smem_decode_static_scratch: split partials, tickets and
// scheduler words for callers that cannot allocate. Host code sees only a
// stand-in symbol; the device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_decode_static_scratch[SMEM_STATIC_SCRATCH_BYTES];

int static_scratch_address(void** out) {
  // The address belongs to the device's context: it is looked up once per
  // (device, context) and looked up again when the current context changed
  // (e.g. after cudaDeviceReset made a new primary context).
  constexpr int kMaxDevices = 64;
  static std::mutex mu;
  static void* addr[kMaxDevices] = {};
  static CUcontext owner[kMaxDevices] = {};
  static PFN_cuCtxGetCurrent_v4000 get_ctx = nullptr;
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return (int)e;
  if (dev < 0 || dev >= kMaxDevices) return (int)cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (!get_ctx) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 4000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return (int)cudaErrorNotSupported;
    get_ctx = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(fn);
  }
  CUcontext ctx = nullptr;
  if (get_ctx(&ctx) != CUDA_SUCCESS) return (int)cudaErrorDeviceUninitialized;
  if (!addr[dev] || !ctx || ctx != owner[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_decode_static_scratch);  // this device is current
    if (e != cudaSuccess) return (int)e;
    if (!p) return (int)cudaErrorInvalidSymbol;
    if (get_ctx(&ctx) != CUDA_SUCCESS || !ctx) return (int)cudaErrorDeviceUninitialized;
    addr[dev] = p;
    owner[dev] = ctx;
  }
  *out = addr[dev];
  return 0;
}

int decode_stage_rows(int D) { return D == 32 ? Dec<32>::SROWS : D == 64 ? Dec<64>::SROWS : Dec<128>::SROWS; }

int encode_pool_map(CUtensorMap* map, void* pool, int L, int H, int D, int capacity, int rows_per_box) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return -1;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)L * H * 2 * kRows, (cuuint64_t)capacity};
  const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)D * 2 * L * H * 2 * kRows};
  // rows of 64 columns (128 bytes, 128-byte swizzle) or of 32 (64 bytes, 64-byte swizzle)
  const cuuint32_t box[3] = {(cuuint32_t)(D < 64 ? D : 64), (cuuint32_t)rows_per_box, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, pool, dims, strides, box, estr,
                            CU_TENSOR_MAP_INTERLEAVE_NONE,
                            D < 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : (int)r;
}

int decode_max_grid(int D, int num_sms) {
  (void)D;
  return num_sms;
}

int decode_warps_per_cta() { return Dec<64>::NW; }

template <int D, bool ROPE, int QN>
static cudaError_t launch_decode_d(const DecodeParams& p, int grid, cudaStream_t st) {
  using C = Dec<D, QN>;
  cudaError_t e = ensure_smem_limit<D + (ROPE ? 1 : 0) + 4 * QN>(decode_kernel<D, ROPE, QN>, C::SMEM);
  if (e != cudaSuccess) return e;
  decode_kernel<D, ROPE, QN><<<grid, C::THREADS, C::SMEM, st>>>(p);
  return cudaGetLastError();
}

int decode_group_width(int D, int G, bool rope) {
  // query heads per grouped unit: the largest of 4 (2 at d_h = 128, whose
  // rings leave less shared memory) dividing the group; 1 with rotary phases
  if (rope || G < 2) return 1;
  const int qmax = D == 128 ? 2 : 4;
  for (int q = qmax; q >= 2; q >>= 1)
    if (G % q == 0) return q;
  return 1;
}

cudaError_t launch_decode(const DecodeParams& p, int D, int grid, cudaStream_t st) {
  const bool rope = p.rope_tab != nullptr;
  if (p.qn > 1) {
    if (rope) return cudaErrorInvalidValue;
    if (D == 32) return launch_decode_d<32, false, 4>(p, grid, st);
    if (D == 64) return launch_decode_d<64, false, 4>(p, grid, st);
    if (D == 128) return launch_decode_d<128, false, 2>(p, grid, st);
    return cudaErrorInvalidValue;
  }
  if (D == 32) return rope ? launch_decode_d<32, true, 1>(p, grid, st) : launch_decode_d<32, false, 1>(p, grid, st);
  if (D == 64) return rope ? launch_decode_d<64, true, 1>(p, grid, st) : launch_decode_d<64, false, 1>(p, grid, st);
  if (D == 128) return rope ? launch_decode_d<128, true, 1>(p, grid, st) : launch_decode_d<128, false, 1>(p, grid, st);
  return cudaErrorInvalidValue;
}

}  // namespace smem
