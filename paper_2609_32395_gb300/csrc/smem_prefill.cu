// smem_prefill.cu -- one-block reader pass for one layer (block-skip serving).
//
// For the b = 64 query tokens of the final block (arXiv 2609.32395, Sec. 3.1
// "Reuse": a fully cached context is served by running the reader on the
// final block alone; Sec. 2 "Model" and App. A "Reader" for the attention):
//   Osa[t] = softmax_{u<=t}(s Qs[t].Ks[u]) Vs        block-local causal SA
//   Oca[t] = softmax_r(s Qc[t].k_r) v_r               block-causal CA
// where r runs over the null row and the rows of every table block with index
// below the query block, in ascending block index.
//
// The CA scores and P.V form a dense (64 x N.R) x (N.R x d_h) contraction, so
// they run on the 5th-generation tensor cores: per CTA, one (head, split)
// work unit. A producer warp streams the split's K and V tiles (64 rows x
// d_h, 128-byte swizzle) into a ring with tensor TMA; an MMA warp issues
// S = Q.K^T (M = 64 queries, N = 64 keys) into one of two TMEM buffers and
// O += P.V (N = d_h, V read MN-major) into a TMEM accumulator; four softmax
// warps read S rows from TMEM (row 16w + t%16, half t/16 of the keys), run a
// base-2 online softmax, and write P as bf16 into a swizzled smem tile. The
// running maximum is raised only when a row's maximum grows by more than 2^8
// (then that row of O is rescaled in TMEM); otherwise the stale maximum keeps
// every P <= 256, and O and l stay consistent with it. The MMA warp issues
// QK^T two tiles ahead of P.V, so a score tile is in TMEM a whole softmax
// pass before it is read. A split writes its partial (m, l, O) and the CTA
// that completes the last split of a head merges all splits in split order
// (null row first); in cluster mode the partials stay in shared memory and
// the cluster merges them over DSMEM. The in-block SA is one masked tile per
// head on the same machinery. Reduction orders depend only on the block
// count.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>

#include "smem_device.cuh"
#include "smem_internal.h"
#include "smem_tc.cuh"

namespace smem {

template <int D>
struct Pf {
  static constexpr int R = kRows;
  static constexpr int B = kBlockTok;
  static constexpr int BOXES = D < 64 ? 1 : D / 64;  // column boxes (128 bytes wide; one of 64 bytes at d_h = 32)
  static constexpr int BOX = 64 * (D < 64 ? D * 2 : 128);  // one [64 rows][box width] box
  static constexpr int TILE = BOXES * BOX;        // K or V of one block and head
  static constexpr int STAGE = 2 * TILE;
  // A stage holds, per column box bx, the K box then the V box of the same
  // columns (one TMA copy of 128 pool rows each): K box bx at bx * KVS, V
  // box bx at bx * KVS + BOX. Fewer, larger copies keep the producer thread
  // below its TMA instruction rate.
  static constexpr int KVS = 2 * BOX;
  // ring stages: two CTAs per SM at d_h <= 64; at d_h = 128 one CTA per SM
  // whose six 32 KB stages keep ~190 KB of copies in flight (four measured
  // 74% of HBM over a long context, six 97%: the stream is bound by bytes
  // in flight times the load latency)
  static constexpr int NS = D == 32 ? 8 : (D == 64 ? 5 : 6);
  static constexpr int PBYTES = 64 * 64 * 2;      // P tile [64 queries][64 keys] bf16
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_RING = TILE;
  static constexpr int OFF_P = OFF_RING + NS * STAGE;
  static constexpr int OFF_BAR = OFF_P + 2 * PBYTES;
  // barriers: q_full | full[NS] | empty[NS] | s_full[2] | s_free[2] | p_full[2] | o_done[2] | drain | merge
  static constexpr int NBARS = 1 + 2 * NS + 10;
  static constexpr int OFF_MISC = OFF_BAR + NBARS * 8;
  static constexpr int SMEM = OFF_MISC + 64 + 1024;
  static constexpr int THREADS = 192;             // 4 softmax warps, producer, MMA
  static constexpr int MIN_CTAS = D <= 64 ? 2 : 1; // resident CTAs per SM (smem and TMEM allow it)
  static constexpr uint32_t TMEM_COLS = 256;      // S0 | S1 | O
  static constexpr uint32_t COL_O = 128;
  static constexpr uint32_t ID_QK = tc::idesc_bf16(64, 64, 0, 0);
  static constexpr uint32_t ID_PV = tc::idesc_bf16(64, D, 0, 1);
  static constexpr int PART_BYTES = B * (D + 4) * 4;          // one split's partial rows
  static constexpr int MERGE_SPR = NS * STAGE / PART_BYTES;   // split partials staged per round
};

static_assert(2 * (Pf<64>::SMEM + 1024) <= 228 * 1024, "two d_h = 64 CTAs per SM");
static_assert(Pf<128>::SMEM <= 227 * 1024, "one d_h = 128 CTA per SM");

// Shared-memory descriptors of the K-major Q/K tiles (k-th step of 16
// columns) and of the MN-major V tile (k-th step of 16 rows).
// `stride`: bytes from one column box to the next (BOX for the query tile,
// KVS for a key tile in a stage).
template <int D>
__device__ __forceinline__ uint64_t qk_desc(uint32_t base, int k, int stride) {
  if constexpr (D == 32) return tc::sdesc_sw64(base + k * 32, 16, 512);
  else return tc::sdesc_sw128(base + (k >> 2) * stride + (k & 3) * 32, 16, 1024);
}
template <int D>
__device__ __forceinline__ uint64_t v_desc(uint32_t base, int k) {
  if constexpr (D == 32) return tc::sdesc_sw64(base + k * 1024, Pf<D>::KVS, 512);
  else return tc::sdesc_sw128(base + k * 2048, Pf<D>::KVS, 1024);
}

// O columns of a softmax thread (its half of the row), read or written in TMEM.
template <int D>
__device__ __forceinline__ void ld_o(uint32_t trow, uint32_t (&o)[D / 2]) {
  if constexpr (D == 32) {
    tc::ld_16x32bx2_x16<16>(trow, o);
  } else {
#pragma unroll
    for (int cb = 0; cb < D / 64; ++cb) {
      uint32_t t[32];
      tc::ld_16x32bx2_x32<D / 2>(trow + 32 * cb, t);
#pragma unroll
      for (int c = 0; c < 32; ++c) o[cb * 32 + c] = t[c];
    }
  }
}
template <int D>
__device__ __forceinline__ void st_o(uint32_t trow, const uint32_t (&o)[D / 2]) {
  if constexpr (D == 32) {
    tc::st_16x32bx2_x16<16>(trow, o);
  } else {
#pragma unroll
    for (int cb = 0; cb < D / 64; ++cb) {
      uint32_t t[32];
#pragma unroll
      for (int c = 0; c < 32; ++c) t[c] = o[cb * 32 + c];
      tc::st_16x32bx2_x32<D / 2>(trow + 32 * cb, t);
    }
  }
}

constexpr float kRescaleLog2 = 8.0f;  // raise the running max when it grows by more than 2^8

// 2^x by the hardware's approximate base-2 exponential (PTX ex2.approx.ftz:
// relative error near 2^-22, subnormal results flushed to zero). The
// arguments here are at most kRescaleLog2 and the results are rounded to
// bf16 for the P.V product.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

struct PrefillParams {
  CUtensorMap pool;          // [C][L*H*2*R][D], box 64 columns x 128 rows (a block's K then V)
  CUtensorMap qs, ks, vs, qc;  // [b][H][D], box 64 x 1 x 64
  const int* table_row;
  const uint16_t* null_kv;
  const uint16_t* qc_ptr;
  uint16_t* osa;
  uint16_t* oca;
  float* part;
  unsigned* counters;
  int* err;
  int L, H, layer, nblk, split_blks, n_splits, capacity, max_splits, max_blocks;
  int Hkv;             // key/value heads (H / Hkv query heads share one)
  int mode;            // bit 0: in-block self-attention, bit 1: cross-attention
  int n_sa;            // self-attention CTAs of the cluster-free grid (0 or H)
  int tok_c;           // elements between consecutive tokens of Qc
  float scale_log2;
  const float2* rope_tab;  // rotary table [kRopePhases][D/2] (ROPE kernels only)
  const int* bidx_row;     // block index of each table entry of the sequence
  int rope_w, q_blk;       // saturating window W, the query block's index
  int rope_half;           // D/2: pairs per table row
};

// (x[2m], x[2m+1]) of 8 values turned by table pairs cs[0..3].
__device__ __forceinline__ void rot8(float* t, const float2* cs) {
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 c = cs[e];
    const float x0 = t[2 * e], x1 = t[2 * e + 1];
    t[2 * e] = x0 * c.x - x1 * c.y;
    t[2 * e + 1] = x0 * c.y + x1 * c.x;
  }
}

// Turns a [64 rows][D] bf16 tile (D/64 boxes of [64][128 B], 128-byte
// swizzle) in place by one table row; one warp, then a proxy fence so that
// the tensor cores see the new values.
template <int D>
__device__ void rotate_tile(uint8_t* tile, const float2* cs_row, int lane, int stride) {
  constexpr int CH = D / 8;  // 16-byte chunks per row
  for (int i = lane; i < 64 * CH; i += 32) {
    const int r = i / CH, c = i % CH;
    uint8_t* ptr = D == 32 ? tile + r * 64 + ((c ^ ((r >> 1) & 3)) << 4)
                           : tile + (c >> 3) * stride + r * 128 + ((((c & 7) ^ (r & 7))) << 4);
    float t[8];
    unpack8(*reinterpret_cast<const uint4*>(ptr), t);
    rot8(t, cs_row + c * 4);
    *reinterpret_cast<uint4*>(ptr) = make_uint4(pack_bf16x2(t[0], t[1]), pack_bf16x2(t[2], t[3]),
                                                pack_bf16x2(t[4], t[5]), pack_bf16x2(t[6], t[7]));
  }
  fence_proxy_async_smem();
  __syncwarp();
}

// A query row's cross-attention null-row score (its columns col0 ..
// col0+n-1): with rotary phases the null row's key sits at phase
// max(0, i - W), so the query turns by min(i, W).
template <bool ROPE>
__device__ __forceinline__ float null_dot(const PrefillParams& p, const uint16_t* q, const uint16_t* kn, int col0,
                                          int n) {
  float dot = 0.f;
  const float2* cs = ROPE ? p.rope_tab + (size_t)min(p.q_blk, p.rope_w) * (p.rope_half) + col0 / 2 : nullptr;
  for (int c = 0; c < n; c += 2) {
    float x0 = bf16lo(q[col0 + c]), x1 = bf16lo(q[col0 + c + 1]);
    if (ROPE) {
      const float2 r = cs[c / 2];
      const float y0 = x0 * r.x - x1 * r.y;
      x1 = x0 * r.y + x1 * r.x;
      x0 = y0;
    }
    dot = fmaf(x0, bf16lo(kn[col0 + c]), dot);
    dot = fmaf(x1, bf16lo(kn[col0 + c + 1]), dot);
  }
  return dot;
}

// Cluster mode (d_h = 64): one cluster of n_splits + 1 CTAs per head, rank 0
// the in-block SA tile and rank k the split k-1. Each split CTA parks its
// partial rows (m, l, O) in its own shared memory, and rank 0 parks the null
// row as a partial of its own (m = its score, l = 1, O = its value row);
// after a cluster barrier every CTA merges a slice of the 64 rows, one row
// per warp, summing in rank order (null row first). Lane s fetches rank s's
// (m, l) and the warp shares them by shuffles; every lane fetches its columns
// of every rank's O; all remote loads of a row go out in one batch. A warp
// arrives on the closing cluster barrier once it has consumed the last remote
// values it reads (a relaxed arrival: the values are in registers by then, so
// it need not wait for the warp's output stores), and the caller waits on it:
// no CTA leaves while another still reads its shared memory.
template <int D>
__device__ void cluster_merge(const PrefillParams& p, int h, uint32_t rank, uint32_t cs, uint32_t stage_saddr,
                              int warp, int lane) {
  constexpr int CPL = D / 32;  // columns per lane
  const int rp = (kBlockTok + (int)cs - 1) / (int)cs;
  const int r0 = (int)rank * rp, r1 = min(kBlockTok, r0 + rp);
  if (r0 + warp >= r1) tc::cluster_arrive_relaxed();  // no row for this warp
  for (int row = r0 + warp; row < r1; row += 6) {
    const uint32_t row_saddr = stage_saddr + (uint32_t)(row * (D + 4) * 4);
    const float2 mlv = lane < (int)cs ? tc::ld_dsmem_f32x2(tc::dsmem_addr(row_saddr, (uint32_t)lane))
                                      : make_float2(-INFINITY, 0.f);
    float2 ov[kPrefillMaxSplits][CPL / 2];
#pragma unroll
    for (int s2 = 0; s2 < kPrefillMaxSplits; ++s2) {
      const uint32_t ra = s2 < (int)cs ? tc::dsmem_addr(row_saddr, (uint32_t)s2) : 0u;
#pragma unroll
      for (int e = 0; e < CPL / 2; ++e)
        ov[s2][e] = s2 < (int)cs ? tc::ld_dsmem_f32x2(ra + 16 + (lane * CPL + 2 * e) * 4) : make_float2(0.f, 0.f);
    }
    float M = mlv.x;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    const float fl = exp2f(mlv.x - M);  // lane s: rank s's factor
    float Lsum = 0.f, A[CPL];
#pragma unroll
    for (int e = 0; e < CPL; ++e) A[e] = 0.f;
#pragma unroll
    for (int s2 = 0; s2 < kPrefillMaxSplits; ++s2) {
      if (s2 >= (int)cs) break;
      const float f = __shfl_sync(0xffffffffu, fl, s2);
      Lsum = fmaf(f, __shfl_sync(0xffffffffu, mlv.y, s2), Lsum);
#pragma unroll
      for (int e = 0; e < CPL / 2; ++e) {
        A[2 * e] = fmaf(f, ov[s2][e].x, A[2 * e]);
        A[2 * e + 1] = fmaf(f, ov[s2][e].y, A[2 * e + 1]);
      }
    }
    if (row + 6 >= r1) tc::cluster_arrive_relaxed();  // this warp's last remote values are consumed
    const float inv = 1.f / Lsum;
    const size_t qoff = ((size_t)row * p.H + h) * D;
    uint32_t* o32 = reinterpret_cast<uint32_t*>(p.oca + qoff) + lane * (CPL / 2);
#pragma unroll
    for (int e = 0; e < CPL / 2; ++e) o32[e] = pack_bf16x2(A[2 * e] * inv, A[2 * e + 1] * inv);
  }
}

template <int D, bool CL, bool ROPE>
__global__ void __launch_bounds__(Pf<D>::THREADS, Pf<D>::MIN_CTAS) prefill_kernel(const __grid_constant__ PrefillParams p) {
  using C = Pf<D>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint8_t* qt = base + C::OFF_Q;
  uint8_t* ring = base + C::OFF_RING;
  uint8_t* pt = base + C::OFF_P;
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::OFF_BAR);
  uint64_t* q_full = bars;
  uint64_t* full = bars + 1;
  uint64_t* empty = full + C::NS;
  uint64_t* s_full = empty + C::NS;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* o_done = p_full + 2;
  uint64_t* drain = o_done + 2;
  uint64_t* mbar_merge = drain + 1;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(base + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + C::OFF_MISC + 4);
  volatile unsigned* ticket = reinterpret_cast<volatile unsigned*>(base + C::OFF_MISC + 8);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // without clusters the short self-attention CTAs come first and leave
  // their SMs early; in cluster mode a head is a cluster and rank 0 its SA
  const uint32_t cs = (uint32_t)p.n_splits + 1;
  const uint32_t crank = CL ? tc::cluster_ctarank() : 0u;
  const bool sa = CL ? crank == 0 : (int)blockIdx.x < p.n_sa;
  const int cb = (int)blockIdx.x - p.n_sa;
  const int h = CL ? (int)(blockIdx.x / cs) : (sa ? (int)blockIdx.x : cb % p.H);
  const int split = CL ? (int)crank - 1 : (sa ? 0 : cb / p.H);
  const int b0 = split * p.split_blks;
  // an SA CTA without the SA half to do only joins the merge (cluster mode)
  // or writes the empty-memory cross-attention output
  const int nt = sa ? ((p.mode & 1) ? 1 : 0) : min(p.split_blks, p.nblk - b0);
  const bool work = nt > 0;

  if (threadIdx.x == 128) {
    // the tensor maps are kernel parameters, not the previous kernel's output
    const CUtensorMap* maps[5] = {&p.pool, &p.qs, &p.ks, &p.vs, &p.qc};
#pragma unroll
    for (int i = 0; i < 5; ++i)
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(maps[i])) : "memory");
  }
  if (threadIdx.x == 0) {
    griddep_launch();
    mbar_init(q_full, 1);
    for (int s = 0; s < C::NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_free[b], 4);
      mbar_init(&p_full[b], 4);
      mbar_init(&o_done[b], 1);
    }
    mbar_init(drain, 1);
    mbar_init(mbar_merge, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 4) tc::alloc(tslot, C::TMEM_COLS);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = *tslot;
  // launched with programmatic dependent launch: everything above overlaps
  // the previous kernel; every global read and write comes after this wait
  griddep_wait();

  if (warp == 4) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0 && work) {
      const CUtensorMap* qmap = sa ? &p.qs : &p.qc;
      mbar_arrive_expect_tx(q_full, C::TILE);
#pragma unroll
      for (int bx = 0; bx < C::BOXES; ++bx) tc::tma_load_3d(qt + bx * C::BOX, qmap, bx * 64, h, 0, q_full);
      int issued = 0;
      for (int j = 0; j < nt; ++j) {
        const int st = j % C::NS;
        if (j >= C::NS && !mbar_wait_bounded(&empty[st], ((j / C::NS) - 1) & 1, abort_flag)) {
          if (!*abort_flag) record_error(p.err, kDevErrWaitEmpty);
          *abort_flag = 1;
          break;
        }
        uint8_t* kd = ring + st * C::STAGE;
        if (sa) {
          mbar_arrive_expect_tx(&full[st], C::STAGE);
#pragma unroll
          for (int bx = 0; bx < C::BOXES; ++bx) {
            tc::tma_load_3d(kd + bx * C::KVS, &p.ks, bx * 64, h / (p.H / p.Hkv), 0, &full[st]);
            tc::tma_load_3d(kd + bx * C::KVS + C::BOX, &p.vs, bx * 64, h / (p.H / p.Hkv), 0, &full[st]);
          }
        } else {
          const bool in_range =
              SMEM_DCHECK(b0 + j >= 0 && b0 + j < p.nblk && p.nblk <= p.max_blocks && split < p.max_splits, p.err);
          const int slot = in_range ? p.table_row[b0 + j] : -1;
          if (slot < 0 || slot >= p.capacity) {
            record_error(p.err, kDevErrBounds);
            mbar_arrive(&full[st]);
          } else {
            mbar_arrive_expect_tx(&full[st], C::STAGE);
            const int y = ((p.layer * p.Hkv + h / (p.H / p.Hkv)) * 2) * C::R;
#pragma unroll
            for (int bx = 0; bx < C::BOXES; ++bx)  // the K rows and then the V rows of these columns
              tc::tma_load_3d(kd + bx * C::KVS, &p.pool, bx * 64, y, slot, &full[st]);
          }
        }
        ++issued;
      }
      if (*abort_flag) {
        mbar_wait_bounded(q_full, 0, nullptr);
        for (int j = 0; j < issued; ++j) mbar_wait_bounded(&full[j % C::NS], (j / C::NS) & 1, nullptr);
      }
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------- MMA issuer
    // The whole warp runs the loop, so control flow and descriptors stay
    // warp-uniform; one elected lane issues the MMAs. QK^T runs two tiles
    // ahead of P.V: S[j%2] is refilled with tile j+2 as soon as the softmax
    // warps have read tile j out of it (s_free), so every score tile is ready
    // a whole softmax pass before it is needed. With rotary phases the warp
    // turns the query tile by W once and the key tile of every near block j
    // (the last W table entries) by W - (i - j), so that each score sees the
    // relative phase min(i - j, W).
    if (work) {
      const bool leader = tc::elect_one();
      const bool rot = ROPE && !sa;
      bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(q_full, 0, abort_flag));
      int near0 = 0, jv0 = 0, jv1 = 0;
      if (rot) {
        near0 = max(b0, p.nblk - p.rope_w);
        if (near0 + lane < b0 + nt) jv0 = p.bidx_row[near0 + lane];
        if (near0 + 32 + lane < b0 + nt) jv1 = p.bidx_row[near0 + 32 + lane];
        if (ok) {
          tc::fence_after();
          rotate_tile<D>(qt, p.rope_tab + (size_t)p.rope_w * (D / 2), lane, C::BOX);
        }
      }
      const uint32_t qa = smem_u32(qt);
      // S[j%2] = Q . K_j^T
      auto issue_qk = [&](int j) -> bool {
        const int st = j % C::NS, sb = j & 1;
        bool r = __all_sync(0xffffffffu, mbar_wait_bounded(&full[st], (j / C::NS) & 1, abort_flag));
        if (r && j >= 2) r = __all_sync(0xffffffffu, mbar_wait_bounded(&s_free[sb], ((j >> 1) - 1) & 1, abort_flag));
        if (!r) return false;
        tc::fence_after();
        if (rot && b0 + j >= near0) {
          const int o = b0 + j - near0;
          const int jb = __shfl_sync(0xffffffffu, o < 32 ? jv0 : jv1, o & 31);
          const int dk = max(0, p.rope_w - (p.q_blk - jb));
          if (dk > 0) rotate_tile<D>(ring + st * C::STAGE, p.rope_tab + (size_t)dk * (D / 2), lane, C::KVS);
        }
        const uint32_t ka = smem_u32(ring + st * C::STAGE);
        uint64_t ad[D / 16], bd[D / 16];
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          ad[k] = qk_desc<D>(qa, k, C::BOX);
          bd[k] = qk_desc<D>(ka, k, C::KVS);
        }
        if (leader) {
#pragma unroll
          for (int k = 0; k < D / 16; ++k) tc::mma_bf16(tmem + 64 * sb, ad[k], bd[k], C::ID_QK, k > 0);
          tc::commit(&s_full[sb]);
        }
        __syncwarp();
        return true;
      };
      if (ok) tc::fence_after();
      for (int j = 0; ok && j < min(2, nt); ++j) ok = issue_qk(j);
      for (int j = 0; ok && j < nt; ++j) {
        if (j + 2 < nt && !(ok = issue_qk(j + 2))) break;
        // O += P_j . V_j
        const int st = j % C::NS, pb = j & 1;
        ok = __all_sync(0xffffffffu, mbar_wait_bounded(&p_full[pb], (j >> 1) & 1, abort_flag));
        if (!ok) break;
        tc::fence_after();
        const uint32_t pa = smem_u32(pt + pb * C::PBYTES);
        const uint32_t va = smem_u32(ring + st * C::STAGE + C::BOX);
        uint64_t ad[4], bd[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          ad[k] = tc::sdesc_sw128(pa + k * 32, 16, 1024);
          bd[k] = v_desc<D>(va, k);
        }
        if (leader) {
#pragma unroll
          for (int k = 0; k < 4; ++k) tc::mma_bf16(tmem + C::COL_O, ad[k], bd[k], C::ID_PV, (j > 0 || k > 0));
          tc::commit(&empty[st]);
          tc::commit(&o_done[pb]);
        }
        __syncwarp();
      }
      if (!ok) {
        if (leader && !*abort_flag) record_error(p.err, kDevErrWaitMma);
        __syncwarp();
        *abort_flag = 1;
      }
      // all issued MMAs complete before the CTA can release TMEM
      if (leader) {
        tc::commit(drain);
        mbar_wait_bounded(drain, 0, nullptr);
      }
      __syncwarp();
    }
  } else {
    // ---------------------------------------------------------- softmax warps
    const int r = 16 * warp + (lane & 15);  // query row
    const int hf = lane >> 4;               // key half of the S tile
    const uint32_t trow = tmem + ((uint32_t)(32 * warp) << 16);
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nt && ok; ++j) {
      const int sb = j & 1;
      ok = __all_sync(0xffffffffu, mbar_wait_bounded(&s_full[sb], (j >> 1) & 1, abort_flag));
      if (!ok) break;
      tc::fence_after();
      uint32_t sr[32];
      tc::ld_16x32bx2_x32<32>(trow + 64 * sb, sr);
      tc::wait_ld();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[sb]);
      float x[32];
#pragma unroll
      for (int c = 0; c < 32; ++c) x[c] = __uint_as_float(sr[c]);
      if (sa) {  // causal mask of the in-block tile
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (hf * 32 + c > r) x[c] = -INFINITY;
      }
      // row maximum of the raw scores as a tree; the base-2 scale is
      // positive and rounding is monotone, so the scaled maximum equals the
      // maximum of the scaled scores
      float t[16];
#pragma unroll
      for (int c = 0; c < 16; ++c) t[c] = fmaxf(x[c], x[c + 16]);
#pragma unroll
      for (int w2 = 8; w2 >= 1; w2 >>= 1)
#pragma unroll
        for (int c = 0; c < w2; ++c) t[c] = fmaxf(t[c], t[c + w2]);
      float tmax = t[0] * p.scale_log2;
      tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 16));
      const float m_new = fmaxf(m_used, tmax);
      const bool need = m_new > m_used + kRescaleLog2;
      if (j > 0 && __any_sync(0xffffffffu, need)) {
        // rescale this warp's rows of O once the previous P.V has landed
        ok = __all_sync(0xffffffffu, mbar_wait_bounded(&o_done[(j - 1) & 1], ((j - 1) >> 1) & 1, abort_flag));
        if (!ok) break;
        tc::fence_after();
        const float alpha = need ? exp2f(m_used - m_new) : 1.f;
        {
          uint32_t o[D / 2];
          ld_o<D>(trow + C::COL_O, o);
          tc::wait_ld();
#pragma unroll
          for (int c = 0; c < D / 2; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * alpha);
          st_o<D>(trow + C::COL_O, o);
        }
        tc::wait_st();
      }
      if (need) {
        l *= exp2f(m_used - m_new);
        m_used = m_new;
      }
      // P = 2^(s * scale - m): one FMA and one ex2 per score; the row sum
      // in four independent partial sums
      uint32_t pk[16];
      float la[4] = {0.f, 0.f, 0.f, 0.f};
      const float nm = -m_used;
#pragma unroll
      for (int c = 0; c < 32; c += 2) {
        const float p0 = ex2_approx(fmaf(x[c], p.scale_log2, nm));
        const float p1 = ex2_approx(fmaf(x[c + 1], p.scale_log2, nm));
        la[(c >> 1) & 3] += p0 + p1;
        pk[c >> 1] = pack_bf16x2(p0, p1);
      }
      l += (la[0] + la[1]) + (la[2] + la[3]);
      // P buffer sb was last read by P.V of tile j-2
      if (j >= 2) {
        ok = __all_sync(0xffffffffu, mbar_wait_bounded(&o_done[sb], ((j - 2) >> 1) & 1, abort_flag));
        if (!ok) break;
      }
      uint8_t* prow = pt + sb * C::PBYTES + r * 128;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int chunk = hf * 4 + q;
        *reinterpret_cast<uint4*>(prow + ((chunk ^ (r & 7)) << 4)) =
            make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
      }
      fence_proxy_async_smem();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[sb]);
    }
    if (!ok) {
      if (lane == 0 && !*abort_flag) record_error(p.err, kDevErrWaitFull);
      *abort_flag = 1;
    }
    // ---------------------------------------------------------- epilogue
    if (ok && work)
      ok = __all_sync(0xffffffffu, mbar_wait_bounded(&o_done[(nt - 1) & 1], ((nt - 1) >> 1) & 1, abort_flag));
    float o[D / 2];
    if (ok && work) {
      tc::fence_after();
      {
        uint32_t t[D / 2];
        ld_o<D>(trow + C::COL_O, t);
        tc::wait_ld();
#pragma unroll
        for (int c = 0; c < D / 2; ++c) o[c] = __uint_as_float(t[c]);
      }
    }
    const float lrow = l + __shfl_xor_sync(0xffffffffu, l, 16);
    const int col0 = hf * (D / 2);  // this thread's columns of O
    const bool direct = sa || (!CL && p.n_splits == 1 && !p.null_kv);
    if (ok && direct && work) {
      uint16_t* out = (sa ? p.osa : p.oca) + ((size_t)r * p.H + h) * D + col0;
      const float inv = 1.f / lrow;
#pragma unroll
      for (int c = 0; c < D / 2; c += 8) {
        uint4 w;
        w.x = pack_bf16x2(o[c] * inv, o[c + 1] * inv);
        w.y = pack_bf16x2(o[c + 2] * inv, o[c + 3] * inv);
        w.z = pack_bf16x2(o[c + 4] * inv, o[c + 5] * inv);
        w.w = pack_bf16x2(o[c + 6] * inv, o[c + 7] * inv);
        *reinterpret_cast<uint4*>(out + c) = w;
      }
    }
    if (ok && sa && p.nblk == 0 && (p.mode & 2)) {
      // no readable memory block: oca is the null row's value or zero
      uint16_t* out = p.oca + ((size_t)r * p.H + h) * D + col0;
      const uint16_t* vn =
          p.null_kv ? p.null_kv + ((size_t)p.layer * p.Hkv + h / (p.H / p.Hkv)) * 2 * D + D + col0 : nullptr;
#pragma unroll
      for (int c = 0; c < D / 2; c += 8)
        *reinterpret_cast<uint4*>(out + c) = vn ? *reinterpret_cast<const uint4*>(vn + c) : make_uint4(0, 0, 0, 0);
    }
    if constexpr (CL) {
      if (p.n_splits > 0) {
        // park this thread's half row of the CTA's partial in the (idle) K/V
        // ring for the cluster merge: rank 0 the null row (m = its score,
        // l = 1, O = its value row; m = -inf, l = 0, O = 0 without one), a
        // split its (m, l, O)
        float pm = -INFINITY, pl = 0.f, v[D / 2];
        if (sa) {
          const uint16_t* kn = p.null_kv
                                   ? p.null_kv + ((size_t)p.layer * p.Hkv + h / (p.H / p.Hkv)) * 2 * D
                                   : nullptr;
          if (kn) {
            float dot = null_dot<ROPE>(p, p.qc_ptr + (size_t)r * p.tok_c + (size_t)h * D, kn, col0, D / 2);
            dot += __shfl_xor_sync(0xffffffffu, dot, 16);
            pm = dot * p.scale_log2;
            pl = 1.f;
          }
#pragma unroll
          for (int c = 0; c < D / 2; ++c) v[c] = kn ? bf16lo(kn[D + col0 + c]) : 0.f;
        } else {
          const bool have = ok && work;
          pm = have ? m_used : -INFINITY;
          pl = have ? lrow : 0.f;
#pragma unroll
          for (int c = 0; c < D / 2; ++c) v[c] = have ? o[c] : 0.f;
        }
        float* pp = reinterpret_cast<float*>(ring) + (size_t)r * (D + 4);
#pragma unroll
        for (int c = 0; c < D / 2; c += 4)
          *reinterpret_cast<float4*>(pp + 4 + col0 + c) = make_float4(v[c], v[c + 1], v[c + 2], v[c + 3]);
        if (hf == 0) {
          pp[0] = pm;
          pp[1] = pl;
        }
      }
    }
    const bool part_ok = CL || SMEM_DCHECK(h < p.H && split < p.max_splits && p.n_splits <= p.max_splits, p.err);
    if (!CL && ok && !direct && part_ok) {
      float* pp = p.part + (((size_t)h * p.max_splits + split) * C::B + r) * (D + 4);
#pragma unroll
      for (int c = 0; c < D / 2; c += 4)
        *reinterpret_cast<float4*>(pp + 4 + col0 + c) = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
      if (hf == 0) {
        pp[0] = m_used;
        pp[1] = lrow;
      }
      __threadfence();
    }
    // the four softmax warps agree on the outcome before the ticket
    const bool all_ok = CL || bar_all(1, 128, ok);  // the ticket merge only
    if (!CL && all_ok && !direct && part_ok) {
      if (threadIdx.x == 0) *ticket = atomicAdd(&p.counters[h], 1u);
      named_bar_sync(1, 128);
      if (*ticket == (unsigned)(p.n_splits - 1)) {
        __threadfence();
        // merge all splits of this head for row r, columns col0.., in split order
        const size_t qoff = ((size_t)r * p.H + h) * D;
        const size_t qcoff = (size_t)r * p.tok_c + (size_t)h * D;
        float nscore = -INFINITY;
        if (p.null_kv) {
          const uint16_t* kn = p.null_kv + ((size_t)p.layer * p.Hkv + h / (p.H / p.Hkv)) * 2 * D;
          float dot = null_dot<ROPE>(p, p.qc_ptr + qcoff, kn, col0, D / 2);
          dot += __shfl_xor_sync(0xffffffffu, dot, 16);
          nscore = dot * p.scale_log2;
        }
        const float* pb = p.part + ((size_t)h * p.max_splits * C::B + r) * (D + 4);
        const size_t ps = (size_t)C::B * (D + 4);
        const int ns = p.n_splits;
        // every split's (m, l) in one batch of independent loads
        float ms[kPrefillMaxSplits], ls[kPrefillMaxSplits];
#pragma unroll
        for (int s2 = 0; s2 < kPrefillMaxSplits; ++s2) {
          const float2 v = s2 < ns ? __ldcg(reinterpret_cast<const float2*>(pb + s2 * ps)) : make_float2(-INFINITY, 0.f);
          ms[s2] = v.x;
          ls[s2] = v.y;
        }
        float M = nscore;
#pragma unroll
        for (int s2 = 0; s2 < kPrefillMaxSplits; ++s2) M = fmaxf(M, ms[s2]);
        float Lsum = 0.f, A[D / 2];
#pragma unroll
        for (int c = 0; c < D / 2; ++c) A[c] = 0.f;
        if (p.null_kv) {
          const float f = exp2f(nscore - M);
          Lsum = f;
          const uint16_t* vn = p.null_kv + ((size_t)p.layer * p.Hkv + h / (p.H / p.Hkv)) * 2 * D + D + col0;
#pragma unroll
          for (int c = 0; c < D / 2; ++c) A[c] = f * bf16lo(vn[c]);
        }
        // O rows of the splits come through the (now idle) K/V ring by bulk
        // copy, MERGE_SPR splits per round, and are summed in split order
        const float* head_part = p.part + (size_t)h * p.max_splits * C::B * (D + 4);
        for (int s0 = 0, round = 0; s0 < ns; s0 += C::MERGE_SPR, ++round) {
          const int cnt = min(C::MERGE_SPR, ns - s0);
          if (threadIdx.x == 0) {
            mbar_arrive_expect_tx(mbar_merge, (uint32_t)(cnt * C::PART_BYTES));
            for (int g2 = 0; g2 < cnt; ++g2)
              bulk_g2s(ring + g2 * C::PART_BYTES, head_part + (size_t)(s0 + g2) * C::B * (D + 4), C::PART_BYTES,
                       mbar_merge);
          }
          if (!bar_all(1, 128, mbar_wait_bounded(mbar_merge, round & 1, nullptr))) {
            if (threadIdx.x == 0) record_error(p.err, kDevErrWaitFull);
            break;  // uniform: every softmax thread saw the same outcome
          }
          for (int g2 = 0; g2 < cnt; ++g2) {
            float msg = 0.f, lsg = 0.f;
#pragma unroll
            for (int t2 = 0; t2 < kPrefillMaxSplits; ++t2)
              if (t2 == s0 + g2) { msg = ms[t2]; lsg = ls[t2]; }
            const float f = exp2f(msg - M);
            Lsum = fmaf(f, lsg, Lsum);
            const float4* row = reinterpret_cast<const float4*>(ring + g2 * C::PART_BYTES + r * (D + 4) * 4 + 16) +
                                col0 / 4;
#pragma unroll
            for (int c = 0; c < D / 8; ++c) {
              const float4 v = row[c];
              A[4 * c] = fmaf(f, v.x, A[4 * c]);
              A[4 * c + 1] = fmaf(f, v.y, A[4 * c + 1]);
              A[4 * c + 2] = fmaf(f, v.z, A[4 * c + 2]);
              A[4 * c + 3] = fmaf(f, v.w, A[4 * c + 3]);
            }
          }
          named_bar_sync(1, 128);  // the staging area is refilled next round
        }
        const float inv = 1.f / Lsum;
        uint16_t* out = p.oca + qoff + col0;
#pragma unroll
        for (int c = 0; c < D / 2; c += 8) {
          uint4 w;
          w.x = pack_bf16x2(A[c] * inv, A[c + 1] * inv);
          w.y = pack_bf16x2(A[c + 2] * inv, A[c + 3] * inv);
          w.z = pack_bf16x2(A[c + 4] * inv, A[c + 5] * inv);
          w.w = pack_bf16x2(A[c + 6] * inv, A[c + 7] * inv);
          *reinterpret_cast<uint4*>(out + c) = w;
        }
        if (threadIdx.x == 0) p.counters[h] = 0u;
      }
    }
  }
  if constexpr (CL) {
    if (p.n_splits > 0) {
      __syncwarp();
      tc::cluster_sync();  // every partial row of the cluster is parked
      cluster_merge<D>(p, h, crank, cs, smem_u32(ring), warp, lane);
      __syncwarp();
      tc::cluster_wait();  // no CTA leaves while another still reads its shared memory
    }
  }
  tc::fence_before();
  __syncthreads();
  if (warp == 4) {
    tc::fence_after();
    tc::dealloc(tmem, C::TMEM_COLS);
  }
}

template <int D, bool ROPE>
static cudaError_t launch_prefill_d(const PrefillParams& p, int grid, cudaStream_t st) {
  using C = Pf<D>;
  cudaError_t e = ensure_smem_limit<1000 + D + (ROPE ? 1 : 0)>(prefill_kernel<D, false, ROPE>, C::SMEM);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(C::THREADS);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  e = cudaLaunchKernelEx(&cfg, prefill_kernel<D, false, ROPE>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <bool ROPE>
static cudaError_t cluster_kernel_setup() {
  cudaError_t e = ensure_smem_limit<2064 + (ROPE ? 1 : 0)>(prefill_kernel<64, true, ROPE>, Pf<64>::SMEM);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(prefill_kernel<64, true, ROPE>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  return e;
}

template <bool ROPE>
static cudaError_t launch_prefill_cluster(const PrefillParams& p, cudaStream_t st) {
  cudaError_t e = cluster_kernel_setup<ROPE>();
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  const unsigned cs = (unsigned)p.n_splits + 1;
  cfg.gridDim = dim3((unsigned)p.H * cs);
  cfg.blockDim = dim3(Pf<64>::THREADS);
  cfg.dynamicSmemBytes = Pf<64>::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 2 : 1;
  e = cudaLaunchKernelEx(&cfg, prefill_kernel<64, true, ROPE>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// A kernel with the cluster prefill's launch footprint (threads and dynamic
// shared memory) but no tensor-memory allocation: the occupancy query counts
// one CTA per SM for kernels that allocate tensor memory at run time, while
// the hardware holds two of these (256 of 512 TMEM columns each; registers
// and shared memory both allow two).
__global__ void __launch_bounds__(192, 2) prefill_footprint_kernel(int* p) {
  extern __shared__ uint8_t sm[];
  if (p) p[threadIdx.x] = sm[threadIdx.x];
}

int prefill_cluster_max(int H, int D) {
  // the largest cluster (at most 16 CTAs) of which one per head can be
  // resident at once on the current device; 0: cluster mode unavailable
  if (D != 64) return 0;
  if (cluster_kernel_setup<false>() != cudaSuccess || cluster_kernel_setup<true>() != cudaSuccess ||
      cudaFuncSetAttribute(prefill_footprint_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, Pf<64>::SMEM) !=
          cudaSuccess ||
      cudaFuncSetAttribute(prefill_footprint_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
          cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  for (int cs : {16, 12, 8, 4}) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(H * cs));
    cfg.blockDim = dim3(Pf<64>::THREADS);
    cfg.dynamicSmemBytes = Pf<64>::SMEM;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, prefill_footprint_kernel, &cfg) == cudaSuccess && n >= H) return cs;
    cudaGetLastError();
  }
  return 0;
}

static int encode_bhd(CUtensorMap* map, const void* ptr, int H, int D, int tok_stride) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return -1;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)kBlockTok};
  const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)tok_stride * 2};
  const cuuint32_t box[3] = {(cuuint32_t)(D < 64 ? D : 64), 1, (cuuint32_t)kBlockTok};
  const cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box,
                            estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            D < 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : (int)r;
}

cudaError_t launch_prefill(const PrefillArgs& a, cudaStream_t st) {
  static thread_local PrefillParams P;
  P.pool = *a.pool_map;
  const int Hkv = a.Hkv ? a.Hkv : a.H;
  const int tok_s = a.tok_s ? a.tok_s : a.H * a.D;
  const int tok_kv = a.tok_kv ? a.tok_kv : (a.tok_s ? a.tok_s : Hkv * a.D);
  const int tok_c = a.tok_c ? a.tok_c : a.H * a.D;
  const int mode = a.mode ? a.mode : 3;
  // a half that is not requested keeps a harmless map (its pointer is valid)
  const void* qs = (mode & 1) ? a.qs : a.qc;
  const void* ks = (mode & 1) ? a.ks : a.qc;
  const void* vs = (mode & 1) ? a.vs : a.qc;
  const void* qc = (mode & 2) ? a.qc : a.qs;
  const int ts = (mode & 1) ? tok_s : tok_c, tc2 = (mode & 2) ? tok_c : tok_s;
  const int tkv = (mode & 1) ? tok_kv : tok_c, hkv = (mode & 1) ? Hkv : a.H;
  if (encode_bhd(&P.qs, qs, a.H, a.D, ts) || encode_bhd(&P.ks, ks, hkv, a.D, tkv) ||
      encode_bhd(&P.vs, vs, hkv, a.D, tkv) || encode_bhd(&P.qc, qc, a.H, a.D, tc2))
    return cudaErrorInvalidValue;
  P.Hkv = Hkv;
  P.mode = mode;
  P.tok_c = tok_c;
  P.table_row = a.table_row;
  P.null_kv = a.null_kv;
  P.qc_ptr = a.qc;
  P.osa = a.osa;
  P.oca = a.oca;
  P.part = a.part;
  P.counters = a.counters;
  P.err = a.err;
  P.L = a.L;
  P.H = a.H;
  P.layer = a.layer;
  P.nblk = a.nblk;
  P.split_blks = a.split_blks;
  P.n_splits = (mode & 2) ? a.n_splits : 0;
  P.capacity = a.capacity;
  P.max_blocks = a.max_blocks;
  P.max_splits = kPrefillMaxSplits;
  P.scale_log2 = a.scale_log2;
  P.n_sa = ((mode & 1) || ((mode & 2) && a.nblk == 0)) ? a.H : 0;
  const int grid = P.n_splits * a.H + P.n_sa;
  P.rope_tab = a.rope_tab;
  P.bidx_row = a.bidx_row;
  P.rope_w = a.rope_w;
  P.q_blk = a.q_blk;
  P.rope_half = a.D / 2;
  const bool rope = a.rope_tab != nullptr;
  if (a.D == 64 && a.cluster && P.n_splits > 0)
    return rope ? launch_prefill_cluster<true>(P, st) : launch_prefill_cluster<false>(P, st);
  if (a.D == 32) return rope ? launch_prefill_d<32, true>(P, grid, st) : launch_prefill_d<32, false>(P, grid, st);
  if (a.D == 64) return rope ? launch_prefill_d<64, true>(P, grid, st) : launch_prefill_d<64, false>(P, grid, st);
  if (a.D == 128) return rope ? launch_prefill_d<128, true>(P, grid, st) : launch_prefill_d<128, false>(P, grid, st);
  return cudaErrorInvalidValue;
}

}  // namespace smem
