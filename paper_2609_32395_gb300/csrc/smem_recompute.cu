// smem_recompute.cu -- cross-attention that reads the memory rows themselves
// instead of materialized per-layer keys and values (the "recompute K/V"
// regime of arXiv 2609.32395, Sec. 3.1 and App. "Serving": the cache keeps
// only the memory rows mu, d values per row shared by every reader layer,
// and each layer's keys mu W_kc and values mu W_vc are re-derived per step).
//
// The keys and values are linear in mu, so per head h (Sec. 2 "Model")
//   q_h . (mu_r W_kc,h) = (W_kc,h q_h) . mu_r = q'_h . mu_r
//   sum_r p_r (mu_r W_vc,h) = (sum_r p_r mu_r) W_vc,h
// and the layer's cross-attention is an attention of d-wide queries q'_h
// over the d-wide rows mu_r whose output O'_h = sum_r p_r mu_r is mapped by
// W_vc,h afterwards. The two small per-head maps run on the projection
// kernel (smem_gemm.cu) before and after this one; this kernel streams every row once per layer (2d
// bytes per row, half the materialized 4 H d_h) and keeps all queries that
// share a row set in one CTA:
//   S^T [64 rows][NQ queries] = mu_tile Q'^T   (K = d)
//   O'^T [d][NQ]             += mu_tile^T P^T  (M = 128 per column pair, K = 64)
// both on the tensor cores (tcgen05, fp32 accumulators in TMEM); the scores
// are issued as M = 128 MMAs over chunk pairs (see the kernel). A decode step
// puts up to NQ heads of one sequence in one CTA (NQ = H rounded up to 16,
// or tiles of heads when the accumulators would not fit); a one-block
// prefill puts NQ of the block's 64 queries of one head in a CTA. The row
// tile is streamed twice -- once into a score ring for S,
// once into a value ring for P.V (the second pass normally hits L2) -- so
// any d fits in shared memory; the two rings are separate so that value
// chunks waiting for their tile's softmax never hold up the score stream
// from HBM. Softmax runs column-wise (one query per column) with the same
// conditional rescale as the prefill kernel (raise the running maximum only
// when it grows by more than 2^8). Every unit (a split of a row set) writes
// its partial (m, l, O'); a second kernel, one CTA per (group, 128 columns),
// merges the splits in split order, null row first (the null row nu is just
// one more d-wide row). Reduction orders depend only on the block count, so
// outputs are bitwise independent of the edit path. An opt-in decode variant
// (mu_slice_kernel) splits d across a cluster and reads each tile once.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "smem_device.cuh"
#include "smem_internal.h"
#include "smem_tc.cuh"

namespace smem {

namespace {

constexpr int kMuBox = 64 * 128;        // one [64 rows][64 columns] bf16 box
constexpr int kMuThreads = 192;         // 4 softmax warps, producer, MMA
constexpr float kMuRescaleLog2 = 8.0f;  // raise the running max when it grows by more than 2^8

template <int NQ>
struct MuCfg {
  static constexpr int C2 = NQ / 2;                 // S columns per thread
  static constexpr int PBYTES = NQ * 128;           // P tile [NQ][64 rows] bf16
  static constexpr uint32_t ID_S = tc::idesc_bf16(64, NQ, 0, 0);
  static constexpr uint32_t ID_S2 = tc::idesc_bf16(128, 2 * NQ, 0, 0);  // chunk-pair scores
  static constexpr uint32_t ID_PV = tc::idesc_bf16(128, NQ, 1, 0);
};

template <int NQ>
__device__ __forceinline__ void ld_s(uint32_t taddr, uint32_t (&r)[NQ / 2]) {
  if constexpr (NQ == 64) tc::ld_16x32bx2_x32<32>(taddr, r);
  else if constexpr (NQ == 32) tc::ld_16x32bx2_x16<16>(taddr, r);
  else tc::ld_16x32bx2_x8<8>(taddr, r);
}

__device__ __forceinline__ void store_bf16(uint16_t* p, float v) {
  __nv_bfloat16 h = __float2bfloat16_rn(v);
  *reinterpret_cast<__nv_bfloat16*>(p) = h;
}

}  // namespace

template <int NQ>
__global__ void __launch_bounds__(kMuThreads, 1) mu_attention_kernel(const __grid_constant__ MuParams p) {
  using C = MuCfg<NQ>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int d = p.d;
  const int NC = d / 64;   // 64-column chunks of a row (even)
  const int cpb = p.cpb;   // chunks per stage (2 or 4, dividing NC): one TMA box of 64 cpb rows
  const int SPT = NC / cpb;                      // stages per tile
  const uint32_t SB = (uint32_t)cpb * kMuBox;    // stage bytes
  const CUtensorMap* pool = cpb == 4 ? &p.pool4 : &p.pool2;
  const int nss = p.ns;    // score-ring stages
  const int nsv = p.nsv;   // value-ring stages
  uint8_t* qt = base;
  uint8_t* sring = base + p.off_ring;
  uint8_t* vring = base + p.off_v;
  uint8_t* pt = base + p.off_p;
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + p.off_bar);
  uint64_t* q_full = bars;
  uint64_t* full_s = bars + 1;
  uint64_t* empty_s = full_s + nss;
  uint64_t* full_v = empty_s + nss;
  uint64_t* empty_v = full_v + nsv;
  uint64_t* s_full = empty_v + nsv;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* o_done = p_full + 2;
  uint64_t* drain = o_done + 2;
  uint8_t* misc = base + p.off_misc;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 4);
  float* red = reinterpret_cast<float*>(misc + 16);  // [2][4][NQ] column maxima per warp
  float* alpha = red + 2 * 4 * NQ;                   // [2][NQ] rescale factors
  float* lsum = alpha + 2 * NQ;                      // [4][NQ] column sums per warp
  float* mfin = lsum + 4 * NQ;                       // [NQ]
  float* xs = mfin + NQ;                             // [2][64][NQ / 2] partial-score exchange

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // this CTA's unit: split `split` of group g
  int lo = 0, hi = p.n_groups - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.groups[mid].unit_begin <= (int)blockIdx.x) lo = mid;
    else hi = mid - 1;
  }
  const int g = lo;
  const MuGroup& G = p.groups[g];
  const int split = (int)blockIdx.x - G.unit_begin;
  const int b0 = split * G.split_blks;
  const int nt = G.nblk > 0 ? min(G.split_blks, G.nblk - b0) : 0;
  const int* trow = p.table + (size_t)G.seq * p.max_blocks;
  // Scores: one M = 128 MMA covers a chunk pair (c, c+1) -- A = the two
  // chunks' 128 rows, B = the queries' K-slices of both chunks (2 NQ rows) --
  // and its diagonal blocks D[0:64][0:NQ] and D[64:128][NQ:2NQ] accumulate the
  // even- and odd-chunk partial scores (the off-diagonal blocks are unused).
  // Half the MMA instructions of one M = 64 MMA per chunk; the instruction
  // rate, not the data, bounds these small shapes. NSB score buffers of
  // 2 NQ columns (two when tensor memory allows), then O'.
  const int NSB = p.nsb;
  uint32_t ncols = 32;
  while (ncols < (uint32_t)(NQ * (2 * NSB + NC / 2))) ncols <<= 1;
  const uint32_t colO = 2 * NSB * NQ;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < nss; ++s) {
      mbar_init(&full_s[s], 1);
      mbar_init(&empty_s[s], 1);
    }
    for (int s = 0; s < nsv; ++s) {
      mbar_init(&full_v[s], 1);
      mbar_init(&empty_v[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_free[b], 4);
      mbar_init(&p_full[b], 4);
      mbar_init(&o_done[b], 1);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 4 && nt > 0) tc::alloc(tslot, ncols);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = nt > 0 ? *tslot : 0u;
  const int total = nt * SPT;  // stages of the unit on each stream

  if (warp == 4) {
    // ------------------------------------------------------------ TMA producer
    // Two streams: the score pass (stage k of the unit -- cpb chunks of one
    // tile, one TMA box -- into score stage k % nss, from HBM) and the value
    // pass of the same stages (into value stage k % nsv, normally from L2).
    // A tile's value pass starts once all of its score stages are issued.
    // The thread polls both rings, so a value stage held until its tile's P
    // is ready never stalls the scores. Boxes of several chunks keep the
    // TMA instruction rate of one thread well below its limit.
    if (lane == 0 && nt > 0) {
      mbar_arrive_expect_tx(q_full, (uint32_t)(NC * C::PBYTES));
      for (int c = 0; c < NC; ++c) tc::tma_load_3d(qt + c * C::PBYTES, &p.q, c * 64, G.n0, G.qg, q_full);
      int kS = 0, kV = 0, slot_s = 0, slot_v = 0;
      bool ok = true;
      unsigned long long t_last = global_timer_ns();
      while (kS < total || kV < total) {
        bool prog = false;
        if (kS < total && (kS < nss || mbar_test_wait(&empty_s[kS % nss], ((kS / nss) - 1) & 1))) {
          const int j = kS % SPT, st = kS % nss;
          if (j == 0) {
            slot_s = trow[b0 + kS / SPT];
            if (slot_s < 0 || slot_s >= p.capacity) record_error(p.err, kDevErrBounds);
          }
          if (slot_s >= 0 && slot_s < p.capacity) {
            mbar_arrive_expect_tx(&full_s[st], SB);
            tc::tma_load_3d(sring + st * SB, pool, 0, j * cpb * kRows, slot_s, &full_s[st]);
          } else {
            mbar_arrive(&full_s[st]);
          }
          ++kS;
          prog = true;
        }
        if (kV < total && (kV / SPT + 1) * SPT <= kS &&
            (kV < nsv || mbar_test_wait(&empty_v[kV % nsv], ((kV / nsv) - 1) & 1))) {
          const int j = kV % SPT, st = kV % nsv;
          if (j == 0) slot_v = trow[b0 + kV / SPT];
          if (slot_v >= 0 && slot_v < p.capacity) {
            mbar_arrive_expect_tx(&full_v[st], SB);
            tc::tma_load_3d(vring + st * SB, pool, 0, j * cpb * kRows, slot_v, &full_v[st]);
          } else {
            mbar_arrive(&full_v[st]);
          }
          ++kV;
          prog = true;
        }
        if (prog) {
          t_last = global_timer_ns();
        } else if (*abort_flag || global_timer_ns() - t_last > kWaitLimitNs) {
          if (!*abort_flag) record_error(p.err, kDevErrWaitEmpty);
          *abort_flag = 1;
          ok = false;
          break;
        }
      }
      if (!ok) {
        // let every copy already issued land before the CTA can exit
        mbar_wait_bounded(q_full, 0, nullptr);
        for (int j = kS > nss ? kS - nss : 0; j < kS; ++j) mbar_wait_bounded(&full_s[j % nss], (j / nss) & 1, nullptr);
        for (int j = kV > nsv ? kV - nsv : 0; j < kV; ++j) mbar_wait_bounded(&full_v[j % nsv], (j / nsv) & 1, nullptr);
      }
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------- MMA issuer
    // Polls two queues: the P.V of the oldest tile whose P is ready (value
    // stage by stage, a column pair per MMA), and the next score stage
    // (landed, and for a tile's first stage its S buffer free). Neither
    // blocks the other. The whole warp runs the loop -- lane 0's poll results
    // are shared, control flow and descriptors stay warp-uniform -- and one
    // elected lane issues the MMAs and commits.
    if (nt > 0) {
      const bool leader = tc::elect_one();
      bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(q_full, 0, abort_flag));
      tc::fence_after();
      const uint32_t qa = smem_u32(qt);
      const uint32_t sa = smem_u32(sring);
      const uint32_t va = smem_u32(vring);
      int kS = 0, kV = 0, tP = 0;
      unsigned long long t_last = global_timer_ns();
      while (ok && tP < nt) {
        bool prog = false;
        if (tP < kS / SPT) {
          const int st = kV % nsv;
          bool go = lane == 0 && (kV % SPT != 0 || mbar_test_wait(&p_full[tP & 1], (tP >> 1) & 1)) &&
                    mbar_test_wait(&full_v[st], (kV / nsv) & 1);
          go = __shfl_sync(0xffffffffu, go, 0);
          if (go) {
            tc::fence_after();
            const uint32_t a0 = va + st * SB;
            const uint32_t b = smem_u32(pt + (tP & 1) * C::PBYTES);
            for (int q = 0; q < cpb / 2; ++q) {
              const int cp = (kV % SPT) * (cpb / 2) + q;  // column pair of the row
              uint64_t ad[4], bd[4];
#pragma unroll
              for (int kk = 0; kk < 4; ++kk) {
                ad[kk] = tc::sdesc_sw128(a0 + 2 * q * kMuBox + kk * 2048, kMuBox, 1024);
                bd[kk] = tc::sdesc_sw128(b + kk * 32, 16, 1024);
              }
              if (leader) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                  tc::mma_bf16(tmem + colO + cp * NQ, ad[kk], bd[kk], C::ID_PV, (tP > 0 || kk > 0));
              }
            }
            if (leader) {
              tc::commit(&empty_v[st]);
              if ((kV + 1) % SPT == 0) tc::commit(&o_done[tP & 1]);
            }
            __syncwarp();
            ++kV;
            if (kV % SPT == 0) ++tP;
            prog = true;
          }
        }
        if (kS < total) {
          const int t = kS / SPT, j = kS % SPT, sb = t % NSB, st = kS % nss;
          bool go = lane == 0 && (j > 0 || t < NSB || mbar_test_wait(&s_free[sb], ((t / NSB) - 1) & 1)) &&
                    mbar_test_wait(&full_s[st], (kS / nss) & 1);
          go = __shfl_sync(0xffffffffu, go, 0);
          if (go) {
            tc::fence_after();
            for (int q = 0; q < cpb / 2; ++q) {
              const int c = j * cpb + 2 * q;  // even chunk of the pair
              const uint32_t a = sa + st * SB + 2 * q * kMuBox, b = qa + c * C::PBYTES;
              uint64_t ad[4], bd[4];
#pragma unroll
              for (int kk = 0; kk < 4; ++kk) {
                ad[kk] = tc::sdesc_sw128(a + kk * 32, 16, 1024);
                bd[kk] = tc::sdesc_sw128(b + kk * 32, 16, 1024);
              }
              if (leader) {
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                  tc::mma_bf16(tmem + (uint32_t)(sb * 2 * NQ), ad[kk], bd[kk], C::ID_S2, (c | kk) > 0);
              }
            }
            if (leader) {
              tc::commit(&empty_s[st]);
              if (j == SPT - 1) tc::commit(&s_full[sb]);
            }
            __syncwarp();
            ++kS;
            prog = true;
          }
        }
        if (prog) {
          t_last = global_timer_ns();
        } else {
          const bool give_up = lane == 0 && (*abort_flag || global_timer_ns() - t_last > kWaitLimitNs);
          if (__shfl_sync(0xffffffffu, give_up, 0)) ok = false;
        }
      }
      if (!ok) {
        if (leader && !*abort_flag) record_error(p.err, kDevErrWaitMma);
        __syncwarp();
        *abort_flag = 1;
      }
      if (leader) {
        tc::commit(drain);
        mbar_wait_bounded(drain, 0, nullptr);
      }
      __syncwarp();
    }
  } else {
    // ---------------------------------------------------------- softmax warps
    // Thread = TMEM lane tid of the M = 128 score tile: warps 0-1 hold the
    // even-chunk partials of tile rows 0-63, warps 2-3 the odd-chunk ones.
    // Each thread finishes one column half (queries hc*NQ/2 ..) of its row:
    // it hands the other half of its partial to the thread of the same row
    // and the other partial, and sums even + odd (the same order for both).
    const int tid = threadIdx.x;     // 0..127: TMEM lane of S and of O'
    const int hr = warp & 1;         // row half: tile rows 32 hr .. 32 hr + 31
    const int hc = warp >> 1;        // 0: even partial, finishes queries [0, NQ/2); 1: odd, [NQ/2, NQ)
    const int r = 32 * hr + lane;    // tile row
    const int col0 = hc * C::C2;
    const uint32_t tlane = tmem + ((uint32_t)(32 * warp) << 16);
    float m_used[C::C2], lp[C::C2];
#pragma unroll
    for (int c = 0; c < C::C2; ++c) {
      m_used[c] = -INFINITY;
      lp[c] = 0.f;
    }
    // Every exit from this loop is decided through bar_all over the four
    // warps, so they take the same named barriers in the same order.
    bool ok = true;
    for (int t = 0; t < nt; ++t) {
      const int sb = t % NSB, pb = t & 1;
      ok = bar_all(3, 128, mbar_wait_bounded(&s_full[sb], (t / NSB) & 1, abort_flag));
      if (!ok) break;
      tc::fence_after();
      float x[C::C2];
      {
        uint32_t v[NQ / 16][16];
#pragma unroll
        for (int cb = 0; cb < NQ / 16; ++cb) tc::ld_32x32b_x16(tlane + sb * 2 * NQ + hc * NQ + cb * 16, v[cb]);
        tc::wait_ld();
        tc::fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_free[sb]);
        // v holds queries [0, NQ); lo = [0, NQ/2), hi = [NQ/2, NQ) (compile-time indices)
        float* xo = xs + ((size_t)hc * 64 + r) * C::C2;
#pragma unroll
        for (int c = 0; c < C::C2; ++c) {
          const float lo = __uint_as_float(v[c / 16][c % 16]);
          const float hi = __uint_as_float(v[(C::C2 + c) / 16][(C::C2 + c) % 16]);
          xo[c] = hc == 0 ? hi : lo;
        }
        named_bar_sync(1, 128);
        const float* xi = xs + ((size_t)(1 - hc) * 64 + r) * C::C2;
#pragma unroll
        for (int c = 0; c < C::C2; ++c) {
          const float lo = __uint_as_float(v[c / 16][c % 16]);
          const float hi = __uint_as_float(v[(C::C2 + c) / 16][(C::C2 + c) % 16]);
          x[c] = hc == 0 ? lo + xi[c] : xi[c] + hi;
        }
      }
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        float v = x[c];
#pragma unroll
        for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) red[(pb * 2 + hr) * NQ + col0 + c] = v;
      }
      named_bar_sync(1, 128);
      bool need_mine = false;
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        const int col = col0 + c;
        const float tmax = fmaxf(red[(pb * 2) * NQ + col], red[(pb * 2 + 1) * NQ + col]);
        float a_c = 1.f;
        if (tmax > m_used[c] + kMuRescaleLog2) {
          a_c = exp2f(m_used[c] - tmax);
          lp[c] *= a_c;
          m_used[c] = tmax;
          need_mine = true;
        }
        if (hr == 0 && lane == 0) alpha[pb * NQ + col] = a_c;
      }
      // any column of the tile raised its maximum (t > 0: O' holds earlier tiles)
      const bool any = !bar_all(2, 128, !need_mine);
      if (t > 0 && any) {
        ok = bar_all(3, 128, mbar_wait_bounded(&o_done[(t - 1) & 1], ((t - 1) >> 1) & 1, abort_flag));
        if (!ok) break;
        tc::fence_after();
        for (int cp = 0; cp < NC / 2; ++cp) {
#pragma unroll
          for (int cb = 0; cb < NQ / 16; ++cb) {
            uint32_t o[16];
            const uint32_t ta = tlane + colO + cp * NQ + cb * 16;
            tc::ld_32x32b_x16(ta, o);
            tc::wait_ld();
#pragma unroll
            for (int j = 0; j < 16; ++j) o[j] = __float_as_uint(__uint_as_float(o[j]) * alpha[pb * NQ + cb * 16 + j]);
            tc::st_32x32b_x16(ta, o);
          }
        }
        tc::wait_st();
      }
      // P buffer pb was last read by P.V of tile t-2
      if (t >= 2) {
        ok = bar_all(3, 128, mbar_wait_bounded(&o_done[pb], ((t - 2) >> 1) & 1, abort_flag));
        if (!ok) break;
      }
      uint8_t* pbuf = pt + pb * C::PBYTES;
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        const int col = col0 + c;
        const float pr = exp2f(x[c] - m_used[c]);
        lp[c] += pr;
        store_bf16(reinterpret_cast<uint16_t*>(pbuf + col * 128 + ((((r >> 3) ^ (col & 7)) & 7) << 4) + (r & 7) * 2),
                   pr);
      }
      fence_proxy_async_smem();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[pb]);
    }
    if (!ok) {
      if (lane == 0 && !*abort_flag) record_error(p.err, kDevErrWaitFull);
      *abort_flag = 1;
    }
    // ---------------------------------------------------------- epilogue
    const size_t part_stride = (size_t)d + 4;
    float* part_u = p.part + (size_t)blockIdx.x * NQ * part_stride;
    if (nt > 0) {
      if (ok) ok = bar_all(3, 128, mbar_wait_bounded(&o_done[(nt - 1) & 1], ((nt - 1) >> 1) & 1, abort_flag));
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        float v = lp[c];
#pragma unroll
        for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) {
          lsum[hr * NQ + col0 + c] = v;
          if (hr == 0) mfin[col0 + c] = m_used[c];
        }
      }
      const bool all_ok = bar_all(1, 128, ok);
      if (all_ok) {
        tc::fence_after();
        for (int cp = 0; cp < NC / 2; ++cp) {
#pragma unroll
          for (int cb = 0; cb < NQ / 16; ++cb) {
            uint32_t o[16];
            tc::ld_32x32b_x16(tlane + colO + cp * NQ + cb * 16, o);
            tc::wait_ld();
#pragma unroll
            for (int j = 0; j < 16; ++j)
              __stcg(part_u + (size_t)(cb * 16 + j) * part_stride + 4 + cp * 128 + tid, __uint_as_float(o[j]));
          }
        }
        if (tid < NQ) {
          part_u[(size_t)tid * part_stride] = mfin[tid];
          part_u[(size_t)tid * part_stride + 1] = lsum[tid] + lsum[NQ + tid];
        }
      }
    }
  }
  tc::fence_before();
  __syncthreads();
  if (warp == 4 && nt > 0) {
    tc::fence_after();
    tc::dealloc(tmem, ncols);
  }
}

// Decode form on a cluster of CL CTAs that cut the row width d into column
// slices of wsl = d / CL: CTA `rank` streams only its slice of every tile
// (64 rows x wsl), once, and keeps it in shared memory from its score MMA to
// its P.V MMA (no second pass). The tile's scores are the sum of the CL slice
// partials; every CTA sends its fp32 partial S^T [64][NQ] to every peer with
// st.async (completing on the peer's exchange barrier), sums the CL partials
// in rank order -- the same fp32 sum in every CTA -- and runs the identical
// softmax, so P, m and l agree bitwise across the cluster and each CTA
// accumulates its own slice of O'. The exchange is double-buffered by tile
// parity; a CTA sends tile t+2's partial only after it consumed every
// peer's tile t+1 partial, which each peer sent only after it finished
// reading tile t's partials, so a buffer is never overwritten while read.
template <int NQ>
__global__ void __launch_bounds__(kMuThreads, 1) mu_slice_kernel(const __grid_constant__ MuParams p) {
  using C = MuCfg<NQ>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int CL = p.cl;
  const int NCS = p.wsl / 64;  // 64-column chunks of a slice (even)
  const int nslot = p.ns;      // tile slots of the ring
  const uint32_t rank = tc::cluster_ctarank();
  const int unit = (int)blockIdx.x / CL;
  uint8_t* qt = base;
  uint8_t* ring = base + p.off_ring;
  uint8_t* pt = base + p.off_p;
  float* xb = reinterpret_cast<float*>(base + p.off_x);  // [2][CL][64 rows][NQ]
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + p.off_bar);
  uint64_t* q_full = bars;
  uint64_t* full = bars + 1;
  uint64_t* empty = full + nslot;
  uint64_t* s_full = empty + nslot;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* o_done = p_full + 2;
  uint64_t* x_full = o_done + 2;
  uint64_t* drain = x_full + 2;
  uint8_t* misc = base + p.off_misc;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 4);
  float* red = reinterpret_cast<float*>(misc + 16);  // [2][4][NQ] column maxima per warp
  float* alpha = red + 2 * 4 * NQ;                   // [2][NQ] rescale factors
  float* lsum = alpha + 2 * NQ;                      // [4][NQ] column sums per warp
  float* mfin = lsum + 4 * NQ;                       // [NQ]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int lo = 0, hi = p.n_groups - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.groups[mid].unit_begin <= unit) lo = mid;
    else hi = mid - 1;
  }
  const MuGroup& G = p.groups[lo];
  const int split = unit - G.unit_begin;
  const int b0 = split * G.split_blks;
  const int nt = G.nblk > 0 ? min(G.split_blks, G.nblk - b0) : 0;  // the same in every CTA of the cluster
  const int* trow = p.table + (size_t)G.seq * p.max_blocks;
  uint32_t ncols = 32;
  while (ncols < (uint32_t)(NQ * (2 + NCS / 2))) ncols <<= 1;
  const uint32_t colO = 2 * NQ;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < nslot; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_free[b], 4);
      mbar_init(&p_full[b], 4);
      mbar_init(&o_done[b], 1);
      mbar_init(&x_full[b], 1);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 4 && nt > 0) tc::alloc(tslot, ncols);
  tc::fence_before();
  tc::cluster_sync();  // every CTA's barriers exist before any peer signals them
  tc::fence_after();
  const uint32_t tmem = nt > 0 ? *tslot : 0u;

  if (warp == 4) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0 && nt > 0) {
      mbar_arrive_expect_tx(q_full, (uint32_t)(NCS * C::PBYTES));
      for (int c = 0; c < NCS; ++c)
        tc::tma_load_3d(qt + c * C::PBYTES, &p.q, (int)rank * p.wsl + c * 64, G.n0, G.qg, q_full);
      bool ok = true;
      int issued = 0;
      for (int t = 0; t < nt; ++t) {
        const int sl = t % nslot;
        if (t >= nslot && !mbar_wait_bounded(&empty[sl], ((t / nslot) - 1) & 1, abort_flag)) {
          if (!*abort_flag) record_error(p.err, kDevErrWaitEmpty);
          *abort_flag = 1;
          ok = false;
          break;
        }
        const int slot = trow[b0 + t];
        if (slot >= 0 && slot < p.capacity) {
          mbar_arrive_expect_tx(&full[sl], (uint32_t)(NCS * kMuBox));
          for (int c = 0; c < NCS; c += p.cpb)  // boxes of cpb chunks
            tc::tma_load_3d(ring + (sl * NCS + c) * kMuBox, p.cpb == 4 ? &p.pool4 : &p.pool2, 0,
                            ((int)rank * NCS + c) * kRows, slot, &full[sl]);
        } else {
          record_error(p.err, kDevErrBounds);
          mbar_arrive(&full[sl]);
        }
        ++issued;
      }
      if (!ok) {
        // let every copy already issued land before the CTA can exit
        mbar_wait_bounded(q_full, 0, nullptr);
        for (int j = issued > nslot ? issued - nslot : 0; j < issued; ++j)
          mbar_wait_bounded(&full[j % nslot], (j / nslot) & 1, nullptr);
      }
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0 && nt > 0) {
      bool ok = mbar_wait_bounded(q_full, 0, abort_flag);
      tc::fence_after();
      const uint32_t qa = smem_u32(qt);
      const uint32_t ra = smem_u32(ring);
      // P.V of tile t: O'^T[wsl][NQ] += slice^T P^T, one M = 128 MMA per column pair
      auto issue_pv = [&](int t) {
        const int pb = t & 1;
        if (ok) ok = mbar_wait_bounded(&p_full[pb], (t >> 1) & 1, abort_flag);
        if (!ok) return;
        tc::fence_after();
        const uint32_t b = smem_u32(pt + pb * C::PBYTES);
        const uint32_t a0 = ra + (uint32_t)((t % nslot) * NCS * kMuBox);
        for (int cp = 0; cp < NCS / 2; ++cp) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc::mma_bf16(tmem + colO + cp * NQ, tc::sdesc_sw128(a0 + 2 * cp * kMuBox + kk * 2048, kMuBox, 1024),
                         tc::sdesc_sw128(b + kk * 32, 16, 1024), C::ID_PV, (t > 0 || kk > 0));
        }
        tc::commit(&empty[t % nslot]);
        tc::commit(&o_done[pb]);
      };
      for (int t = 0; t < nt && ok; ++t) {
        const int sb = t & 1, sl = t % nslot;
        if (t >= 2) ok = mbar_wait_bounded(&s_free[sb], ((t >> 1) - 1) & 1, abort_flag);
        if (ok) ok = mbar_wait_bounded(&full[sl], (t / nslot) & 1, abort_flag);
        if (!ok) break;
        tc::fence_after();
        // partial S^T[64][NQ] of this slice: K = wsl
        const uint32_t a0 = ra + (uint32_t)(sl * NCS * kMuBox);
        for (int c = 0; c < NCS; ++c) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc::mma_bf16(tmem + sb * NQ, tc::sdesc_sw128(a0 + c * kMuBox + kk * 32, 16, 1024),
                         tc::sdesc_sw128(qa + c * C::PBYTES + kk * 32, 16, 1024), C::ID_S, (c | kk) > 0);
        }
        tc::commit(&s_full[sb]);
        if (t > 0) issue_pv(t - 1);
      }
      if (ok) issue_pv(nt - 1);
      if (!ok) {
        if (!*abort_flag) record_error(p.err, kDevErrWaitMma);
        *abort_flag = 1;
      }
      tc::commit(drain);
      mbar_wait_bounded(drain, 0, nullptr);
    }
  } else {
    // ---------------------------------------------------------- softmax warps
    const int tid = threadIdx.x;            // 0..127: TMEM lane of O'
    const int r = 16 * warp + (lane & 15);  // row of the tile
    const int hf = lane >> 4;               // column half of S
    const int col0 = hf * C::C2;
    const uint32_t tlane = tmem + ((uint32_t)(32 * warp) << 16);
    const uint32_t xbytes = (uint32_t)((CL - 1) * 64 * NQ * 4);
    float m_used[C::C2], lp[C::C2];
#pragma unroll
    for (int c = 0; c < C::C2; ++c) {
      m_used[c] = -INFINITY;
      lp[c] = 0.f;
    }
    bool ok = true;
    for (int t = 0; t < nt; ++t) {
      const int sb = t & 1;
      ok = bar_all(3, 128, mbar_wait_bounded(&s_full[sb], (t >> 1) & 1, abort_flag));
      if (!ok) break;
      tc::fence_after();
      uint32_t sr[C::C2];
      ld_s<NQ>(tlane + sb * NQ, sr);
      tc::wait_ld();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[sb]);
      float x[C::C2];
      if (CL > 1) {
        if (tid == 0) mbar_arrive_expect_tx(&x_full[sb], xbytes);
        const uint32_t mine = smem_u32(xb + ((size_t)(sb * CL + (int)rank) * 64 + r) * NQ + col0);
        const uint32_t xbar = smem_u32(&x_full[sb]);
        for (int k = 1; k < CL; ++k) {
          const uint32_t peer = (rank + (uint32_t)k) % (uint32_t)CL;
          const uint32_t dst = tc::dsmem_addr(mine, peer);
          const uint32_t pbar = tc::dsmem_addr(xbar, peer);
#pragma unroll
          for (int c = 0; c < C::C2; c += 4) tc::st_async_v4(dst + c * 4, sr[c], sr[c + 1], sr[c + 2], sr[c + 3], pbar);
        }
        ok = bar_all(3, 128, mbar_wait_bounded(&x_full[sb], (t >> 1) & 1, abort_flag));
        if (!ok) break;
        // the CL slice partials summed in rank order (identical in every CTA)
        const float* xr = xb + ((size_t)(sb * CL) * 64 + r) * NQ + col0;
#pragma unroll
        for (int c = 0; c < C::C2; c += 4) {
          float4 acc = rank == 0 ? make_float4(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1]),
                                               __uint_as_float(sr[c + 2]), __uint_as_float(sr[c + 3]))
                                 : *reinterpret_cast<const float4*>(xr + c);
          for (int k = 1; k < CL; ++k) {
            const float4 v = k == (int)rank ? make_float4(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1]),
                                                          __uint_as_float(sr[c + 2]), __uint_as_float(sr[c + 3]))
                                            : *reinterpret_cast<const float4*>(xr + (size_t)k * 64 * NQ + c);
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
          }
          x[c] = acc.x;
          x[c + 1] = acc.y;
          x[c + 2] = acc.z;
          x[c + 3] = acc.w;
        }
      } else {
#pragma unroll
        for (int c = 0; c < C::C2; ++c) x[c] = __uint_as_float(sr[c]);
      }
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        float v = x[c];
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 4));
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 8));
        if ((lane & 15) == 0) red[(sb * 4 + warp) * NQ + col0 + c] = v;
      }
      named_bar_sync(1, 128);
      bool need_mine = false;
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        const int col = col0 + c;
        float tmax = red[(sb * 4) * NQ + col];
#pragma unroll
        for (int w2 = 1; w2 < 4; ++w2) tmax = fmaxf(tmax, red[(sb * 4 + w2) * NQ + col]);
        float a_c = 1.f;
        if (tmax > m_used[c] + kMuRescaleLog2) {
          a_c = exp2f(m_used[c] - tmax);
          lp[c] *= a_c;
          m_used[c] = tmax;
          need_mine = true;
        }
        if (warp == 0 && (lane & 15) == 0) alpha[sb * NQ + col] = a_c;
      }
      const bool any = !bar_all(2, 128, !need_mine);
      if (t > 0 && any) {
        ok = bar_all(3, 128, mbar_wait_bounded(&o_done[(t - 1) & 1], ((t - 1) >> 1) & 1, abort_flag));
        if (!ok) break;
        tc::fence_after();
        for (int cp = 0; cp < NCS / 2; ++cp) {
#pragma unroll
          for (int cb = 0; cb < NQ / 16; ++cb) {
            uint32_t o[16];
            const uint32_t ta = tlane + colO + cp * NQ + cb * 16;
            tc::ld_32x32b_x16(ta, o);
            tc::wait_ld();
#pragma unroll
            for (int j = 0; j < 16; ++j) o[j] = __float_as_uint(__uint_as_float(o[j]) * alpha[sb * NQ + cb * 16 + j]);
            tc::st_32x32b_x16(ta, o);
          }
        }
        tc::wait_st();
      }
      if (t >= 2) {  // P buffer sb was last read by P.V of tile t-2
        ok = bar_all(3, 128, mbar_wait_bounded(&o_done[sb], ((t - 2) >> 1) & 1, abort_flag));
        if (!ok) break;
      }
      uint8_t* pb = pt + sb * C::PBYTES;
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        const int col = col0 + c;
        const float pr = exp2f(x[c] - m_used[c]);
        lp[c] += pr;
        store_bf16(reinterpret_cast<uint16_t*>(pb + col * 128 + ((((r >> 3) ^ (col & 7)) & 7) << 4) + (r & 7) * 2),
                   pr);
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
    const size_t part_stride = (size_t)p.d + 4;
    float* part_u = p.part + (size_t)unit * NQ * part_stride;
    if (nt > 0) {
      if (ok) ok = bar_all(3, 128, mbar_wait_bounded(&o_done[(nt - 1) & 1], ((nt - 1) >> 1) & 1, abort_flag));
#pragma unroll
      for (int c = 0; c < C::C2; ++c) {
        float v = lp[c];
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 2);
        v += __shfl_xor_sync(0xffffffffu, v, 4);
        v += __shfl_xor_sync(0xffffffffu, v, 8);
        if ((lane & 15) == 0) {
          lsum[warp * NQ + col0 + c] = v;
          if (warp == 0) mfin[col0 + c] = m_used[c];
        }
      }
      const bool all_ok = bar_all(1, 128, ok);
      if (all_ok) {
        tc::fence_after();
        for (int cp = 0; cp < NCS / 2; ++cp) {
#pragma unroll
          for (int cb = 0; cb < NQ / 16; ++cb) {
            uint32_t o[16];
            tc::ld_32x32b_x16(tlane + colO + cp * NQ + cb * 16, o);
            tc::wait_ld();
#pragma unroll
            for (int j = 0; j < 16; ++j)
              __stcg(part_u + (size_t)(cb * 16 + j) * part_stride + 4 + (int)rank * p.wsl + cp * 128 + tid,
                     __uint_as_float(o[j]));
          }
        }
        if (rank == 0 && tid < NQ) {
          part_u[(size_t)tid * part_stride] = mfin[tid];
          part_u[(size_t)tid * part_stride + 1] = lsum[tid] + lsum[NQ + tid] + lsum[2 * NQ + tid] + lsum[3 * NQ + tid];
        }
      }
    }
  }
  tc::fence_before();
  __syncthreads();
  if (warp == 4 && nt > 0) {
    tc::fence_after();
    tc::dealloc(tmem, ncols);
  }
  tc::cluster_sync();  // no CTA leaves while a peer may still write into its shared memory
}

// Merge of the split partials of every group: CTA (column block, group),
// thread = one of 128 columns of O'. Splits in split order, null row first.
template <int NQ>
__global__ void __launch_bounds__(128) mu_merge_kernel(const __grid_constant__ MuParams p) {
  __shared__ float snull[4][NQ];
  __shared__ float wsc[kMuMaxSplits + 1][NQ];  // split weights, then the null row's
  const int g = blockIdx.y;
  const MuGroup& G = p.groups[g];
  const int d = p.d;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int dc = blockIdx.x * 128 + tid;
  const int nq_out = min(NQ, p.nrows - G.n0);
  const size_t ps = (size_t)d + 4;
  uint16_t* out = p.out + ((size_t)G.qg * p.nrows + G.n0) * d;
  const float nuv = p.nu ? bf16lo(p.nu[dc]) : 0.f;
  if (G.nblk == 0) {  // no readable memory block: the null row's value or zero
    for (int n = 0; n < nq_out; ++n) out[(size_t)n * d + dc] = p.nu ? p.nu[dc] : (uint16_t)0;
    return;
  }
  // null scores q'_n . nu (q' carries the softmax scale)
  if (p.nu) {
    for (int n = 0; n < NQ; ++n) {
      float dot = 0.f;
      if (n < nq_out) {
        const uint16_t* qrow = p.qptr + ((size_t)G.qg * p.nrows + G.n0 + n) * d;
        for (int c = tid; c < d; c += 128) dot = fmaf(bf16lo(qrow[c]), bf16lo(p.nu[c]), dot);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
      if (lane == 0) snull[warp][n] = dot;
    }
  }
  __syncthreads();
  const int nsp = G.nsplit;
  const float* part_g = p.part + (size_t)G.unit_begin * NQ * ps;
  if (tid < NQ) {
    const int n = tid;
    const float sn = p.nu ? snull[0][n] + snull[1][n] + snull[2][n] + snull[3][n] : -INFINITY;
    float ms[kMuMaxSplits], ls[kMuMaxSplits];
#pragma unroll
    for (int s2 = 0; s2 < kMuMaxSplits; ++s2) {
      const float2 v = s2 < nsp ? __ldcg(reinterpret_cast<const float2*>(part_g + ((size_t)s2 * NQ + n) * ps))
                                : make_float2(-INFINITY, 0.f);
      ms[s2] = v.x;
      ls[s2] = v.y;
    }
    float M = sn;
#pragma unroll
    for (int s2 = 0; s2 < kMuMaxSplits; ++s2) M = fmaxf(M, ms[s2]);
    float L = p.nu ? exp2f(sn - M) : 0.f;
    float f[kMuMaxSplits];
#pragma unroll
    for (int s2 = 0; s2 < kMuMaxSplits; ++s2) {
      f[s2] = s2 < nsp ? exp2f(ms[s2] - M) : 0.f;
      L = fmaf(f[s2], ls[s2], L);
    }
    const float inv = 1.f / L;
#pragma unroll
    for (int s2 = 0; s2 < kMuMaxSplits; ++s2) wsc[s2][n] = f[s2] * inv;
    wsc[kMuMaxSplits][n] = p.nu ? exp2f(sn - M) * inv : 0.f;
  }
  __syncthreads();
  for (int n = 0; n < nq_out; ++n) {
    float v[kMuMaxSplits];
#pragma unroll
    for (int s2 = 0; s2 < kMuMaxSplits; ++s2)
      v[s2] = s2 < nsp ? __ldcg(part_g + ((size_t)s2 * NQ + n) * ps + 4 + dc) : 0.f;
    float acc = wsc[kMuMaxSplits][n] * nuv;
#pragma unroll
    for (int s2 = 0; s2 < kMuMaxSplits; ++s2)
      if (s2 < nsp) acc = fmaf(wsc[s2][n], v[s2], acc);
    store_bf16(out + (size_t)n * d + dc, acc);
  }
}

namespace {

int encode3d(CUtensorMap* map, const void* ptr, uint64_t d0, uint64_t d1, uint64_t d2, uint32_t b1) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return -1;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {d0 * 2, d0 * d1 * 2};
  const cuuint32_t box[3] = {64, b1, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, estr,
                            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : (int)r;
}

// Shared-memory plan of a launch (one CTA per SM): Q' chunks, the score
// ring, the value ring, two P tiles, barriers, scratch. Stages of four
// chunks (one 32 KB box) where d allows and at least two score and two
// value stages fit, else of two; about a third of the stages go to the
// value ring. Returns the dynamic shared-memory bytes, -1 if no plan fits.
int mu_smem_plan(MuParams& P, int nq, int d) {
  const int nc = d / 64;
  const int qbytes = nc * nq * 128;
  const int pbytes = 2 * nq * 128;
  P.off_ring = (qbytes + 1023) / 1024 * 1024;
  // misc: 16 B words + red[2][4][NQ] + alpha[2][NQ] + lsum[4][NQ] + mfin[NQ] + exchange [64][NQ]
  const int misc = 16 + (8 + 2 + 4 + 1 + 64) * nq * 4;
  const int chunks = (kMuSmemBudget - P.off_ring - pbytes - misc - 1024) / kMuBox;
  P.cpb = 0;
  for (int cpb : {4, 2}) {
    if (nc % cpb) continue;
    const int stages = chunks / cpb;
    const int nsv = stages / 3 > 2 ? stages / 3 : 2;
    int nss = stages - nsv;
    if (nss > 16) nss = 16;
    if (nss < 2) continue;
    P.cpb = cpb;
    P.ns = nss;
    P.nsv = nsv;
    break;
  }
  if (!P.cpb) return -1;
  // two score buffers (2 NQ columns each) when tensor memory holds them next to O'
  P.nsb = nq * (4 + nc / 2) <= 512 ? 2 : 1;
  const int sb = P.cpb * kMuBox;
  P.off_v = P.off_ring + P.ns * sb;
  P.off_p = P.off_v + P.nsv * sb;
  P.off_bar = P.off_p + pbytes;
  const int nbars = 1 + 2 * P.ns + 2 * P.nsv + 9;  // q_full, two full/empty rings, s_full/s_free/p_full/o_done pairs, drain
  P.off_misc = (P.off_bar + nbars * 8 + 15) / 16 * 16;
  return P.off_misc + misc + 1024;
}

template <int NQ>
cudaError_t launch_mu_nq(const MuParams& P, int smem, cudaStream_t st) {
  cudaError_t e = ensure_smem_limit<3000 + NQ>(mu_attention_kernel<NQ>, kMuSmemBudget + 2048);
  if (e != cudaSuccess) return e;
  mu_attention_kernel<NQ><<<P.n_units, kMuThreads, smem, st>>>(P);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  mu_merge_kernel<NQ><<<dim3((unsigned)(P.d / 128), (unsigned)P.n_groups), 128, 0, st>>>(P);
  return cudaGetLastError();
}

}  // namespace

// Shared-memory plan of the column-slice kernel: Q' slice, tile slots,
// two P tiles, the exchange buffers, barriers, scratch. -1 if fewer than
// three tile slots fit.
int mu_slice_plan(MuParams& P, int nq, int wsl, int cl) {
  const int ncs = wsl / 64;
  const int qbytes = ncs * nq * 128;
  const int pbytes = 2 * nq * 128;
  const int xbytes = 2 * cl * 64 * nq * 4;
  const int tile = ncs * kMuBox;
  P.off_ring = (qbytes + 1023) / 1024 * 1024;
  int nslot = (kMuSmemBudget - P.off_ring - pbytes - xbytes - 4096) / tile;
  if (nslot > 8) nslot = 8;
  if (nslot < 3) return -1;
  P.ns = nslot;
  P.nsv = 0;
  P.cpb = ncs % 4 == 0 && (cl * wsl / 64) % 4 == 0 ? 4 : 2;
  P.cl = cl;
  P.wsl = wsl;
  P.off_p = P.off_ring + nslot * tile;
  P.off_x = P.off_p + pbytes;
  P.off_bar = P.off_x + xbytes;
  const int nbars = 1 + 2 * nslot + 11;  // q_full, full/empty, s_full/s_free/p_full/o_done/x_full pairs, drain
  P.off_misc = (P.off_bar + nbars * 8 + 15) / 16 * 16;
  const int misc = 16 + (8 + 2 + 4 + 1) * nq * 4;
  return P.off_misc + misc + 1024;
}

template <int NQ>
cudaError_t launch_slice_nq(const MuParams& P, int smem, cudaStream_t st) {
  cudaError_t e = ensure_smem_limit<3100 + NQ>(mu_slice_kernel<NQ>, kMuSmemBudget + 2048);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[1];
  cfg.gridDim = dim3((unsigned)(P.n_units * P.cl));
  cfg.blockDim = dim3(kMuThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)P.cl;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, mu_slice_kernel<NQ>, P);
  if (e != cudaSuccess) return e;
  mu_merge_kernel<NQ><<<dim3((unsigned)(P.d / 128), (unsigned)P.n_groups), 128, 0, st>>>(P);
  return cudaGetLastError();
}

// Clusters of the column-slice kernel resident at once on the current
// device (0: the configuration cannot run).
template <int NQ>
int slice_clusters(int cl, int smem) {
  if (ensure_smem_limit<3100 + NQ>(mu_slice_kernel<NQ>, kMuSmemBudget + 2048) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[1];
  cfg.gridDim = dim3((unsigned)(cl * 64));
  cfg.blockDim = dim3(kMuThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cl;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, mu_slice_kernel<NQ>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

int mu_query_tile(int nq_total, int d) {
  // the widest query tile whose accumulators fit TMEM: NQ (2 + d/128) <= 512
  for (int nq : {64, 32, 16}) {
    if (nq * (2 + d / 128) > 512) continue;
    if (nq <= 16 || nq_total > nq / 2) return nq;
  }
  return 0;
}

int mu_prefill_query_tile(int nblk, int H, int d) {
  // the widest tile (fewest re-reads of the rows from L2) whose two score
  // buffers fit tensor memory next to O' and that still gives every SM a
  // unit; the narrowest otherwise. (A single score buffer serializes each
  // tile's score MMAs behind the previous tile's softmax: at d = 768, tiles
  // of 32 queries serve 64 / 256 blocks 22% / 15% faster than tiles of 64.)
  for (int nq : {64, 32}) {
    if (nq * (4 + d / 128) > 512) continue;
    const int groups = H * (kBlockTok / nq);
    const int sb = mu_prefill_split_blocks(nblk, groups);
    if (groups * ((nblk + sb - 1) / sb) >= 152) return nq;
  }
  return 16;
}

int encode_mu_pool_map(CUtensorMap* map, void* pool, int d, int capacity, int chunks_per_box) {
  // a slot is [d/64 chunks][R][64]: chunk c of a block is rows c*R .. c*R+R-1
  // of the view, and a box of chunks_per_box consecutive chunks is one copy
  return encode3d(map, pool, 64, (uint64_t)kRows * (d / 64), (uint64_t)capacity, (uint32_t)(kRows * chunks_per_box));
}

MuDecodePlan mu_decode_plan(int H, int d) {
  const MuDecodePlan two_pass{mu_query_tile(H, d), 0, 0};
  const int nq = (H + 15) / 16 * 16;
  if (nq > 64) return two_pass;
  // slices of 256 columns where d allows, clusters of at most 8 CTAs, an
  // exchange of at most 2 x 64 KB-equivalent partials (cl x nq <= 128)
  for (int wsl : {256, 128, 384, 512}) {
    if (d % wsl) continue;
    const int cl = d / wsl;
    if (cl > 8 || cl * nq > 128) continue;
    MuParams P{};
    const int smem = mu_slice_plan(P, nq, wsl, cl);
    if (smem < 0) continue;
    const int n = nq == 16 ? slice_clusters<16>(cl, smem) : nq == 32 ? slice_clusters<32>(cl, smem)
                                                                      : slice_clusters<64>(cl, smem);
    if (n > 0) return MuDecodePlan{nq, cl, wsl};
  }
  return two_pass;
}

cudaError_t launch_mu_slice(MuParams& P, const MuDecodePlan& pl, cudaStream_t st) {
  if (P.n_units == 0) return cudaSuccess;
  if (pl.cl < 1 || P.d != pl.cl * pl.wsl) return cudaErrorInvalidValue;
  if (encode3d(&P.q, P.qptr, (uint64_t)P.d, (uint64_t)P.nrows, (uint64_t)P.n_qg, (uint32_t)pl.nq))
    return cudaErrorInvalidValue;
  const int smem = mu_slice_plan(P, pl.nq, pl.wsl, pl.cl);
  if (smem < 0 || smem > kMuSmemBudget + 2048) return cudaErrorInvalidValue;
  if (pl.nq == 16) return launch_slice_nq<16>(P, smem, st);
  if (pl.nq == 32) return launch_slice_nq<32>(P, smem, st);
  if (pl.nq == 64) return launch_slice_nq<64>(P, smem, st);
  return cudaErrorInvalidValue;
}

cudaError_t launch_mu_attention(MuParams& P, int nq, cudaStream_t st) {
  if (P.n_units == 0) return cudaSuccess;
  P.cl = 0;
  P.wsl = 0;
  if (encode3d(&P.q, P.qptr, (uint64_t)P.d, (uint64_t)P.nrows, (uint64_t)P.n_qg, (uint32_t)nq)) return cudaErrorInvalidValue;
  const int smem = mu_smem_plan(P, nq, P.d);
  if (smem < 0 || smem > kMuSmemBudget + 2048) return cudaErrorInvalidValue;
  if (nq == 64) return launch_mu_nq<64>(P, smem, st);
  if (nq == 32) return launch_mu_nq<32>(P, smem, st);
  if (nq == 16) return launch_mu_nq<16>(P, smem, st);
  return cudaErrorInvalidValue;
}

}  // namespace smem
