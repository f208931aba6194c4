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
// count -- or (item, head) for SA. Units are dealt round-robin to persistent
// CTAs. Each CTA has one producer warp that streams the units' K/V tiles
// (one memory block = R rows of K and of V for one head, 2 x 8 KB at
// d_h = 64) from the paged pool into a ring of shared-memory stages with bulk
// TMA copies completing on mbarriers, and four consumer warps that each own a
// quarter of every tile's rows: 16-byte shared loads, fp32 dot products
// reduced across the lanes of a row, warp-level online softmax in base 2,
// fp32 accumulation of P.V. At the end of a unit the four warps merge in warp
// order; a CA unit writes its split partial (m, l, acc[d_h]) and the CTA
// that completes the last split of an (item, head) merges all splits in split
// order (null row first) and writes bf16 oca. No CTA ever waits for another.
// Every reduction order is fixed by the block count, so the same block set
// gives the same bits whatever the slots or the edit history.
#include <cuda_runtime.h>

#include <cmath>

#include "smem_device.cuh"
#include "smem_internal.h"

namespace smem {

template <int D>
struct DecCfg {
  static constexpr int R = kRows;
  static constexpr int TILE_BYTES = R * D * 2;  // K or V of one block and head
  static constexpr int STAGE_BYTES = 2 * TILE_BYTES;
  static constexpr int NSTAGE = D == 64 ? 6 : 3;
  static constexpr int NCW = 4;                     // consumer warps
  static constexpr int THREADS = (NCW + 1) * 32;    // + one producer warp
  static constexpr int LPR = D / 8;                 // lanes per row (16 B each)
  static constexpr int RPI = 32 / LPR;              // rows per warp load
  static constexpr int ROWS_PER_WARP = R / NCW;
  static constexpr int ITERS = ROWS_PER_WARP / RPI;
  static constexpr int OFF_BARS = NSTAGE * STAGE_BYTES;
  static constexpr int OFF_COMB = OFF_BARS + 2 * NSTAGE * 8;
  static constexpr int OFF_MISC = OFF_COMB + NCW * (D + 2) * 4;
  static constexpr int SMEM = OFF_MISC + 64;
};

struct Unit {
  int sa;     // 1: self-attention unit
  int item;
  int h;
  int split;  // CA only
  int b0;     // first table position (CA)
  int nt;     // tiles
};

__device__ __forceinline__ Unit unit_of(const DecodeParams& p, int u) {
  Unit U;
  const int nca = p.n_pairs * p.H;
  if (u < nca) {
    const int pair = u / p.H;
    U.sa = 0;
    U.h = u - pair * p.H;
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
    U.nt = 1;
  }
  return U;
}

__device__ __forceinline__ bool bar_any(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.or.pred po, %2, %3, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

template <int D>
__global__ void __launch_bounds__(DecCfg<D>::THREADS, 2)
    decode_kernel(const __grid_constant__ DecodeParams p) {
  using C = DecCfg<D>;
  extern __shared__ __align__(128) uint8_t smem_raw[];
  uint8_t* stages = smem_raw;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem_raw + C::OFF_BARS);
  uint64_t* empty = full + C::NSTAGE;
  float* comb = reinterpret_cast<float*>(smem_raw + C::OFF_COMB);  // [NCW][D+2]
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem_raw + C::OFF_MISC);
  volatile unsigned* ticket = reinterpret_cast<volatile unsigned*>(smem_raw + C::OFF_MISC + 4);
  volatile float* null_score = reinterpret_cast<volatile float*>(smem_raw + C::OFF_MISC + 8);

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int total = (p.n_pairs + p.n_items) * p.H;

  if (tid == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], C::NCW);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  const size_t head_elems = (size_t)2 * C::R * D;  // K and V rows of one head

  // ------------------------------------------------------------------ producer
  if (warp == C::NCW) {
    if (lane != 0) return;
    uint32_t fill = 0;
    uint32_t last_round[C::NSTAGE];
    bool issued[C::NSTAGE];
#pragma unroll
    for (int s = 0; s < C::NSTAGE; ++s) { issued[s] = false; last_round[s] = 0; }
    bool ok = true;
    for (int u = blockIdx.x; u < total && ok; u += gridDim.x) {
      const Unit U = unit_of(p, u);
      const DecodeItem& it = p.items[U.item];
      for (int t = 0; t < U.nt; ++t, ++fill) {
        const int st = fill % C::NSTAGE;
        const uint32_t round = fill / C::NSTAGE;
        if (round > 0 && !mbar_wait_bounded(&empty[st], (round - 1) & 1, abort_flag)) {
          if (!*abort_flag) record_error(p.err, kDevErrWaitEmpty);
          *abort_flag = 1;
          ok = false;
          break;
        }
        uint8_t* kdst = stages + st * C::STAGE_BYTES;
        uint8_t* vdst = kdst + C::TILE_BYTES;
        if (!U.sa) {
          const int slot = p.table[(size_t)it.seq * p.max_blocks + U.b0 + t];
          if (slot < 0 || slot >= p.capacity) {
            record_error(p.err, kDevErrBounds);
            mbar_arrive(&full[st]);  // stale stage contents; the error is flagged
          } else {
            const uint16_t* src =
                p.pool + (size_t)slot * p.slot_elems + ((size_t)p.layer * p.H + U.h) * head_elems;
            mbar_arrive_expect_tx(&full[st], C::STAGE_BYTES);
            bulk_g2s(kdst, src, C::TILE_BYTES, &full[st]);
            bulk_g2s(vdst, src + C::R * D, C::TILE_BYTES, &full[st]);
          }
        } else {
          const int pos = it.pos;
          const uint32_t row_bytes = D * 2;
          const uint16_t* ib =
              p.inblock + (((size_t)it.seq * p.L + p.layer) * p.H + U.h) * (size_t)2 * kBlockTok * D;
          const size_t qoff = ((size_t)U.item * p.H + U.h) * D;
          mbar_arrive_expect_tx(&full[st], 2u * (uint32_t)(pos + 1) * row_bytes);
          if (pos > 0) {
            bulk_g2s(kdst, ib, (uint32_t)pos * row_bytes, &full[st]);
            bulk_g2s(vdst, ib + (size_t)kBlockTok * D, (uint32_t)pos * row_bytes, &full[st]);
          }
          bulk_g2s(kdst + pos * row_bytes, p.k_new + qoff, row_bytes, &full[st]);
          bulk_g2s(vdst + pos * row_bytes, p.v_new + qoff, row_bytes, &full[st]);
        }
        issued[st] = true;
        last_round[st] = round;
      }
    }
    if (!ok) {
      // give copies already in flight (bounded) time to land before exit
#pragma unroll
      for (int s = 0; s < C::NSTAGE; ++s)
        if (issued[s]) mbar_wait_bounded(&full[s], last_round[s] & 1, nullptr);
    }
    return;
  }

  // ----------------------------------------------------------------- consumers
  const int w = warp;
  const int g = lane / C::LPR;  // row group within a warp load
  const int c = lane % C::LPR;  // 16-byte column chunk
  constexpr unsigned FULL = 0xffffffffu;
  uint32_t fill = 0;

  for (int u = blockIdx.x; u < total; u += gridDim.x) {
    const Unit U = unit_of(p, u);
    const DecodeItem& it = p.items[U.item];
    const size_t qoff = ((size_t)U.item * p.H + U.h) * D;
    const int n_valid = U.sa ? it.pos + 1 : C::R;

    float q[8];
    {
      const uint4 qv = *reinterpret_cast<const uint4*>((U.sa ? p.qs : p.qc) + qoff + c * 8);
      unpack8(qv, q);
#pragma unroll
      for (int j = 0; j < 8; ++j) q[j] *= p.scale_log2;
    }
    float m = -INFINITY, l = 0.f, acc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = 0.f;
    bool failed = false;

    for (int t = 0; t < U.nt; ++t, ++fill) {
      const int st = fill % C::NSTAGE;
      const uint32_t round = fill / C::NSTAGE;
      if (!failed && !mbar_wait_bounded(&full[st], round & 1, abort_flag)) {
        if (!*abort_flag) record_error(p.err, kDevErrWaitFull);
        *abort_flag = 1;
        failed = true;
      }
      if (failed) continue;
      const uint8_t* kt = stages + st * C::STAGE_BYTES;
      const uint8_t* vt = kt + C::TILE_BYTES;

      float s[C::ITERS];
      float tmax = -INFINITY;
#pragma unroll
      for (int i = 0; i < C::ITERS; ++i) {
        const int r = w * C::ROWS_PER_WARP + i * C::RPI + g;
        float dot = 0.f;
        if (r < n_valid) {
          const uint4 kv = *reinterpret_cast<const uint4*>(kt + r * (D * 2) + c * 16);
          float kf[8];
          unpack8(kv, kf);
#pragma unroll
          for (int j = 0; j < 8; ++j) dot = fmaf(q[j], kf[j], dot);
        }
#pragma unroll
        for (int o = 1; o < C::LPR; o <<= 1) dot += __shfl_xor_sync(FULL, dot, o);
        s[i] = r < n_valid ? dot : -INFINITY;
        tmax = fmaxf(tmax, s[i]);
      }
#pragma unroll
      for (int o = C::LPR; o < 32; o <<= 1) tmax = fmaxf(tmax, __shfl_xor_sync(FULL, tmax, o));
      const float m_new = fmaxf(m, tmax);
      if (m_new != -INFINITY) {
        const float alpha = exp2f(m - m_new);
        l *= alpha;
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] *= alpha;
#pragma unroll
        for (int i = 0; i < C::ITERS; ++i) {
          const int r = w * C::ROWS_PER_WARP + i * C::RPI + g;
          if (r < n_valid) {
            const float pr = exp2f(s[i] - m_new);
            l += pr;
            const uint4 vv = *reinterpret_cast<const uint4*>(vt + r * (D * 2) + c * 16);
            float vf[8];
            unpack8(vv, vf);
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] = fmaf(pr, vf[j], acc[j]);
          }
        }
        m = m_new;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }

    // merge the row groups of this warp (fixed butterfly)
#pragma unroll
    for (int o = C::LPR; o < 32; o <<= 1) {
      l += __shfl_xor_sync(FULL, l, o);
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] += __shfl_xor_sync(FULL, acc[j], o);
    }
    if (g == 0) {
      float* cw = comb + w * (D + 2);
#pragma unroll
      for (int j = 0; j < 8; ++j) cw[2 + c * 8 + j] = acc[j];
      if (c == 0) { cw[0] = m; cw[1] = l; }
    }
    if (bar_any(1, C::NCW * 32, failed)) break;  // uniform across consumer warps

    // merge the four warps in warp order; thread j owns column j
    const int nsplit = U.sa ? 1 : ceil_div(it.nblk, decode_split_blocks(it.nblk));
    const bool direct = U.sa || (nsplit == 1 && !p.null_kv);
    if (tid < D) {
      float M = -INFINITY;
#pragma unroll
      for (int ww = 0; ww < C::NCW; ++ww) M = fmaxf(M, comb[ww * (D + 2)]);
      float Lsum = 0.f, A = 0.f;
#pragma unroll
      for (int ww = 0; ww < C::NCW; ++ww) {
        const float f = exp2f(comb[ww * (D + 2)] - M);
        Lsum = fmaf(f, comb[ww * (D + 2) + 1], Lsum);
        A = fmaf(f, comb[ww * (D + 2) + 2 + tid], A);
      }
      if (direct) {
        uint16_t* out = U.sa ? p.osa : p.oca;
        const __nv_bfloat16 o = __float2bfloat16_rn(A / Lsum);
        out[qoff + tid] = *reinterpret_cast<const uint16_t*>(&o);
      } else {
        float* pp = p.part + ((size_t)(it.pair_begin + U.split) * p.H + U.h) * (D + 2);
        pp[2 + tid] = A;
        if (tid == 0) { pp[0] = M; pp[1] = Lsum; }
      }
    }
    if (U.sa) {
      // store the new token's k, v as in-block row p for the next steps
      if (w == 0 && lane < 2 * C::LPR) {
        const int kv = lane / C::LPR, cc = lane % C::LPR;
        uint16_t* ib = p.inblock + (((size_t)it.seq * p.L + p.layer) * p.H + U.h) * (size_t)2 * kBlockTok * D +
                       (size_t)kv * kBlockTok * D + (size_t)it.pos * D;
        const uint16_t* src = (kv ? p.v_new : p.k_new) + qoff;
        *reinterpret_cast<uint4*>(ib + cc * 8) = *reinterpret_cast<const uint4*>(src + cc * 8);
      }
      // a sequence with no readable memory block: oca is the null row's
      // value (a softmax over one row) or zero
      if (it.nblk == 0 && tid < D) {
        float val = 0.f;
        if (p.null_kv) val = bf16lo(p.null_kv[((size_t)p.layer * p.H + U.h) * 2 * D + D + tid]);
        const __nv_bfloat16 o = __float2bfloat16_rn(val);
        p.oca[qoff + tid] = *reinterpret_cast<const uint16_t*>(&o);
      }
    } else if (!direct) {
      __threadfence();
      named_bar_sync(1, C::NCW * 32);
      if (tid == 0) *ticket = atomicAdd(&p.counters[U.item * p.H + U.h], 1u);
      named_bar_sync(1, C::NCW * 32);
      if (*ticket == (unsigned)(nsplit - 1)) {
        __threadfence();
        if (p.null_kv && w == 0) {
          // null-row score with the same scaled-q dot product as the rows
          const uint16_t* kn = p.null_kv + ((size_t)p.layer * p.H + U.h) * 2 * D;
          float dot = 0.f;
          if (lane < C::LPR) {
            const uint4 kv = *reinterpret_cast<const uint4*>(kn + lane * 8);
            float kf[8];
            unpack8(kv, kf);
            float qq[8];
            unpack8(*reinterpret_cast<const uint4*>(p.qc + qoff + lane * 8), qq);
#pragma unroll
            for (int j = 0; j < 8; ++j) dot = fmaf(qq[j] * p.scale_log2, kf[j], dot);
          }
#pragma unroll
          for (int o = 1; o < C::LPR; o <<= 1) dot += __shfl_xor_sync(FULL, dot, o);
          if (lane == 0) *null_score = dot;
        }
        named_bar_sync(1, C::NCW * 32);
        if (tid < D) {
          const float* pb = p.part + ((size_t)it.pair_begin * p.H + U.h) * (D + 2);
          const size_t ps = (size_t)p.H * (D + 2);
          float M = p.null_kv ? *null_score : -INFINITY;
          for (int s = 0; s < nsplit; ++s) M = fmaxf(M, __ldcg(pb + s * ps));
          float Lsum = 0.f, A = 0.f;
          if (p.null_kv) {
            const float f = exp2f(*null_score - M);
            Lsum = f;
            A = f * bf16lo(p.null_kv[((size_t)p.layer * p.H + U.h) * 2 * D + D + tid]);
          }
          for (int s = 0; s < nsplit; ++s) {
            const float f = exp2f(__ldcg(pb + s * ps) - M);
            Lsum = fmaf(f, __ldcg(pb + s * ps + 1), Lsum);
            A = fmaf(f, __ldcg(pb + s * ps + 2 + tid), A);
          }
          const __nv_bfloat16 o = __float2bfloat16_rn(A / Lsum);
          p.oca[qoff + tid] = *reinterpret_cast<const uint16_t*>(&o);
        }
        if (tid == 0) p.counters[U.item * p.H + U.h] = 0u;
      }
    }
    named_bar_sync(1, C::NCW * 32);  // comb[] and the ticket are reused next unit
  }
}

int decode_max_grid(int D, int num_sms) {
  (void)D;
  return 2 * num_sms;
}

cudaError_t launch_decode(const DecodeParams& p, int D, int grid, cudaStream_t st) {
  if (D == 64) {
    using C = DecCfg<64>;
    cudaError_t e = cudaFuncSetAttribute(decode_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    decode_kernel<64><<<grid, C::THREADS, C::SMEM, st>>>(p);
  } else if (D == 128) {
    using C = DecCfg<128>;
    cudaError_t e = cudaFuncSetAttribute(decode_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    decode_kernel<128><<<grid, C::THREADS, C::SMEM, st>>>(p);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace smem
