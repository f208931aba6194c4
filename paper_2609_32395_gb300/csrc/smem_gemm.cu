// smem_gemm.cu -- the dense projections of the reader layer on tcgen05 tensor
// cores (arXiv 2609.32395, Sec. 2 "Model", App. A "Reader": pre-LN residual
// branches with Q/K/V/O maps and a 4d GELU FFN; memory rows projected to each
// layer's keys and values).
//
// out[m][n] = epilogue( alpha * sum_k A[m][k] W[k][n] ), bf16 operands, fp32
// accumulation in tensor memory. The reader's shapes are skinny (64 query
// tokens of a block, or one token per decoded sequence, against d x d .. d x
// 4d weights), so a projection streams its weights once and its time is set
// by latency, not by math. The kernel is laid out for that:
//
//   * a CTA owns 128 rows (tokens) x BN output columns; MMA M = 128, N = BN
//     (64 or 128), K = 16 per instruction, issued by one thread;
//   * the K range is cut over a thread-block cluster of up to 8 CTAs: each
//     accumulates its share of K in tensor memory, parks the fp32 partial in
//     its shared memory, and every CTA then adds the partials of a slice of
//     the rows over distributed shared memory in rank order (a fixed order:
//     bitwise reproducible, no global workspace, no atomics);
//   * weights arrive by TMA (128-byte swizzle) into a 4-stage ring; the first
//     stages are requested before the kernel waits for the previous kernel
//     (programmatic dependent launch), since weights do not depend on it;
//   * the A operand is written into shared memory by six producer warps: the
//     bf16 activations, or -- for the pre-LN projections -- LayerNorm of the
//     fp32 residual stream computed on the fly. Row statistics come from the
//     cluster: each CTA reduces its own K slice (mean and centred sum of
//     squares, two passes), the slices are combined in rank order (the
//     pairwise update of Chan, Golub and LeVeque), so no CTA reads more of a
//     row than its slice;
//   * epilogues: bf16 store (optionally into per-head column groups, the pool
//     slot layout), fp32 residual add, GELU (x * Phi(x), erff) to bf16, and
//     for the q|k|v projection of a one-block prefill the rotary turn of the
//     query and key columns by token offset plus the copy of the key/value
//     columns into the block's in-block rows.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cudaTypedefs.h>

#include <algorithm>

#include "smem_device.cuh"
#include "smem_internal.h"
#include "smem_tc.cuh"

namespace smem {

namespace {

constexpr int kBM = 128;          // rows (tokens) per CTA
constexpr int kNS = 4;            // ring stages
constexpr int kThreads = 256;     // warp 0: weight TMA, warp 1: MMA + TMEM, warps 2-7: A producers
constexpr int kAProd = 192;       // A-producer threads (warps 2-7); warps 4-7 also run the epilogue
constexpr int kMaxCluster = 8;

template <int BN>
struct Gm {
  static constexpr int A_BYTES = kBM * 128;  // [128 rows][64 k] bf16, 128-byte swizzle
  static constexpr int W_BYTES = BN * 128;   // [64 k][BN] as BN/64 boxes of 8 KB, or [BN][64 k]
  static constexpr int STAGE = A_BYTES + W_BYTES;
  static constexpr int PSTRIDE = BN + 4;     // floats per row of a parked partial
  static constexpr int OFF_STAT = kNS * STAGE;          // [128] float2: (mean, M2) of this CTA's K slice
  static constexpr int OFF_NORM = OFF_STAT + kBM * 8;   // [128] float2: (mean, rstd) of the whole row
  static constexpr int OFF_BAR = OFF_NORM + kBM * 8;    // full_w[NS] | full_a[NS] | empty[NS] | acc
  static constexpr int NBAR = 3 * kNS + 1;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;   // TMEM slot, abort flag
  static constexpr int SMEM = OFF_MISC + 16 + 1024;
  static_assert(kBM * PSTRIDE * 4 <= kNS * STAGE, "partials fit in the ring");
};

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void ld_tmem_32x32b_x32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 " SMEM_REGLIST32 ", [%32];"
               : SMEM_R32(r)
               : "r"(taddr)
               : "memory");
}

__device__ __forceinline__ float4 ld_dsmem_f32x4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

__device__ __forceinline__ float bf16_round(float v) { return __bfloat162float(__float2bfloat16_rn(v)); }

__device__ __forceinline__ float gelu_erf(float v) { return 0.5f * v * (1.f + erff(v * 0.70710678118654752f)); }

// Barrier over every thread of the cluster (or of the CTA without one).
__device__ __forceinline__ void group_sync(int ks) {
  if (ks > 1) tc::cluster_sync();
  else __syncthreads();
}

// Epilogue of NV consecutive output columns col.. of row `row` (tile-local
// row r for the rotary phase / in-block row); v holds alpha * accumulator.
template <int NV>
__device__ __forceinline__ void epilogue(const GemmParams& p, int bz, int row, int col, float* v) {
  if (p.epi == kEpiAddF32) {
    const int g = col / p.col_group, cc = col - g * p.col_group;
    float* o = static_cast<float*>(p.out) + (size_t)bz * p.o_bs + (size_t)g * p.group_stride + (size_t)row * p.ldo + cc;
#pragma unroll
    for (int e = 0; e < NV; e += 4) {
      float4 x = *reinterpret_cast<float4*>(o + e);
      x.x += v[e];
      x.y += v[e + 1];
      x.z += v[e + 2];
      x.w += v[e + 3];
      *reinterpret_cast<float4*>(o + e) = x;
    }
    return;
  }
  if (p.epi == kEpiGeluBf16) {
#pragma unroll
    for (int e = 0; e < NV; ++e) v[e] = gelu_erf(v[e]);
  } else if (p.rope_tab && col < p.rope_cols) {
    // q|k columns of a prefill turn by the token's in-block offset (rounded
    // to bf16 first, as the stored projection)
    const float2* tab = p.rope_tab + (size_t)row * (p.rope_D / 2) + (col % p.rope_D) / 2;
#pragma unroll
    for (int e = 0; e < NV; e += 2) {
      const float x0 = bf16_round(v[e]), x1 = bf16_round(v[e + 1]);
      const float2 c = tab[e / 2];
      v[e] = x0 * c.x - x1 * c.y;
      v[e + 1] = x0 * c.y + x1 * c.x;
    }
  }
  uint32_t w[NV / 2];
#pragma unroll
  for (int e = 0; e < NV; e += 2) w[e / 2] = pack_bf16x2(v[e], v[e + 1]);
  const int g = col / p.col_group, cc = col - g * p.col_group;
  uint16_t* o = static_cast<uint16_t*>(p.out) + (size_t)bz * p.o_bs + (size_t)g * p.group_stride + (size_t)row * p.ldo + cc;
#pragma unroll
  for (int e = 0; e < NV / 8; ++e)
    *reinterpret_cast<uint4*>(o + 8 * e) = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
  if (NV == 4) *reinterpret_cast<uint2*>(o) = make_uint2(w[0], w[1]);
  if (p.ib && col >= p.ib_col0 && col < p.ib_col0 + 2 * p.ib_kvd) {
    // key/value columns of a prefill also become the block's in-block rows
    const int c2 = col - p.ib_col0;
    const int kv = c2 / p.ib_kvd, h = (c2 - kv * p.ib_kvd) / p.ib_D, e0 = c2 % p.ib_D;
    uint16_t* ib = p.ib + ((size_t)(h * 2 + kv) * kBlockTok + row) * p.ib_D + e0;
#pragma unroll
    for (int e = 0; e < NV / 8; ++e)
      *reinterpret_cast<uint4*>(ib + 8 * e) = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
    if (NV == 4) *reinterpret_cast<uint2*>(ib) = make_uint2(w[0], w[1]);
  }
}

template <int BN>
__global__ void __launch_bounds__(kThreads, 1) gemm_kernel(const __grid_constant__ GemmParams p) {
  using C = Gm<BN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ks = p.ks;
  const int rank = ks > 1 ? (int)tc::cluster_ctarank() : 0;
  const int n0 = (blockIdx.x / ks) * BN;
  const int m0 = blockIdx.y * kBM;
  const int bz = blockIdx.z;
  const int mrows = min(kBM, p.M - m0);
  const int c0 = (int)((long long)p.chunks * rank / ks);
  const int c1 = (int)((long long)p.chunks * (rank + 1) / ks);
  const int nch = c1 - c0;
  uint64_t* full_w = reinterpret_cast<uint64_t*>(base + C::OFF_BAR);
  uint64_t* full_a = full_w + kNS;
  uint64_t* empty = full_a + kNS;
  uint64_t* acc_bar = empty + kNS;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(base + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + C::OFF_MISC + 4);
  float2* stat = reinterpret_cast<float2*>(base + C::OFF_STAT);
  float2* norm = reinterpret_cast<float2*>(base + C::OFF_NORM);

  if (threadIdx.x == 0) {
    griddep_launch();  // the next kernel may start its own prologue
    for (int s = 0; s < kNS; ++s) {
      mbar_init(&full_w[s], 1);
      mbar_init(&full_a[s], kAProd);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.wmap)) : "memory");
  }
  if (warp == 1) tc::alloc(tslot, BN);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = *tslot;

  auto load_w = [&](int i) {  // chunk i of this split into stage i % NS (thread 0 of warp 0)
    const int st = i % kNS;
    uint8_t* wb = base + st * C::STAGE + C::A_BYTES;
    const int k = (c0 + i) * 64;
    mbar_arrive_expect_tx(&full_w[st], C::W_BYTES);
    if (p.b_kmajor) {
      tma_load_2d(wb, &p.wmap, k + p.w_boff * bz, n0, &full_w[st]);
    } else {
#pragma unroll
      for (int j = 0; j < BN / 64; ++j) tma_load_2d(wb + j * 8192, &p.wmap, n0 + j * 64 + p.w_boff * bz, k, &full_w[st]);
    }
  };
  // weights do not depend on the previous kernel: request the first stages now
  int issued = 0;
  if (warp == 0 && lane == 0)
    for (; issued < min(kNS, nch); ++issued) load_w(issued);

  const bool aprod = warp >= 2;
  const int atid = threadIdx.x - 64;  // 0..191 for the A producers
  // everything below may read the previous kernel's outputs or write this
  // kernel's (the split-K reduction runs on every thread)
  griddep_wait();
  // ---- LayerNorm statistics of this CTA's K slice (two passes), per row
  const int kb = min(c0 * 64, p.K), ke = min(c1 * 64, p.K);
  if (p.ln && aprod) {
    const float* xa = static_cast<const float*>(p.a) + (size_t)bz * p.a_bs;
    const int n4 = (ke - kb) / 4;
    for (int r = warp - 2; r < mrows; r += 6) {
      const float4* xr = reinterpret_cast<const float4*>(xa + (size_t)(m0 + r) * p.lda + kb);
      float s = 0.f;
      for (int c = lane; c < n4; c += 32) {
        const float4 v = xr[c];
        s += (v.x + v.y) + (v.z + v.w);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      const float mean = n4 ? s / (float)(4 * n4) : 0.f;
      float q = 0.f;
      for (int c = lane; c < n4; c += 32) {
        const float4 v = xr[c];
        const float a = v.x - mean, b = v.y - mean, cc = v.z - mean, d = v.w - mean;
        q += (a * a + b * b) + (cc * cc + d * d);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
      if (lane == 0) stat[r] = make_float2(mean, q);
    }
  }
  group_sync(ks);  // every split's statistics are visible in the cluster
  if (p.ln && aprod) {
    // combine the slices in rank order: counts, means and centred sums of squares
    for (int r = atid; r < mrows; r += kAProd) {
      float cnt = 0.f, mean = 0.f, m2 = 0.f;
      for (int s = 0; s < ks; ++s) {
        const int sb = min((int)((long long)p.chunks * s / ks) * 64, p.K);
        const int se = min((int)((long long)p.chunks * (s + 1) / ks) * 64, p.K);
        const float nb = (float)(se - sb);
        if (nb == 0.f) continue;
        float2 v;
        if (ks > 1) {
          const uint32_t ra = tc::dsmem_addr(smem_u32(&stat[r]), (uint32_t)s);
          v = tc::ld_dsmem_f32x2(ra);
        } else {
          v = stat[r];
        }
        if (cnt == 0.f) {
          cnt = nb;
          mean = v.x;
          m2 = v.y;
        } else {
          const float tot = cnt + nb, delta = v.x - mean;
          mean = mean + delta * (nb / tot);
          m2 = m2 + v.y + delta * delta * (cnt * nb / tot);
          cnt = tot;
        }
      }
      norm[r] = make_float2(mean, rsqrtf(m2 / (float)p.K + p.eps));
    }
    named_bar_sync(1, kAProd);
  }

  bool ok = true;
  if (warp == 0) {
    // ------------------------------------------------------------ weight TMA
    if (lane == 0) {
      for (int i = issued; i < nch; ++i) {
        const int st = i % kNS;
        if (!mbar_wait_bounded(&empty[st], ((i / kNS) - 1) & 1, abort_flag)) {
          ok = false;
          break;
        }
        load_w(i);
        ++issued;
      }
      if (!ok) {
        record_error(p.err, kDevErrWaitEmpty);
        *abort_flag = 1;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(128, BN, 0, p.b_kmajor ? 0 : 1);
      for (int i = 0; i < nch; ++i) {
        const int st = i % kNS;
        ok = mbar_wait_bounded(&full_w[st], (i / kNS) & 1, abort_flag) &&
             mbar_wait_bounded(&full_a[st], (i / kNS) & 1, abort_flag);
        if (!ok) break;
        tc::fence_after();
        const uint32_t aa = smem_u32(base + st * C::STAGE);
        const uint32_t wa = aa + C::A_BYTES;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint64_t bd = p.b_kmajor ? tc::sdesc_sw128(wa + k * 32, 16, 1024)
                                         : tc::sdesc_sw128(wa + k * 2048, 8192, 1024);
          tc::mma_bf16(tmem, tc::sdesc_sw128(aa + k * 32, 16, 1024), bd, idesc, (i > 0 || k > 0) ? 1u : 0u);
        }
        tc::commit(&empty[st]);
      }
      if (!ok) {
        record_error(p.err, kDevErrWaitFull);
        *abort_flag = 1;
      }
      tc::commit(acc_bar);  // arrives once every MMA issued above has completed
    }
  } else {
    // ------------------------------------------------------------ A producers
    const int j = atid & 7;  // 16-byte column group of the chunk this thread fills
    for (int i = 0; i < nch && ok; ++i) {
      const int st = i % kNS;
      if (i >= kNS && !mbar_wait_bounded(&empty[st], ((i / kNS) - 1) & 1, abort_flag)) {
        ok = false;
        break;
      }
      uint8_t* at = base + st * C::STAGE;
      const int kc = (c0 + i) * 64 + j * 8;  // first column of this thread's group
      const bool col_in = kc < p.K;
      float g[8], bb[8];
      if (p.ln && col_in) {
        const float4 g0 = *reinterpret_cast<const float4*>(p.ln_g + kc);
        const float4 g1 = *reinterpret_cast<const float4*>(p.ln_g + kc + 4);
        const float4 b0 = *reinterpret_cast<const float4*>(p.ln_b + kc);
        const float4 b1 = *reinterpret_cast<const float4*>(p.ln_b + kc + 4);
        g[0] = g0.x, g[1] = g0.y, g[2] = g0.z, g[3] = g0.w, g[4] = g1.x, g[5] = g1.y, g[6] = g1.z, g[7] = g1.w;
        bb[0] = b0.x, bb[1] = b0.y, bb[2] = b0.z, bb[3] = b0.w, bb[4] = b1.x, bb[5] = b1.y, bb[6] = b1.z, bb[7] = b1.w;
      }
      for (int r = atid >> 3; r < kBM; r += kAProd / 8) {
        uint4 w = make_uint4(0u, 0u, 0u, 0u);
        if (r < mrows && col_in) {
          if (p.ln) {
            const float* xr = static_cast<const float*>(p.a) + (size_t)bz * p.a_bs + (size_t)(m0 + r) * p.lda + kc;
            const float4 v0 = *reinterpret_cast<const float4*>(xr);
            const float4 v1 = *reinterpret_cast<const float4*>(xr + 4);
            const float2 nr = norm[r];
            const float x[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
            uint32_t h[4];
#pragma unroll
            for (int e = 0; e < 4; ++e)
              h[e] = pack_bf16x2((x[2 * e] - nr.x) * nr.y * g[2 * e] + bb[2 * e],
                                 (x[2 * e + 1] - nr.x) * nr.y * g[2 * e + 1] + bb[2 * e + 1]);
            w = make_uint4(h[0], h[1], h[2], h[3]);
          } else {
            w = *reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(p.a) + (size_t)bz * p.a_bs +
                                                (size_t)(m0 + r) * p.lda + kc);
          }
        }
        *reinterpret_cast<uint4*>(at + r * 128 + ((j ^ (r & 7)) << 4)) = w;
      }
      fence_proxy_async_smem();
      mbar_arrive(&full_a[st]);
    }
    if (!ok) {
      record_error(p.err, kDevErrWaitEmpty);
      *abort_flag = 1;
    }
  }

  // ---- epilogue: warps 4-7 read the accumulator rows (TMEM lanes 32(w-4)..)
  float* part = reinterpret_cast<float*>(base);  // the ring, free once every MMA completed
  if (warp >= 4) {
    const int q = warp - 4;
    const int r = 32 * q + lane;
    const bool done = mbar_wait_bounded(acc_bar, 0, nullptr);
    if (!done && lane == 0) record_error(p.err, kDevErrWaitMma);
    tc::fence_after();
#pragma unroll 1
    for (int cb = 0; cb < BN / 32; ++cb) {
      uint32_t u[32];
      ld_tmem_32x32b_x32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(cb * 32), u);
      tc::wait_ld();
      const int col = n0 + cb * 32;
      if (r < mrows) {
        float v[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) v[e] = done ? __uint_as_float(u[e]) * p.alpha : 0.f;
        if (ks == 1) {
          if (col < p.N) epilogue<32>(p, bz, m0 + r, col, v);
        } else {
#pragma unroll
          for (int e = 0; e < 32; e += 4)
            *reinterpret_cast<float4*>(part + r * C::PSTRIDE + cb * 32 + e) = make_float4(v[e], v[e + 1], v[e + 2], v[e + 3]);
        }
      }
    }
    tc::fence_before();
  }
  if (ks > 1) {
    tc::cluster_sync();  // every split's partial rows are parked
    // rank s adds the partials of rows [s * rp, (s + 1) * rp) in rank order
    const int rp = (mrows + ks - 1) / ks;
    const int r0 = rank * rp, r1 = min(mrows, r0 + rp);
    constexpr int G4 = BN / 4;
    for (int it = threadIdx.x; it < (r1 - r0) * G4; it += kThreads) {
      const int r = r0 + it / G4, c = (it % G4) * 4;
      if (n0 + c >= p.N) continue;
      const uint32_t la = smem_u32(part + r * C::PSTRIDE + c);
      float4 s = ld_dsmem_f32x4(tc::dsmem_addr(la, 0));
      for (int t = 1; t < ks; ++t) {
        const float4 v = ld_dsmem_f32x4(tc::dsmem_addr(la, (uint32_t)t));
        s.x += v.x;
        s.y += v.y;
        s.z += v.z;
        s.w += v.w;
      }
      float v[4] = {s.x, s.y, s.z, s.w};
      epilogue<4>(p, bz, m0 + r, n0 + c, v);
    }
    tc::cluster_sync();  // no CTA leaves while a peer may still read its partials
  } else {
    __syncthreads();
  }
  if (warp == 1) {
    tc::fence_after();
    tc::dealloc(tmem, BN);
  }
  if (warp == 0 && lane == 0 && !ok) {
    // copies already requested land before the CTA exits (bounded)
    for (int i = 0; i < issued; ++i) mbar_wait_bounded(&full_w[i % kNS], (i / kNS) & 1, nullptr);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  return fn;
}

template <int BN>
cudaError_t launch_bn(GemmParams& p, int tiles_n, int mtiles, int batch, bool pdl, cudaStream_t st) {
  using C = Gm<BN>;
  cudaError_t e = ensure_smem_limit<100 + BN>(gemm_kernel<BN>, C::SMEM);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(tiles_n * p.ks), (unsigned)mtiles, (unsigned)batch);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (p.ks > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = (unsigned)p.ks;
    at[na].val.clusterDim.y = 1;
    at[na].val.clusterDim.z = 1;
    ++na;
  }
  if (pdl) {
    at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = at;
  cfg.numAttrs = (unsigned)na;
  return cudaLaunchKernelEx(&cfg, gemm_kernel<BN>, p);
}

}  // namespace

// Tile and split plan of a projection: the widest N tile and the largest
// cluster (<= 8 CTAs, at most one 64-column K chunk per CTA minimum) that
// keep the grid within one wave of the device's SMs. A function of the shape
// and the SM count only.
GemmPlan gemm_plan(int M, int N, int K, int batch, int num_sms) {
  const int chunks = (K + 63) / 64;
  const int mtiles = (M + kBM - 1) / kBM;
  GemmPlan best{128, 1, 0};
  for (int bn : {128, 64}) {
    const int tiles = (N + bn - 1) / bn * mtiles * batch;
    int ks = tiles >= num_sms ? 1 : std::max(1, num_sms / tiles);
    ks = std::min(ks, std::min(kMaxCluster, std::max(1, chunks)));
    const int ctas = tiles * ks;
    if (ctas > best.ctas) best = GemmPlan{bn, ks, ctas};
  }
  return best;
}

cudaError_t launch_gemm(const GemmCall& g, int num_sms, cudaStream_t st) {
  if (g.M <= 0 || g.N <= 0 || g.batch <= 0) return cudaSuccess;
  if (g.N % 32 || g.K % 32 || g.K <= 0) return cudaErrorInvalidValue;
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const GemmPlan pl = gemm_plan(g.M, g.N, g.K, g.batch, num_sms);
  static thread_local GemmParams p;
  p = GemmParams{};
  const cuuint64_t dims[2] = {(cuuint64_t)g.w_cols, (cuuint64_t)g.w_rows};
  const cuuint64_t strides[1] = {(cuuint64_t)g.ldw * 2};
  const cuuint32_t box[2] = {64u, g.b_kmajor ? (cuuint32_t)pl.bn : 64u};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = enc(&p.wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(g.w), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  p.a = g.a;
  p.ln_g = g.ln_g;
  p.ln_b = g.ln_b;
  p.out = g.out;
  p.rope_tab = g.rope_tab;
  p.ib = g.ib;
  p.a_bs = g.a_bs;
  p.o_bs = g.o_bs;
  p.group_stride = g.group_stride;
  p.lda = g.lda;
  p.ldo = g.ldo;
  p.M = g.M;
  p.N = g.N;
  p.K = g.K;
  p.ln = g.ln_g != nullptr;
  p.b_kmajor = g.b_kmajor;
  p.w_boff = g.w_boff;
  p.epi = g.epi;
  p.col_group = g.col_group > 0 ? g.col_group : g.N;
  p.ks = pl.ks;
  p.chunks = (g.K + 63) / 64;
  p.rope_cols = g.rope_cols;
  p.rope_D = g.rope_D;
  p.ib_col0 = g.ib_col0;
  p.ib_kvd = g.ib_kvd;
  p.ib_D = g.ib_D;
  p.alpha = g.alpha;
  p.eps = kLayerNormEps;
  p.err = g.err;
  const int tiles_n = (g.N + pl.bn - 1) / pl.bn;
  const int mtiles = (g.M + kBM - 1) / kBM;
  return pl.bn == 128 ? launch_bn<128>(p, tiles_n, mtiles, g.batch, g.pdl, st)
                      : launch_bn<64>(p, tiles_n, mtiles, g.batch, g.pdl, st);
}

}  // namespace smem
