// smem_gemm.cu -- the dense projections of the reader layer on tcgen05 tensor
// cores, and its LayerNorm (arXiv 2609.32395, Sec. 2 "Model", App. A
// "Reader": pre-LN residual branches with Q/K/V/O maps and a 4d GELU FFN;
// memory rows projected to each layer's keys and values).
//
// out[m][n] = epilogue( alpha * sum_k A[m][k] W[k][n] ), bf16 operands, fp32
// accumulation in tensor memory. The reader's shapes are skinny (64 query
// tokens of a block, or one token per decoded sequence, against d x d .. d x
// 4d weights), so a projection streams its weights once and its time is set
// by latency, not by math. The kernel is laid out for that:
//
//   * a CTA of four warps owns 128 rows (tokens) x BN output columns; MMA
//     M = 128, N = BN (64 or 128), K = 16 per instruction, issued by one
//     thread; warp 0 issues the copies, warp 1 the MMAs, then all four read
//     the accumulator (TMEM lanes 32w..32w+31) and run the epilogue;
//   * both operands arrive by TMA (128-byte swizzle) into a 4-stage ring:
//     weights as W[k][n] (MN-major boxes) or W[n][k] (K-major), activations as
//     a [batch][M][K] view (rows and columns past M and K read as zero). The
//     weight copies of the first stages are requested before the kernel waits
//     for the previous kernel (programmatic dependent launch): weights never
//     depend on it;
//   * the K range is cut over a thread-block cluster of up to 8 CTAs when the
//     output tiles alone would leave SMs idle: each CTA accumulates its share
//     of K, parks the fp32 partial in its shared memory, and every CTA then
//     adds the partials of a slice of the rows over distributed shared memory
//     in rank order (a fixed order: bitwise reproducible, no global workspace,
//     no atomics). The plan keeps every cluster in one wave (a GPC hosts only
//     whole clusters);
//   * epilogues: bf16 store (optionally into per-head column groups, the pool
//     slot layout), fp32 residual add, GELU (x * Phi(x), erff) to bf16, and
//     for the q|k|v projection of a one-block prefill the rotary turn of the
//     query and key columns by token offset plus the copy of the key/value
//     columns into the block's in-block rows.
//
// LayerNorm runs as its own small kernel (one warp per token, fp32 two-pass
// moments, bf16 out), launched with programmatic dependent launch as well.
// A form that normalised the fp32 rows inside the projection (per-slice
// statistics combined across the cluster) measured slower: its producer
// warps spent a few microseconds per phase, mostly waiting for instruction
// fetch, against about one for this kernel.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdlib>

#include "smem_device.cuh"
#include "smem_internal.h"
#include "smem_tc.cuh"

namespace smem {

namespace {

constexpr int kBM = 128;          // rows (tokens) per CTA
constexpr int kNS = 4;            // ring stages
constexpr int kThreads = 128;     // warp 0: TMA, warp 1: TMEM + MMA; then all four: epilogue
constexpr int kMaxCluster = 8;
constexpr int kLnThreads = 256;   // LayerNorm: 8 warps, one token each

// Shared memory: a ring of `ns` stages (ns <= kNS, sized per launch to the
// K chunks a CTA streams, so that short projections leave room for the next
// kernel's CTAs), then the barriers; the drained ring also parks the split
// partials (ring_bytes covers them).
template <int BN>
struct Gm {
  static constexpr int A_BYTES = kBM * 128;  // [128 rows][64 k] bf16, 128-byte swizzle
  static constexpr int W_BYTES = BN * 128;   // [64 k][BN] as BN/64 boxes of 8 KB, or [BN][64 k]
  static constexpr int STAGE = A_BYTES + W_BYTES;
  static constexpr int PSTRIDE = BN + 4;     // floats per row of a parked partial
  static constexpr int NBAR = 2 * kNS + 1;   // full[NS] | empty[NS] | acc
  static constexpr int MISC = NBAR * 8 + 16;  // barriers, TMEM slot, abort flag
  static constexpr int SMEM_MAX = kNS * STAGE + MISC + 1024;
  static_assert(kBM * PSTRIDE * 4 <= kNS * STAGE, "partials fit in the ring");
  // ring bytes of a launch: its stages, and at least the parked rows
  static int ring_bytes(int ns, int mrows, int ks) {
    const int r = ns * STAGE, pk = ks > 1 ? mrows * PSTRIDE * 4 : 0;
    return ((r > pk ? r : pk) + 1023) / 1024 * 1024;
  }
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
  const int ns = p.ns;
  uint64_t* full = reinterpret_cast<uint64_t*>(base + p.ring_bytes);
  uint64_t* empty = full + kNS;
  uint64_t* acc_bar = empty + kNS;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(base + p.ring_bytes + C::NBAR * 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + p.ring_bytes + C::NBAR * 8 + 4);

  if (threadIdx.x == 0) {
    griddep_launch();  // the next kernel may start its own prologue
    for (int s = 0; s < ns; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.wmap)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.amap)) : "memory");
  }
  if (warp == 1) tc::alloc(tslot, BN);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = *tslot;

  // chunk i of this split into stage i % NS (thread 0): weights and the A tile,
  // both completing full[st]
  auto load_w = [&](int i) {
    const int st = i % ns;
    uint8_t* wb = base + st * C::STAGE + C::A_BYTES;
    const int k = (c0 + i) * 64;
    mbar_arrive_expect_tx(&full[st], C::W_BYTES + C::A_BYTES);
    if (p.b_kmajor) {
      tma_load_2d(wb, &p.wmap, k + p.w_boff * bz, n0, &full[st]);
    } else {
#pragma unroll
      for (int j = 0; j < BN / 64; ++j) tma_load_2d(wb + j * 8192, &p.wmap, n0 + j * 64 + p.w_boff * bz, k, &full[st]);
    }
  };
  auto load_a = [&](int i) {
    if (p.a_bmajor) tc::tma_load_3d(base + (i % ns) * C::STAGE, &p.amap, (c0 + i) * 64, bz, m0, &full[i % ns]);
    else tc::tma_load_3d(base + (i % ns) * C::STAGE, &p.amap, (c0 + i) * 64, m0, bz, &full[i % ns]);
  };
  int issued = 0;
  if (threadIdx.x == 0)
    for (; issued < min(ns, nch); ++issued) load_w(issued);  // weights do not depend on the previous kernel
  // everything below may read the previous kernel's outputs or write this
  // kernel's
  griddep_wait();

  bool ok = true;
  if (threadIdx.x == 0) {
    // ------------------------------------------------------------ copies
    for (int i = 0; i < issued; ++i) load_a(i);
    for (int i = issued; i < nch; ++i) {
      const int st = i % ns;
      if (!mbar_wait_bounded(&empty[st], ((i / ns) - 1) & 1, abort_flag)) {
        ok = false;
        break;
      }
      load_w(i);
      load_a(i);
      ++issued;
    }
    if (!ok) {
      record_error(p.err, kDevErrWaitEmpty);
      *abort_flag = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // The whole warp runs the loop (warp-uniform control flow and
    // descriptors); one elected lane issues the MMAs and commits.
    const bool leader = tc::elect_one();
    const uint32_t idesc = tc::idesc_bf16(128, BN, 0, p.b_kmajor ? 0 : 1);
    for (int i = 0; i < nch; ++i) {
      const int st = i % ns;
      ok = __all_sync(0xffffffffu, mbar_wait_bounded(&full[st], (i / ns) & 1, abort_flag));
      if (!ok) break;
      tc::fence_after();
      const uint32_t aa = smem_u32(base + st * C::STAGE);
      const uint32_t wa = aa + C::A_BYTES;
      uint64_t ad[4], bd[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        ad[k] = tc::sdesc_sw128(aa + k * 32, 16, 1024);
        bd[k] = p.b_kmajor ? tc::sdesc_sw128(wa + k * 32, 16, 1024) : tc::sdesc_sw128(wa + k * 2048, 8192, 1024);
      }
      if (leader) {
#pragma unroll
        for (int k = 0; k < 4; ++k) tc::mma_bf16(tmem, ad[k], bd[k], idesc, (i > 0 || k > 0) ? 1u : 0u);
        tc::commit(&empty[st]);
      }
      __syncwarp();
    }
    if (!ok) {
      if (leader) record_error(p.err, kDevErrWaitFull);
      *abort_flag = 1;
    }
    if (leader) tc::commit(acc_bar);  // arrives once every MMA issued above has completed
  }
  __syncwarp();

  // ---- epilogue: warp w reads the accumulator rows 32w.. (TMEM lanes 32w..)
  float* part = reinterpret_cast<float*>(base);  // the ring, free once every MMA completed
  const int r = 32 * warp + lane;
  if (32 * warp < mrows) {
    const bool done = mbar_wait_bounded(acc_bar, 0, nullptr);
    if (!done && lane == 0) record_error(p.err, kDevErrWaitMma);
    tc::fence_after();
#pragma unroll 1
    for (int cb = 0; cb < BN / 32; ++cb) {
      uint32_t u[32];
      ld_tmem_32x32b_x32(tmem + ((uint32_t)(32 * warp) << 16) + (uint32_t)(cb * 32), u);
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
  }
  tc::fence_before();
  if (ks > 1) {
    tc::cluster_sync();  // every split's partial rows are parked
    // rank s adds the partials of rows [s * rp, (s + 1) * rp) in rank order
    const int rp = (mrows + ks - 1) / ks;
    const int r0 = rank * rp, r1 = min(mrows, r0 + rp);
    constexpr int G4 = BN / 4;
    for (int it = threadIdx.x; it < (r1 - r0) * G4; it += kThreads) {
      const int rr = r0 + it / G4, c = (it % G4) * 4;
      if (n0 + c >= p.N) continue;
      const uint32_t la = smem_u32(part + rr * C::PSTRIDE + c);
      float4 pv[kMaxCluster];  // every split's partial is requested before the sum
#pragma unroll
      for (int t = 0; t < kMaxCluster; ++t)
        pv[t] = t < ks ? ld_dsmem_f32x4(tc::dsmem_addr(la, (uint32_t)t)) : make_float4(0.f, 0.f, 0.f, 0.f);
      float4 s4 = pv[0];
#pragma unroll
      for (int t = 1; t < kMaxCluster; ++t) {
        if (t >= ks) break;
        s4.x += pv[t].x;
        s4.y += pv[t].y;
        s4.z += pv[t].z;
        s4.w += pv[t].w;
      }
      float v[4] = {s4.x, s4.y, s4.z, s4.w};
      epilogue<4>(p, bz, m0 + rr, n0 + c, v);
    }
    tc::cluster_sync();  // no CTA leaves while a peer may still read its partials
  } else {
    __syncthreads();
  }
  if (warp == 1) {
    tc::fence_after();
    tc::dealloc(tmem, BN);
  }
  if (threadIdx.x == 0 && !ok) {
    // copies already requested land before the CTA exits (bounded)
    for (int i = 0; i < issued; ++i) mbar_wait_bounded(&full[i % ns], (i / ns) & 1, nullptr);
  }
}

// h = LayerNorm(x) * g + b in fp32 (mean, then the biased variance of the
// centred values), rounded to bf16. x [n][d] fp32, d a multiple of 4.
__global__ void __launch_bounds__(kLnThreads) layernorm_kernel(const float* __restrict__ x, int n, int d,
                                                                const float* __restrict__ g,
                                                                const float* __restrict__ b, float eps,
                                                                uint16_t* __restrict__ h) {
  if (threadIdx.x == 0) griddep_launch();
  griddep_wait();
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * (kLnThreads / 32) + (threadIdx.x >> 5);
  if (row >= n) return;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)row * d);
  const int c4 = d / 4;
  float s = 0.f;
  for (int c = lane; c < c4; c += 32) {
    const float4 v = xr[c];
    s += (v.x + v.y) + (v.z + v.w);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  const float mean = s / (float)d;
  float q = 0.f;
  for (int c = lane; c < c4; c += 32) {
    const float4 v = xr[c];
    const float a = v.x - mean, bb = v.y - mean, cc = v.z - mean, dd = v.w - mean;
    q += (a * a + bb * bb) + (cc * cc + dd * dd);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  const float rstd = rsqrtf(q / (float)d + eps);
  const float4* g4 = reinterpret_cast<const float4*>(g);
  const float4* b4 = reinterpret_cast<const float4*>(b);
  uint2* hr = reinterpret_cast<uint2*>(h + (size_t)row * d);
  for (int c = lane; c < c4; c += 32) {
    const float4 v = xr[c], gg = g4[c], bv = b4[c];
    uint2 o;
    o.x = pack_bf16x2((v.x - mean) * rstd * gg.x + bv.x, (v.y - mean) * rstd * gg.y + bv.y);
    o.y = pack_bf16x2((v.z - mean) * rstd * gg.z + bv.z, (v.w - mean) * rstd * gg.w + bv.w);
    hr[c] = o;
  }
}

}  // namespace

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("SMEM_PDL");
    return !(v && v[0] == '0');
  }();
  return on;
}

namespace {

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
  cudaError_t e = ensure_smem_limit<100 + BN>(gemm_kernel<BN>, C::SMEM_MAX);
  if (e != cudaSuccess) return e;
  const int per_cta = (p.chunks + p.ks - 1) / p.ks;  // K chunks of the longest split
  p.ns = per_cta < kNS ? (per_cta > 1 ? per_cta : 1) : kNS;
  p.ring_bytes = C::ring_bytes(p.ns, p.M < kBM ? p.M : kBM, p.ks);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(tiles_n * p.ks), (unsigned)mtiles, (unsigned)batch);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = (size_t)p.ring_bytes + C::MISC + 1024;
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
  if (pdl && pdl_enabled()) {
    at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = at;
  cfg.numAttrs = (unsigned)na;
  return cudaLaunchKernelEx(&cfg, gemm_kernel<BN>, p);
}

}  // namespace

// Clusters of `ks` CTAs of the BN = 64 / 128 kernel that the current device
// holds at once (a GPC hosts only whole clusters), per device, looked up once.
namespace {
int max_active_clusters(int bn, int ks) {
  constexpr int kMaxDev = 16;
  static int table[kMaxDev][2][kMaxCluster + 1] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return 0;
  int& v = table[dev][bn == 128 ? 1 : 0][ks];
  if (v) return v;
  const void* fn = bn == 128 ? reinterpret_cast<const void*>(gemm_kernel<128>)
                             : reinterpret_cast<const void*>(gemm_kernel<64>);
  const int smem = bn == 128 ? Gm<128>::SMEM_MAX : Gm<64>::SMEM_MAX;
  cudaError_t e = bn == 128 ? ensure_smem_limit<228>(gemm_kernel<128>, smem) : ensure_smem_limit<164>(gemm_kernel<64>, smem);
  if (e != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(ks * 64));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = (unsigned)ks;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = 1;
  }
  v = n;
  return n;
}
}  // namespace

// Tile and split plan of a projection: over BN in {128, 64} and clusters of
// 1..8 CTAs (at least one 64-column K chunk per CTA), the most CTAs whose
// clusters the device holds in one wave; ties keep the wider tile. A
// function of the shape and the device only.
GemmPlan gemm_plan(int M, int N, int K, int batch, int num_sms) {
  (void)num_sms;
  const int chunks = (K + 63) / 64;
  const int mtiles = (M + kBM - 1) / kBM;
  GemmPlan best{128, 1, 0};
  for (int bn : {128, 64}) {
    if (bn == 128 && N <= 64) continue;  // a 64-wide output needs no 128 tile
    const int tiles = (N + bn - 1) / bn * mtiles * batch;
    for (int ks = 1; ks <= std::min(kMaxCluster, chunks); ++ks) {
      if (ks > 1 && tiles > max_active_clusters(bn, ks)) break;  // a second wave of clusters
      if (ks == 1 && tiles > max_active_clusters(bn, 1) && best.ctas > 0) break;
      const int ctas = tiles * ks;
      if (ctas > best.ctas) best = GemmPlan{bn, ks, ctas};
    }
  }
  return best;
}

namespace {
// Tensor maps of recently used operands (bf16, 128-byte swizzle), keyed by
// address, rank, extents, strides and box: a layer call reuses every layer's
// weights and the same workspace buffers on every call.
bool cached_map(CUtensorMap* out, const void* ptr, int rank, const uint64_t* dims, const uint64_t* strides,
                const uint32_t* box) {
  struct Entry {
    const void* ptr;
    int rank;
    uint64_t dims[3], strides[2];
    uint32_t box[3];
    CUtensorMap map;
  };
  constexpr int kEntries = 96;
  static thread_local Entry cache[kEntries];
  static thread_local int used = 0, next = 0;
  for (int i = 0; i < used; ++i) {
    const Entry& e = cache[i];
    bool same = e.ptr == ptr && e.rank == rank;
    for (int k = 0; same && k < rank; ++k) same = e.dims[k] == dims[k] && e.box[k] == box[k];
    for (int k = 0; same && k + 1 < rank; ++k) same = e.strides[k] == strides[k];
    if (same) {
      *out = e.map;
      return true;
    }
  }
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc) return false;
  Entry& e = cache[next];
  cuuint64_t d[3], st[2];
  cuuint32_t bx[3], es[3] = {1, 1, 1};
  for (int k = 0; k < rank; ++k) {
    d[k] = dims[k];
    bx[k] = box[k];
  }
  for (int k = 0; k + 1 < rank; ++k) st[k] = strides[k];
  if (enc(&e.map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(ptr), d, st, bx, es,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  e.ptr = ptr;
  e.rank = rank;
  for (int k = 0; k < 3; ++k) {
    e.dims[k] = k < rank ? dims[k] : 0;
    e.box[k] = k < rank ? box[k] : 0;
  }
  for (int k = 0; k < 2; ++k) e.strides[k] = k + 1 < rank ? strides[k] : 0;
  *out = e.map;
  next = (next + 1) % kEntries;
  if (used < kEntries) ++used;
  return true;
}
}  // namespace

cudaError_t launch_layernorm(const float* x, int n, int d, const float* g, const float* b, uint16_t* h, bool pdl,
                             cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)((n + kLnThreads / 32 - 1) / (kLnThreads / 32)));
  cfg.blockDim = dim3(kLnThreads);
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = pdl && pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, layernorm_kernel, x, n, d, g, b, kLayerNormEps, h);
}

cudaError_t launch_gemm(const GemmCall& g, int num_sms, cudaStream_t st) {
  if (g.M <= 0 || g.N <= 0 || g.batch <= 0) return cudaSuccess;
  if (g.N % 32 || g.K % 32 || g.K <= 0) return cudaErrorInvalidValue;
  if (!encode_fn()) return cudaErrorNotSupported;
  const GemmPlan pl = gemm_plan(g.M, g.N, g.K, g.batch, num_sms);
  static thread_local GemmParams p;
  p = GemmParams{};
  const int boxy = g.b_kmajor ? pl.bn : 64;
  {
    const uint64_t dims[3] = {(uint64_t)g.w_cols, (uint64_t)g.w_rows, 1};
    const uint64_t strides[2] = {(uint64_t)g.ldw * 2, (uint64_t)g.ldw * 2 * g.w_rows};
    const uint32_t box[3] = {64u, (uint32_t)boxy, 1u};
    if (!cached_map(&p.wmap, g.w, 2, dims, strides, box)) return cudaErrorInvalidValue;
  }
  // activations: a [batch][M][K] view, or [M][batch][K] when the batch
  // stride is the smaller one (strides increase outward either way); rows
  // and columns past M and K read as zero
  {
    const long long bs = g.batch > 1 ? g.a_bs : (long long)g.lda * g.M;
    p.a_bmajor = g.batch > 1 && bs < g.lda ? 1 : 0;
    const uint64_t dims[3] = {(uint64_t)g.K, (uint64_t)(p.a_bmajor ? g.batch : g.M),
                              (uint64_t)(p.a_bmajor ? g.M : g.batch)};
    const uint64_t strides[2] = {(uint64_t)(p.a_bmajor ? bs : g.lda) * 2, (uint64_t)(p.a_bmajor ? g.lda : bs) * 2};
    const uint32_t box[3] = {64u, p.a_bmajor ? 1u : (uint32_t)kBM, p.a_bmajor ? (uint32_t)kBM : 1u};
    if (!cached_map(&p.amap, g.a, 3, dims, strides, box)) return cudaErrorInvalidValue;
  }
  p.out = g.out;
  p.rope_tab = g.rope_tab;
  p.ib = g.ib;
  p.o_bs = g.o_bs;
  p.group_stride = g.group_stride;
  p.ldo = g.ldo;
  p.M = g.M;
  p.N = g.N;
  p.K = g.K;
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
  p.err = g.err;
  const int tiles_n = (g.N + pl.bn - 1) / pl.bn;
  const int mtiles = (g.M + kBM - 1) / kBM;
  return pl.bn == 128 ? launch_bn<128>(p, tiles_n, mtiles, g.batch, g.pdl, st)
                      : launch_bn<64>(p, tiles_n, mtiles, g.batch, g.pdl, st);
}

}  // namespace smem
