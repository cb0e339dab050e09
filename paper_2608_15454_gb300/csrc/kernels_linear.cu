// Linear layers of the byte modules, the LM module and the multi-byte head:
// y = epilogue(RMSNorm?(x) . W^T) for the pre-norm Llama blocks (Section 4.2).
//
// Two kernels:
//  * k_gemv: the decode path (a few rows). Weight-streaming: every weight element is
//    read from HBM once per launch with 16-byte non-allocating loads; activations are
//    staged in shared memory and reused by the 4 output columns each warp owns. Small N
//    is split along K across CTAs; the last CTA of a column tile sums the partials in a
//    fixed order (deterministic, no atomics on data).
//  * k_gemm: a persistent tiled FFMA GEMM for many rows (prefill, large batches).
#include <cooperative_groups.h>

#include <cstdio>

#include "common.cuh"
#include "epilogue.cuh"

namespace lca {

namespace {

constexpr int kMC = 8;  // rows per chunk (GEMV)
constexpr int kCPW = 4; // output columns per warp (GEMV)
constexpr int kWarps = 4;
constexpr int kColsPerCta = kWarps * kCPW;

__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ void unpack_bf16x2(uint32_t u, float& a, float& b) {
  a = __uint_as_float(u << 16);
  b = __uint_as_float(u & 0xFFFF0000u);
}

// 8 consecutive weights as fp32.
__device__ __forceinline__ void load_w8(const __nv_bfloat16* p, float (&w)[8]) {
  uint4 u = ldg_stream(p);
  unpack_bf16x2(u.x, w[0], w[1]);
  unpack_bf16x2(u.y, w[2], w[3]);
  unpack_bf16x2(u.z, w[4], w[5]);
  unpack_bf16x2(u.w, w[6], w[7]);
}
__device__ __forceinline__ void load_w8(const float* p, float (&w)[8]) {
  uint4 a = ldg_stream(p), b = ldg_stream(p + 4);
  w[0] = __uint_as_float(a.x); w[1] = __uint_as_float(a.y);
  w[2] = __uint_as_float(a.z); w[3] = __uint_as_float(a.w);
  w[4] = __uint_as_float(b.x); w[5] = __uint_as_float(b.y);
  w[6] = __uint_as_float(b.z); w[7] = __uint_as_float(b.w);
}

// D += A.B on the tensor cores: m16n8k16, bf16 operands, fp32 accumulation.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Reduce-scatter of 32 per-lane partial sums: afterwards lane L holds the warp total of
// value index L (row L / kCPW, column L % kCPW). 31 shuffles.
__device__ __forceinline__ float warp_reduce_scatter32(float (&v)[32], int lane) {
#pragma unroll
  for (int off = 16, half = 16; off >= 1; off >>= 1, half >>= 1) {
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int j = 0; j < half; ++j) {
      const float send = up ? v[j] : v[j + half];
      const float keep = up ? v[j + half] : v[j];
      v[j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
    }
  }
  return v[0];
}

template <typename TW>
struct WTraits;
template <>
struct WTraits<__nv_bfloat16> {
  static constexpr int VEC = 1;  // 16-byte vectors per 8 weights
};
template <>
struct WTraits<float> {
  static constexpr int VEC = 2;
};

__device__ __forceinline__ void unpack8(const uint4 (&u)[1], float (&w)[8]) {
  unpack_bf16x2(u[0].x, w[0], w[1]);
  unpack_bf16x2(u[0].y, w[2], w[3]);
  unpack_bf16x2(u[0].z, w[4], w[5]);
  unpack_bf16x2(u[0].w, w[6], w[7]);
}
__device__ __forceinline__ void unpack8(const uint4 (&u)[2], float (&w)[8]) {
  w[0] = __uint_as_float(u[0].x); w[1] = __uint_as_float(u[0].y);
  w[2] = __uint_as_float(u[0].z); w[3] = __uint_as_float(u[0].w);
  w[4] = __uint_as_float(u[1].x); w[5] = __uint_as_float(u[1].y);
  w[6] = __uint_as_float(u[1].z); w[7] = __uint_as_float(u[1].w);
}

// Skinny linear layer. The CTA owns 16 output columns (4 per warp) and a K-range; lanes stride
// K by 8 elements. With KIT > 0 every weight the warp needs (KIT x 4 columns x 16 bytes per lane)
// is loaded into registers before the grid-dependency wait, so the weight stream of this layer
// overlaps the tail of the previous kernels; activations are staged in shared memory afterwards.
template <typename TW, bool NORM, int KIT>
__global__ void __launch_bounds__(kWarps * 32)
k_gemv(LinearArgs a, int ksplit, float* __restrict__ part, int* __restrict__ cnt) {
  TraceScope _trace(TT_GEMV_F32);
  constexpr int VEC = WTraits<TW>::VEC;
  extern __shared__ float smem[];
  const int Kr = a.Kd / ksplit;
  float* xs = smem;              // [kMC][Kr]
  float* inv = smem + kMC * Kr;  // [kMC]
  __shared__ int s_last;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x;
  const int split = blockIdx.y;
  const int grp = blockIdx.z;
  const int k0 = split * Kr;
  const int col0 = tile * kColsPerCta + warp * kCPW;
  const bool colok = col0 < a.N;
  const TW* W = reinterpret_cast<const TW*>(a.W) + (size_t)grp * a.N * a.Kd;

  uint4 wr[KIT > 0 ? KIT : 1][kCPW][VEC];
  if (KIT > 0 && colok) {
#pragma unroll
    for (int it = 0; it < (KIT > 0 ? KIT : 1); ++it) {
      const int kk = lane * 8 + it * 256;
      if (kk < Kr) {
#pragma unroll
        for (int c = 0; c < kCPW; ++c) {
          const uint4* p = reinterpret_cast<const uint4*>(W + (size_t)(col0 + c) * a.Kd + k0 + kk);
#pragma unroll
          for (int v = 0; v < VEC; ++v) wr[it][c][v] = ldg_stream(p + v);
        }
      }
    }
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();

  const int rbase = grp * a.Mg_stride;
  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  if (M < 0) M = 0;

  for (int r0 = 0; r0 < M; r0 += kMC) {
    const int mc = min(kMC, M - r0);
    __syncthreads();
    if (NORM) {
      for (int i = warp; i < mc; i += kWarps) {
        const float* xr = a.x + (size_t)(rbase + r0 + i) * a.ldx;
        float ss = 0.f;
        for (int k = lane * 4; k < a.Kd; k += 128) {
          const float4 v = *reinterpret_cast<const float4*>(xr + k);
          ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) inv[i] = rsqrtf(ss / (float)a.Kd + a.eps);
      }
      __syncthreads();
    }
    // stage the K-range of the chunk's rows (rows >= mc are zero)
    const int n4 = kMC * Kr / 4;
    for (int idx = tid; idx < n4; idx += kWarps * 32) {
      const int i = (idx * 4) / Kr;
      const int kk = idx * 4 - i * Kr;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (i < mc) {
        v = *reinterpret_cast<const float4*>(a.x + (size_t)(rbase + r0 + i) * a.ldx + k0 + kk);
        if (NORM) {
          const float sc = inv[i];
          const float4 g = *reinterpret_cast<const float4*>(a.norm + k0 + kk);
          v.x *= sc * g.x; v.y *= sc * g.y; v.z *= sc * g.z; v.w *= sc * g.w;
        }
      }
      *reinterpret_cast<float4*>(xs + i * Kr + kk) = v;
    }
    __syncthreads();

    if (colok) {
      float acc[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[j] = 0.f;
      if (KIT > 0) {
#pragma unroll
        for (int it = 0; it < (KIT > 0 ? KIT : 1); ++it) {
          const int kk = lane * 8 + it * 256;
          if (kk < Kr) {
            float w[kCPW][8];
#pragma unroll
            for (int c = 0; c < kCPW; ++c) unpack8(wr[it][c], w[c]);
#pragma unroll
            for (int i = 0; i < kMC; ++i) {
              if (i < mc) {
                const float4 xa = *reinterpret_cast<const float4*>(xs + i * Kr + kk);
                const float4 xb = *reinterpret_cast<const float4*>(xs + i * Kr + kk + 4);
#pragma unroll
                for (int c = 0; c < kCPW; ++c) {
                  float sacc = acc[i * kCPW + c];
                  sacc = fmaf(w[c][0], xa.x, sacc); sacc = fmaf(w[c][1], xa.y, sacc);
                  sacc = fmaf(w[c][2], xa.z, sacc); sacc = fmaf(w[c][3], xa.w, sacc);
                  sacc = fmaf(w[c][4], xb.x, sacc); sacc = fmaf(w[c][5], xb.y, sacc);
                  sacc = fmaf(w[c][6], xb.z, sacc); sacc = fmaf(w[c][7], xb.w, sacc);
                  acc[i * kCPW + c] = sacc;
                }
              }
            }
          }
        }
      } else {
        for (int kk = lane * 8; kk < Kr; kk += 256) {
          float w[kCPW][8];
#pragma unroll
          for (int c = 0; c < kCPW; ++c) load_w8(W + (size_t)(col0 + c) * a.Kd + k0 + kk, w[c]);
#pragma unroll
          for (int i = 0; i < kMC; ++i) {
            if (i < mc) {
              const float4 xa = *reinterpret_cast<const float4*>(xs + i * Kr + kk);
              const float4 xb = *reinterpret_cast<const float4*>(xs + i * Kr + kk + 4);
#pragma unroll
              for (int c = 0; c < kCPW; ++c) {
                float sacc = acc[i * kCPW + c];
                sacc = fmaf(w[c][0], xa.x, sacc); sacc = fmaf(w[c][1], xa.y, sacc);
                sacc = fmaf(w[c][2], xa.z, sacc); sacc = fmaf(w[c][3], xa.w, sacc);
                sacc = fmaf(w[c][4], xb.x, sacc); sacc = fmaf(w[c][5], xb.y, sacc);
                sacc = fmaf(w[c][6], xb.z, sacc); sacc = fmaf(w[c][7], xb.w, sacc);
                acc[i * kCPW + c] = sacc;
              }
            }
          }
        }
      }
      const float v = warp_reduce_scatter32(acc, lane);
      const int i = lane / kCPW, c = lane % kCPW;
      const float vn = __shfl_down_sync(0xffffffffu, v, 1);
      if (ksplit == 1) {
        if (i < mc && (c & 1) == 0)
          epi_pair<TW>(a.epi, rbase + r0 + i, col0 + c, v, vn);
      } else if (i < mc) {
        part[((size_t)split * a.M_cap + r0 + i) * a.N + col0 + c] = v;
      }
    }
  }

  if (ksplit == 1) return;
  // split-K: the last CTA of this column tile reduces the partials in split order
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(cnt + tile, 1) == ksplit - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int pairs = kColsPerCta / 2;
  for (int idx = tid; idx < M * pairs; idx += kWarps * 32) {
    const int r = idx / pairs;
    const int c = tile * kColsPerCta + (idx - r * pairs) * 2;
    if (c >= a.N) continue;
    float s0 = 0.f, s1 = 0.f;
    for (int sp = 0; sp < ksplit; ++sp) {
      const float* pp = part + ((size_t)sp * a.M_cap + r) * a.N + c;
      s0 += __ldcg(pp);
      s1 += __ldcg(pp + 1);
    }
    epi_pair<TW>(a.epi, rbase + r, c, s0, s1);
  }
  if (tid == 0) cnt[tile] = 0;
}

// ---------------------------------------------------------------- bulk-copy weight-streaming GEMV
// Skinny linear layer for bf16 weights: the weights of each CTA's tile arrive in shared memory by
// bulk async copies (cp.async.bulk) completing on an mbarrier, issued before the grid-dependency
// wait so that they stream while the previous kernel finishes. Every wait is bounded.
constexpr int kWaitSpins = 1 << 22;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait: false if the phase did not complete within the spin budget.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int spins = kWaitSpins) {
  for (int i = 0; i < spins; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

// Spin budget of the first weight wait of k_gemv_bulk. A test hook (lca_debug_set_wait_spins) can
// shorten it so that the wait reports late at once; the second wait, which drains the copies in
// flight before the CTA reads them or leaves, keeps the full budget.
static __device__ int g_first_wait_spins = kWaitSpins;

// Each CTA prefetches an equal slice of the next layers' weights into L2 (no shared memory or
// registers are used, so the HBM stream continues across kernel boundaries).
__device__ __forceinline__ void prefetch_next(const LinearArgs& a) {
  const int nct = gridDim.x * gridDim.y * gridDim.z;
  const int cta = (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    if (!a.pf[j] || !a.pf_bytes[j]) continue;
    const size_t per = ((a.pf_bytes[j] + nct - 1) / nct + 255) & ~size_t(255);
    const size_t off = per * cta;
    if (off >= a.pf_bytes[j]) continue;
    size_t len = a.pf_bytes[j] - off < per ? a.pf_bytes[j] - off : per;
    const char* p = reinterpret_cast<const char*>(a.pf[j]) + off;
    // one bulk prefetch per 32 KB, issued by the first lanes of warp 0
    for (size_t q = threadIdx.x * 32768; q < len; q += blockDim.x * 32768) {
      const uint32_t n = (uint32_t)((len - q) < 32768 ? (len - q) : 32768) & ~15u;
      if (n) asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p + q), "r"(n) : "memory");
    }
  }
}

// One tile per CTA: NW*4 output columns x Kr inputs (the CTA's K-split), copied into shared
// memory (one bulk async copy per column, rows padded by 16 bytes) before the grid-dependency
// wait; the RMSNorm gain of the K-range is read into shared memory then too. RMSNorm is folded in: rows are staged as
// x * g, split into two bf16 halves (x * g = hi + lo, about 16 significant bits), while their sums
// of squares accumulate, and the per-row inverse RMS scales the dot products. The dot products
// run on the tensor cores (mma m16n8k16: 16 output columns as M, up to 8 rows as N, hi and lo
// against the exact bf16 weights, fp32 accumulation), each warp over every NW-th K-step; the
// warps' partials are summed in shared memory into one (row, column) value per lane, 4 columns
// per warp. Rows are processed in chunks of MCA. With a K-split the `ksplit` CTAs of a column tile form a thread-
// block cluster: each leaves its partial sums in its own shared memory and rank 0 adds the ranks'
// partials through distributed shared memory in rank order (no global scratch).
// (512 threads per SM by registers, four CTAs of four warps, so that a 512-tile launch is resident
// in one wave)
// GS: the rows come pre-split from the producing layer (LinearArgs::gsplit); SP: this layer's
// epilogue also writes its output split for the next layer (EpiArgs::sp_hi). Both are template
// flags so that a launch carries only the code of its own staging and epilogue.
template <int MCA, int NW, bool NORM, bool GS, bool SP>
__global__ void __launch_bounds__(NW * 32, 16 / NW)
k_gemv_bulk(LinearArgs a, int ksplit) {
  TraceScope _trace(TT_GEMV);
  namespace cgr = cooperative_groups;
  constexpr int CT = NW * kCPW;  // columns per CTA
  constexpr int NT = NW * 32;
  extern __shared__ __align__(128) unsigned char sm[];
  const int Kr = a.Kd / ksplit;
  const int KP = Kr + 8;  // padded row (elements): conflict-free fragment loads
  __nv_bfloat16* wt = reinterpret_cast<__nv_bfloat16*>(sm);             // [CT][KP]
  float* gs = reinterpret_cast<float*>(sm + (size_t)CT * KP * 2);        // [Kr] (NORM)
  __nv_bfloat16* xh = reinterpret_cast<__nv_bfloat16*>(gs + Kr);         // [MCA][KP] bf16 high halves
  __nv_bfloat16* xl = xh + (size_t)MCA * KP;                             // [MCA][KP] bf16 low halves
  float* red = reinterpret_cast<float*>(xl + (size_t)MCA * KP);          // [NW][CT][8] warp partials
  float* wss = red + NW * CT * 8;                                        // [NW][MCA] warp sums of squares
  float* rs = wss + NW * MCA;                                            // [MCA] this CTA's sums of squares
  float* tq = rs + MCA;                 // [MCA][CT / 2] split on write: squares per column pair
  float* sgs = tq + MCA * CT / 2;       // [CT] split on write: the consumer's RMSNorm gain
  float* cpart = reinterpret_cast<float*>(                                // [MCA][CT], 16-byte aligned
      (reinterpret_cast<uintptr_t>(sgs + CT) + 15) & ~uintptr_t(15));
  uint64_t* bar = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(cpart + MCA * CT) + 15) & ~uintptr_t(15));
  uint64_t* rbar = bar + 1;                                              // reduction arrivals (rank 0)
  uint64_t* xbar = bar + 2;                                              // pre-split rows landed
  float* rbuf = reinterpret_cast<float*>(bar + 3);                       // [kMaxKSplit][MCA][CT] (rank 0)
  float* rsq = rbuf + kMaxKSplit * MCA * CT;                             // [kMaxKSplit][MCA] (rank 0)

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x;
  const int split = blockIdx.y;
  const int grp = blockIdx.z;
  const int k0 = split * Kr;
  const int ncols = min(CT, a.N - tile * CT);
  const __nv_bfloat16* W = reinterpret_cast<const __nv_bfloat16*>(a.W) + (size_t)grp * a.N * a.Kd +
                           (size_t)tile * CT * a.Kd + k0;
  if (tid == 0) {
    mbar_init(bar, 1);
    mbar_init(xbar, 1);
    fence_mbar_init();
    mbar_expect_tx(bar, (uint32_t)(ncols * Kr * 2));
    for (int c = 0; c < ncols; ++c) bulk_g2s(wt + (size_t)c * KP, W + (size_t)c * a.Kd, (uint32_t)(Kr * 2), bar);
  }
  if (NORM && !GS) {
    // the RMSNorm gain of the K-range (a weight: read before the dependency wait)
    for (int i = tid; i < Kr / 4; i += NT)
      reinterpret_cast<float4*>(gs)[i] = __ldg(reinterpret_cast<const float4*>(a.norm + k0) + i);
  }
  // split on write: the next layer's RMSNorm gain at this tile's columns (a weight)
  if (SP && tid < CT) sgs[tid] = (a.epi.sg && tile * CT + tid < a.N) ? __ldg(a.epi.sg + tile * CT + tid) : 1.f;
  prefetch_next(a);
  if (ksplit > 1) {
    // rank 0's reduction barrier exists before any peer can arrive on it (before the dependency
    // wait, so this cluster barrier stays off the critical path)
    if (tid == 0 && split == 0) {
      mbar_init(rbar, (uint32_t)(ksplit - 1));
      fence_mbar_init();
    }
    cgr::this_cluster().sync();
  } else if (NORM) {
    __syncthreads();
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();

  const int rbase = grp * a.Mg_stride;
  // pre-split rows, bf16 halves [rows][Kd]: one bulk copy per row and half into the staging rows;
  // the first chunk's copies go out before the row count is read (rows up to M_cap exist)
  // with a norm, each row's 16-column partial sums of squares (Kd / 16 floats) come along into the
  // gain's staging area, which a pre-split layer does not use (the producer applied the gain)
  const int nb = a.Kd / 16;
  auto gsplit_issue = [&](int r0, int nr) {
    mbar_expect_tx(xbar, (uint32_t)(nr * Kr * 4 + (NORM ? nr * nb * 4 : 0)));
    for (int i = 0; i < nr; ++i) {
      const size_t o = (size_t)(rbase + r0 + i) * a.Kd + k0;
      bulk_g2s(xh + (size_t)i * KP, a.ghi + o, (uint32_t)(Kr * 2), xbar);
      bulk_g2s(xl + (size_t)i * KP, a.glo + o, (uint32_t)(Kr * 2), xbar);
      if (NORM) bulk_g2s(gs + (size_t)i * nb, a.gss + (size_t)(rbase + r0 + i) * a.gss_ld, (uint32_t)(nb * 4), xbar);
    }
  };
  const int nr0 = min(MCA, a.M_cap);
  if (GS && tid == 0 && nr0 > 0) gsplit_issue(0, nr0);
  uint32_t xphase = 0;      // chunks whose pre-split copies were waited for
  bool x_pending = GS && nr0 > 0;
  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  if (M < 0) M = 0;
  const int col0 = warp * kCPW;  // within the tile
  bool have_w = false;
  const int ei = lane / kCPW, ec = lane % kCPW;  // this lane's (row, column) after the reduction

  for (int r0 = 0; r0 < M; r0 += MCA) {
    const int mc = min(MCA, M - r0);
    // epilogue operands of this lane, loaded while the rows are staged and multiplied
    EpiPre pre{};
    const bool epi_lane = ksplit == 1 && col0 < ncols && ei < mc && (ec & 1) == 0;
    if (epi_lane) pre = epi_load_early(a.epi, rbase + r0 + ei, tile * CT + col0 + ec);
    __syncthreads();
    if (tid < MCA * CT / 2) tq[tid] = 0.f;
    if constexpr (GS) {
      // rows split by the producing layer's epilogue: bulk copies (the first chunk's are in flight)
      if (r0 > 0 && tid == 0) gsplit_issue(r0, mc);
      const int nr = r0 == 0 ? nr0 : mc;
      // the bounded wait for the rows; on a timeout the error is recorded and the copies get one
      // more bounded wait
      const bool late = !mbar_wait(xbar, xphase & 1);
      if (late) mbar_wait(xbar, xphase & 1);
      if (late && tid == 0) atomicOr(a.epi.err, kErrTimeout | kErrWaitGemv);
      ++xphase;
      x_pending = false;
      if (NORM) {
        // each row's sum of squares from the staged partial sums (warp i % NW); the cluster's rank 0
        // alone contributes it to the K-split sum
        for (int i = 0; i < MCA; ++i) {
          float t = 0.f;
          if (i % NW == warp) {
            if (i < nr)
              for (int j = lane; j < nb; j += 32) t += gs[(size_t)i * nb + j];
#pragma unroll
            for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
          }
          if (lane == 0) wss[warp * MCA + i] = (i % NW == warp && split == 0) ? t : 0.f;
        }
      }
    } else {
    // raw rows -> registers (loads batched), then x * g -> shared memory with sums of squares
    constexpr int UNR = 8;
    const int nv = MCA * Kr / 4;
    float ss[MCA];
#pragma unroll
    for (int i = 0; i < MCA; ++i) ss[i] = 0.f;
    for (int base = tid; base < nv; base += NT * UNR) {
      float4 v[UNR];
#pragma unroll
      for (int u = 0; u < UNR; ++u) {
        const int idx = base + u * NT;
        const int i = (idx * 4) / Kr, kk = idx * 4 - i * Kr;
        v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (idx < nv && i < mc)
          v[u] = *reinterpret_cast<const float4*>(a.x + (size_t)(rbase + r0 + i) * a.ldx + k0 + kk);
      }
#pragma unroll
      for (int u = 0; u < UNR; ++u) {
        const int idx = base + u * NT;
        if (idx < nv) {
          float4 q = v[u];
          const int i = (idx * 4) / Kr, kk = idx * 4 - i * Kr;
          if (NORM) {
#pragma unroll
            for (int r = 0; r < MCA; ++r)
              if (r == i) ss[r] += q.x * q.x + q.y * q.y + q.z * q.z + q.w * q.w;
            const float4 g = *reinterpret_cast<const float4*>(gs + kk);
            q.x *= g.x; q.y *= g.y; q.z *= g.z; q.w *= g.w;
          }
          // x * g = hi + lo in bf16
          const __nv_bfloat162 h01 = __floats2bfloat162_rn(q.x, q.y), h23 = __floats2bfloat162_rn(q.z, q.w);
          const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
          const __nv_bfloat162 l01 = __floats2bfloat162_rn(q.x - f01.x, q.y - f01.y);
          const __nv_bfloat162 l23 = __floats2bfloat162_rn(q.z - f23.x, q.w - f23.y);
          *reinterpret_cast<uint2*>(xh + (size_t)i * KP + kk) =
              make_uint2(*reinterpret_cast<const uint32_t*>(&h01), *reinterpret_cast<const uint32_t*>(&h23));
          *reinterpret_cast<uint2*>(xl + (size_t)i * KP + kk) =
              make_uint2(*reinterpret_cast<const uint32_t*>(&l01), *reinterpret_cast<const uint32_t*>(&l23));
        }
      }
    }
    if (NORM) {
      // per-warp partial sums of squares over this CTA's K range (no atomics: summed in warp order)
#pragma unroll
      for (int i = 0; i < MCA; ++i) {
        float t = ss[i];
#pragma unroll
        for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) wss[warp * MCA + i] = t;
      }
    }
    }
    if (r0 == 0) _trace.mark(0);  // first row chunk loaded and staged
    if (epi_lane) epi_load_late(a.epi, pre, tile * CT + col0 + ec);  // overlaps the dot products
    if (!have_w) {
      // the bounded wait for the weight tile; on a timeout the error is recorded, the copies in
      // flight get one more bounded wait, and the kernel runs on (no early exit, so cluster
      // barriers stay matched)
      const bool late = !mbar_wait(bar, 0, g_first_wait_spins);
      if (late) mbar_wait(bar, 0);
      if (__syncthreads_or(late) && tid == 0) atomicOr(a.epi.err, kErrTimeout | kErrWaitGemv);
      have_w = true;
    } else {
      __syncthreads();
    }
    if (r0 == 0) _trace.mark(1);  // weights in shared memory
    if (NORM && tid < MCA) {
      // this CTA's share of each row's sum of squares; read after the next barrier
      float t = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) t += wss[w * MCA + tid];
      rs[tid] = t;
    }
    {
      // tensor-core dot products: warp w takes K-steps w, w + NW, ...; C[column][row] partials
      constexpr int MT = CT / 16;
      const int g = lane >> 2, q4 = lane & 3;
      // the high and low halves' products accumulate separately (two independent MMA chains)
      float cacc[MT][4], cacl[MT][4];
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        cacc[mt][0] = cacc[mt][1] = cacc[mt][2] = cacc[mt][3] = 0.f;
        cacl[mt][0] = cacl[mt][1] = cacl[mt][2] = cacl[mt][3] = 0.f;
      }
      const bool brow = g < mc;
      for (int kb = warp * 16; kb < Kr; kb += NW * 16) {
        uint32_t bh0 = 0u, bh1 = 0u, bl0 = 0u, bl1 = 0u;
        if (brow) {
          const uint32_t* ph = reinterpret_cast<const uint32_t*>(xh + (size_t)g * KP + kb + 2 * q4);
          const uint32_t* pl = reinterpret_cast<const uint32_t*>(xl + (size_t)g * KP + kb + 2 * q4);
          bh0 = ph[0];
          bh1 = ph[4];
          bl0 = pl[0];
          bl1 = pl[4];
        }
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          const uint32_t* pa = reinterpret_cast<const uint32_t*>(wt + (size_t)(mt * 16 + g) * KP + kb + 2 * q4);
          uint32_t af[4];
          af[0] = pa[0];
          af[1] = pa[4 * KP];
          af[2] = pa[4];
          af[3] = pa[4 * KP + 4];
          mma_bf16_16816(cacc[mt], af, bh0, bh1);
          mma_bf16_16816(cacl[mt], af, bl0, bl1);
        }
      }
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
        for (int e = 0; e < 4; ++e) cacc[mt][e] += cacl[mt][e];
        const int f = mt * 16 + g;
        *reinterpret_cast<float2*>(red + ((size_t)(warp * CT + f) * 8 + 2 * q4)) = make_float2(cacc[mt][0], cacc[mt][1]);
        *reinterpret_cast<float2*>(red + ((size_t)(warp * CT + f + 8) * 8 + 2 * q4)) =
            make_float2(cacc[mt][2], cacc[mt][3]);
      }
    }
    __syncthreads();
    if (col0 < ncols) {
      // lane (row ei, column col0 + ec): the sum of the warps' partials
      float v = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) v += red[(w * CT + col0 + ec) * 8 + ei];
      if (r0 == 0) _trace.mark(2);  // first chunk's dot products summed
      if (ksplit == 1) {
        if (NORM && ei < mc) {
          float t = 0.f;
#pragma unroll
          for (int w = 0; w < NW; ++w) t += wss[w * MCA + ei];
          v *= rsqrtf(t / (float)a.Kd + a.eps);
        }
        const float vn = __shfl_down_sync(0xffffffffu, v, 1);
        if (epi_lane) {
          const int cl = col0 + ec;
          if (!SP || !a.epi.sp_only) epi_store<__nv_bfloat16>(a.epi, pre, rbase + r0 + ei, tile * CT + cl, v, vn);
          if constexpr (SP) {
            tq[ei * (CT / 2) + (cl >> 1)] =
                epi_split_pair(a.epi, pre, rbase + r0 + ei, tile * CT + cl, v, vn, sgs[cl], sgs[cl + 1]);
          }
        }
      } else if (ei < MCA) {
        cpart[ei * CT + col0 + ec] = v;
      }
    }
    // split on write with a norm: this tile's sums of squares per 16-column block and row, added
    // in column order (the same sums on every run)
    auto write_tss = [&]() {
      __syncthreads();
      if (tid < mc * (CT / 16)) {
        const int i = tid / (CT / 16), sl = tid - i * (CT / 16);
        float t = 0.f;
#pragma unroll
        for (int p = 0; p < 8; ++p) t += tq[i * (CT / 2) + sl * 8 + p];
        a.epi.ss[(size_t)(rbase + r0 + i) * a.epi.ss_ld + tile * (CT / 16) + sl] = t;
      }
    };
    if (SP && ksplit == 1 && a.epi.ss) write_tss();
    if (ksplit > 1 && M <= MCA) {
      // a single row chunk: the peers push their partials into rank 0's shared memory and
      // arrive on its barrier (release, cluster scope), then leave; rank 0 waits, adds the ranks
      // in order and runs the epilogue. No cluster barrier on the critical path.
      cgr::cluster_group cl = cgr::this_cluster();
      __syncthreads();  // this CTA's partials and row sums are complete
      if (split != 0) {
        float* dst = cl.map_shared_rank(rbuf, 0) + split * MCA * CT;
        for (int idx = tid; idx < mc * CT; idx += NT) dst[idx] = cpart[idx];
        if (NORM && tid < mc) cl.map_shared_rank(rsq, 0)[split * MCA + tid] = rs[tid];
        __syncthreads();
        if (tid == 0) {
          uint32_t remote;
          asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(rbar)), "r"(0));
          asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote) : "memory");
        }
      } else {
        EpiPre pp[2];
        int np = 0;
        for (int idx = tid; idx < mc * (CT / 2) && np < 2; idx += NT, ++np) {
          const int i = idx / (CT / 2), c = (idx - i * (CT / 2)) * 2;
          if (c < ncols) pp[np] = epi_load(a.epi, rbase + r0 + i, tile * CT + c);
        }
        if (tid == 0) {
          bool ok = false;
          for (int it = 0; it < kWaitSpins && !ok; ++it) {
            uint32_t done;
            asm volatile(
                "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], 0;\n"
                " selp.u32 %0, 1, 0, p;\n}"
                : "=r"(done)
                : "r"(smem_u32(rbar))
                : "memory");
            ok = done != 0;
          }
          if (!ok) atomicOr(a.epi.err, kErrTimeout | kErrWaitGemvReduce);
        }
        __syncthreads();
        int j = 0;
        for (int idx = tid; idx < mc * (CT / 2); idx += NT, ++j) {
          const int i = idx / (CT / 2), c = (idx - i * (CT / 2)) * 2;
          if (c >= ncols) continue;
          float t0 = cpart[i * CT + c], t1 = cpart[i * CT + c + 1], sq = NORM ? rs[i] : 0.f;
#pragma unroll
          for (int sp = 1; sp < kMaxKSplit; ++sp) {
            if (sp < ksplit) {
              t0 += rbuf[(sp * MCA + i) * CT + c];
              t1 += rbuf[(sp * MCA + i) * CT + c + 1];
              if (NORM) sq += rsq[sp * MCA + i];
            }
          }
          if (NORM) {
            const float sc = rsqrtf(sq / (float)a.Kd + a.eps);
            t0 *= sc;
            t1 *= sc;
          }
          const EpiPre q = j < 2 ? pp[j] : epi_load(a.epi, rbase + r0 + i, tile * CT + c);
          if (!SP || !a.epi.sp_only) epi_store<__nv_bfloat16>(a.epi, q, rbase + r0 + i, tile * CT + c, t0, t1);
          if constexpr (SP) {
            tq[i * (CT / 2) + (c >> 1)] =
                epi_split_pair(a.epi, q, rbase + r0 + i, tile * CT + c, t0, t1, sgs[c], sgs[c + 1]);
          }
        }
        if (SP && a.epi.ss) write_tss();
      }
    } else if (ksplit > 1) {
      // cluster reduction of the K-split partials of this row chunk
      cgr::cluster_group cl = cgr::this_cluster();
      EpiPre pp[2];
      int pi[2], pc[2], np = 0;
      if (split == 0)
        for (int idx = tid; idx < mc * (CT / 2) && np < 2; idx += NT) {
          pi[np] = idx / (CT / 2);
          pc[np] = (idx - pi[np] * (CT / 2)) * 2;
          if (pc[np] < ncols) pp[np] = epi_load(a.epi, rbase + r0 + pi[np], tile * CT + pc[np]);
          ++np;
        }
      cl.sync();
      if (split == 0) {
        int j = 0;
        for (int idx = tid; idx < mc * (CT / 2); idx += NT, ++j) {
          const int i = idx / (CT / 2), c = (idx - i * (CT / 2)) * 2;
          if (c >= ncols) continue;
          // every rank's partials (and row sums of squares) in one batch of remote loads, then
          // added in rank order
          float t0 = 0.f, t1 = 0.f, sq = 0.f;
#pragma unroll
          for (int sp = 0; sp < kMaxKSplit; ++sp) {
            if (sp < ksplit) {
              const float2 pv = *reinterpret_cast<const float2*>(cl.map_shared_rank(cpart + i * CT + c, sp));
              t0 += pv.x;
              t1 += pv.y;
              if (NORM) sq += *cl.map_shared_rank(rs + i, sp);
            }
          }
          if (NORM) {
            const float sc = rsqrtf(sq / (float)a.Kd + a.eps);
            t0 *= sc;
            t1 *= sc;
          }
          const EpiPre q = j < 2 ? pp[j] : epi_load(a.epi, rbase + r0 + i, tile * CT + c);
          if (!SP || !a.epi.sp_only) epi_store<__nv_bfloat16>(a.epi, q, rbase + r0 + i, tile * CT + c, t0, t1);
          if constexpr (SP) {
            tq[i * (CT / 2) + (c >> 1)] =
                epi_split_pair(a.epi, q, rbase + r0 + i, tile * CT + c, t0, t1, sgs[c], sgs[c + 1]);
          }
        }
        if (SP && a.epi.ss) write_tss();
      }
      cl.sync();
    }
  }
  if (!have_w && !mbar_wait(bar, 0)) {  // no rows: still wait (bounded, twice) for the copy before leaving
    if (tid == 0) atomicOr(a.epi.err, kErrTimeout | kErrWaitGemv);
    mbar_wait(bar, 0);
  }
  if (GS && x_pending && !mbar_wait(xbar, 0)) {  // no rows: the first chunk's row copies too
    if (tid == 0) atomicOr(a.epi.err, kErrTimeout | kErrWaitGemv);
    mbar_wait(xbar, 0);
  }
}

// ---------------------------------------------------------------- tiled GEMM (many rows)
constexpr int kBM = 64, kBN = 64, kBK = 32;

__global__ void k_rowstats(const float* __restrict__ x, int ldx, int Kd, const int* Mp, int M_cap,
                           int groups, int Mg_stride, float eps, float* __restrict__ inv) {
  TraceScope _trace(TT_ROWSTATS);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  int M = *Mp;
  M = M < M_cap ? M : M_cap;
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  const int total = groups * M;
  for (int w = warp; w < total; w += (gridDim.x * blockDim.x) >> 5) {
    const int g = w / M, i = w - g * M;
    const int r = g * Mg_stride + i;
    const float* xr = x + (size_t)r * ldx;
    float ss = 0.f;
    for (int k = lane; k < Kd; k += 32) ss += xr[k] * xr[k];
#pragma unroll
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0) inv[r] = rsqrtf(ss / (float)Kd + eps);
  }
}

template <typename TW, bool NORM>
__global__ void __launch_bounds__(256) k_gemm(LinearArgs a, const float* __restrict__ inv) {
  TraceScope _trace(TT_GEMM);
  __shared__ float As[kBK][kBM + 4];
  __shared__ float Bs[kBK][kBN + 4];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int grp = blockIdx.z;
  const TW* W = reinterpret_cast<const TW*>(a.W) + (size_t)grp * a.N * a.Kd;
  const int rbase = grp * a.Mg_stride;
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  if (M <= 0) return;
  const int ntm = (M + kBM - 1) / kBM, ntn = (a.N + kBN - 1) / kBN;
  for (int t = blockIdx.x; t < ntm * ntn; t += gridDim.x) {
    const int mt = t / ntn, nt = t - mt * ntn;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < a.Kd; k0 += kBK) {
      // A: 64 rows x 32 k, two float4 per thread
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int q = tid * 2 + j;
        const int row = q >> 3, kq = (q & 7) * 4;
        const int r = mt * kBM + row;
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (r < M && k0 + kq < a.Kd) {
          v = *reinterpret_cast<const float4*>(a.x + (size_t)(rbase + r) * a.ldx + k0 + kq);
          if (NORM) {
            const float s = inv[rbase + r];
            const float4 g = *reinterpret_cast<const float4*>(a.norm + k0 + kq);
            v.x *= s * g.x; v.y *= s * g.y; v.z *= s * g.z; v.w *= s * g.w;
          }
        }
        As[kq + 0][row] = v.x; As[kq + 1][row] = v.y;
        As[kq + 2][row] = v.z; As[kq + 3][row] = v.w;
      }
      // B: 64 cols x 32 k, 8 weights per thread
      {
        const int col = tid >> 2, kk = (tid & 3) * 8;
        const int cg = nt * kBN + col;
        float w[8];
        if (cg < a.N && k0 + kk < a.Kd) {
          load_w8(W + (size_t)cg * a.Kd + k0 + kk, w);
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) w[e] = 0.f;
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) Bs[kk + e][col] = w[e];
      }
      __syncthreads();
#pragma unroll 8
      for (int kk = 0; kk < kBK; ++kk) {
        const float4 av = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
        const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
        const float ar[4] = {av.x, av.y, av.z, av.w};
        const float br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(ar[i], br[j], acc[i][j]);
      }
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int r = mt * kBM + ty * 4 + i;
      if (r >= M) continue;
#pragma unroll
      for (int j = 0; j < 4; j += 2) {
        const int c = nt * kBN + tx * 4 + j;
        if (c < a.N) epi_pair<TW>(a.epi, rbase + r, c, acc[i][j], acc[i][j + 1]);
      }
    }
  }
}

template <typename TW, bool NORM, int KIT>
void launch_gemv_kit(const Dev& D, const LinearArgs& a, int ksplit, cudaStream_t s) {
  const int Kr = a.Kd / ksplit;
  const size_t smem = (size_t)kMC * Kr * sizeof(float) + kMC * sizeof(float);
  dim3 grid((a.N + kColsPerCta - 1) / kColsPerCta, ksplit, a.groups);
  ++g_launches;
  launch_pdl(k_gemv<TW, NORM, KIT>, grid, dim3(kWarps * 32), smem, s, a, ksplit, D.lin_part, D.lin_cnt);
}

template <int MCA, int NW, bool NORM>
void gemv_bulk_go(const Dev& D, const LinearArgs& a, int ksplit, cudaStream_t s) {
  constexpr int CT = NW * kCPW;
  const int Kr = a.Kd / ksplit;
  const size_t KP = (size_t)Kr + 8;
  const size_t smem = (size_t)CT * KP * 2 + (size_t)Kr * 4 + 2 * (size_t)MCA * KP * 2 + (size_t)NW * CT * 8 * 4 +
                      (NW * MCA + MCA + MCA * CT / 2 + CT + MCA * CT) * 4 + 16 + 16 + 24 +
                      (ksplit > 1 ? (size_t)kMaxKSplit * MCA * (CT + 1) * 4 : 0) + 64;  // rank 0's buffers
  LinearArgs b = a;
  if (b.gsplit) {
    b.ghi = D.as_hi[b.abuf];
    b.glo = D.as_lo[b.abuf];
    b.gss = D.gv_ss;
    b.gss_ld = D.gv_ss_ld;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((a.N + CT - 1) / CT, ksplit, a.groups);
  cfg.blockDim = dim3(NW * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = ksplit;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  const bool sp = b.epi.sp_hi != nullptr;
  if (b.gsplit) {
    if (sp) cudaLaunchKernelEx(&cfg, k_gemv_bulk<MCA, NW, NORM, true, true>, b, ksplit);
    else cudaLaunchKernelEx(&cfg, k_gemv_bulk<MCA, NW, NORM, true, false>, b, ksplit);
  } else {
    if (sp) cudaLaunchKernelEx(&cfg, k_gemv_bulk<MCA, NW, NORM, false, true>, b, ksplit);
    else cudaLaunchKernelEx(&cfg, k_gemv_bulk<MCA, NW, NORM, false, false>, b, ksplit);
  }
}

template <int MCA, bool NORM>
void gemv_bulk_width(const Dev& D, const LinearArgs& a, int ksplit, cudaStream_t s) {
  // wide layers with many rows: 32-column CTAs keep the grid within one wave
  if constexpr (MCA >= 8) {
    if (ksplit == 1 && a.N >= 4096) {
      gemv_bulk_go<MCA, 8, NORM>(D, a, ksplit, s);
      return;
    }
  }
  gemv_bulk_go<MCA, 4, NORM>(D, a, ksplit, s);
}


template <bool NORM>
bool launch_gemv_tma(const Dev& D, const LinearArgs& a, int rows_typ, cudaStream_t s) {
  const int ksplit = gemv_bulk_ksplit(D, a);
  if (!ksplit) return false;
  // activations staged per chunk of the typical row count (shared memory sets CTAs per SM)
  const int mt = rows_typ < a.M_cap ? rows_typ : a.M_cap;
  if (mt <= 1) gemv_bulk_width<1, NORM>(D, a, ksplit, s);
  else if (mt <= 2) gemv_bulk_width<2, NORM>(D, a, ksplit, s);
  else if (mt <= 4) gemv_bulk_width<4, NORM>(D, a, ksplit, s);
  else gemv_bulk_width<8, NORM>(D, a, ksplit, s);
  return true;
}

template <typename TW, bool NORM>
void launch_gemv(const Dev& D, const LinearArgs& a, cudaStream_t s) {
  if (sizeof(TW) == 2 && D.use_tma && launch_gemv_tma<NORM>(D, a, a.rows_typ > 0 ? a.rows_typ : a.M_cap, s))
    return;
  int ksplit = 1;
  if (a.groups == 1 && a.N <= 2048 && D.lin_part) {
    ksplit = a.Kd >= 2048 ? 8 : 4;
    while (ksplit > 1 && ((a.Kd % ksplit) || ((a.Kd / ksplit) % 8) ||
                          (size_t)ksplit * a.M_cap * a.N > D.lin_part_floats))
      ksplit >>= 1;
  }
  const int Kr = a.Kd / ksplit;
  const int kmax = sizeof(TW) == 2 ? 1024 : 512;  // register budget for the hoisted weights
  if (Kr <= 256) launch_gemv_kit<TW, NORM, 1>(D, a, ksplit, s);
  else if (Kr <= 512) launch_gemv_kit<TW, NORM, 2>(D, a, ksplit, s);
  else if (Kr <= kmax) launch_gemv_kit<TW, NORM, 4>(D, a, ksplit, s);
  else launch_gemv_kit<TW, NORM, 0>(D, a, ksplit, s);
}

template <typename TW, bool NORM>
void launch_gemm(const Dev& D, const LinearArgs& a, cudaStream_t s) {
  if (NORM) {
    ++g_launches;
    launch_pdl(k_rowstats, dim3(256), dim3(256), 0, s, a.x, a.ldx, a.Kd, a.M, a.M_cap, a.groups,
               a.Mg_stride, a.eps, D.inv_rms);
  }
  const int ntm = (a.M_cap + kBM - 1) / kBM, ntn = (a.N + kBN - 1) / kBN;
  int tiles = ntm * ntn;
  int grid = tiles < 152 * 4 ? tiles : 152 * 4;
  ++g_launches;
  launch_pdl(k_gemm<TW, NORM>, dim3(grid, 1, a.groups), dim3(256), 0, s, a, (const float*)D.inv_rms);
}

} // namespace

template <typename TW, bool NORM>
void attrs_one() {
  const int mx = 200 * 1024;
  cudaFuncSetAttribute(k_gemv<TW, NORM, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  cudaFuncSetAttribute(k_gemv<TW, NORM, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  cudaFuncSetAttribute(k_gemv<TW, NORM, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  cudaFuncSetAttribute(k_gemv<TW, NORM, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
}

void kernel_attrs_linear() {
  const int mx = 200 * 1024;
#define LCA_ATTR_BULK1(M, W, N, G, P)                                                                        \
  cudaFuncSetAttribute(k_gemv_bulk<M, W, N, G, P>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);       \
  cudaFuncSetAttribute(k_gemv_bulk<M, W, N, G, P>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
#define LCA_ATTR_BULK(M, W)                                                                                   \
  LCA_ATTR_BULK1(M, W, true, false, false) LCA_ATTR_BULK1(M, W, true, false, true)                          \
  LCA_ATTR_BULK1(M, W, true, true, false) LCA_ATTR_BULK1(M, W, true, true, true)                            \
  LCA_ATTR_BULK1(M, W, false, false, false) LCA_ATTR_BULK1(M, W, false, false, true)                        \
  LCA_ATTR_BULK1(M, W, false, true, false) LCA_ATTR_BULK1(M, W, false, true, true)
  LCA_ATTR_BULK(1, 4) LCA_ATTR_BULK(2, 4) LCA_ATTR_BULK(4, 4) LCA_ATTR_BULK(8, 4) LCA_ATTR_BULK(8, 8)
#undef LCA_ATTR_BULK
#undef LCA_ATTR_BULK1
  attrs_one<__nv_bfloat16, true>();
  attrs_one<__nv_bfloat16, false>();
  attrs_one<float, true>();
  attrs_one<float, false>();
}

// K-split of the bulk-copy GEMV for this layer, or 0 when the layer does not fit it.
int gemv_bulk_ksplit(const Dev& D, const LinearArgs& a) {
  if (a.N % 8 || a.Kd % 256) return 0;
  int ksplit = 1;
  if (a.groups == 1 && a.N <= 2048) {
    ksplit = a.Kd >= 2048 ? D.gemv_ks_big : D.gemv_ks_small;
    while (ksplit > 1 && ((a.Kd % ksplit) || ((a.Kd / ksplit) % 256))) ksplit >>= 1;
  }
  return a.Kd / ksplit > 4096 ? 0 : ksplit;
}

bool gemv_bulk_ok(const Dev& D, const LinearArgs& a) {
  return D.dtype == LCA_BF16 && D.use_tma && gemv_bulk_ksplit(D, a) > 0;
}

void linear(const Dev& D, const LinearArgs& a, bool tiled, cudaStream_t s) {
  const bool norm = a.norm != nullptr;
  ProfScope ps(PK_LINEAR, (double)a.N * a.Kd * a.groups * (D.dtype == LCA_BF16 ? 2 : 4), s);
  if (tiled && D.use_umma && linear_umma(D, a, s)) return;
  // a pre-split input exists only as bf16 halves: callers set presplit only where umma_ready holds
  if (a.presplit) fprintf(stderr, "lca: pre-split layer input on the CUDA-core path (N %d, K %d)\n", a.N, a.Kd);
  if (a.gsplit && (tiled || !gemv_bulk_ok(D, a)))
    fprintf(stderr, "lca: pre-split GEMV input off the bulk-copy GEMV (N %d, K %d)\n", a.N, a.Kd);
  if (D.dtype == LCA_BF16) {
    if (tiled) norm ? launch_gemm<__nv_bfloat16, true>(D, a, s) : launch_gemm<__nv_bfloat16, false>(D, a, s);
    else norm ? launch_gemv<__nv_bfloat16, true>(D, a, s) : launch_gemv<__nv_bfloat16, false>(D, a, s);
  } else {
    if (tiled) norm ? launch_gemm<float, true>(D, a, s) : launch_gemm<float, false>(D, a, s);
    else norm ? launch_gemv<float, true>(D, a, s) : launch_gemv<float, false>(D, a, s);
  }
}

LCA_TRACE_SETTER(trace_set_linear)

} // namespace lca

extern "C" int lca_debug_set_wait_spins(int32_t spins) {
  const int v = spins < 0 ? lca::kWaitSpins : spins;
  lca::stack_set_first_wait(spins);
  return cudaMemcpyToSymbol(lca::g_first_wait_spins, &v, sizeof(v)) == cudaSuccess ? LCA_OK : LCA_E_CUDA;
}
