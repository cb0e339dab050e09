// Tensor-core linear layer for many rows (batched decode, prefill): y = epi(norm?(x) . W^T) with
// tcgen05 (5th-generation tensor cores) on sm_103a.
//
// The layer is bound by streaming W from HBM up to a few hundred rows, so the grid is laid out
// for weight bandwidth: CTA (column tile, K slice, group x row pass) owns a BN-column tile of W
// over one K slice and reads it exactly once for all rows of the pass (up to 512/BN row tiles of
// 128, each with its own TMEM accumulator). The K slices of one column tile form a thread-block
// cluster whose partial sums are added through distributed shared memory.
//
// Warp roles (192 threads, one CTA per SM):
//   * warp 0 streams W tiles (TMA tensor copies, 128-byte swizzle) through a ring of stages;
//     the first ring is issued before the grid-dependency wait, since weights never change;
//   * warp 1 owns TMEM and issues tcgen05.mma (M=128, N=BN, K=16, bf16 x bf16 -> fp32);
//   * warps 2-5 turn the fp32 activations into bf16 A tiles (times the RMSNorm gain, with the
//     row's sum of squares on the side; coalesced: a half-warp reads one row's 64-element block)
//     and run the epilogue. Each activation is split as
//     x = hi + lo with hi = bf16(x) and lo = bf16(x - hi), and both halves are multiplied, so the
//     product keeps about 16 bits of the activation instead of 8 (the weights are exactly bf16).
// Every wait is bounded; a wait that runs out sets the timeout bit of the device error word and
// the kernel finishes without further waiting.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cooperative_groups.h>

#include <algorithm>

#include <cstdio>

#include "common.cuh"
#include "epilogue.cuh"

namespace lca {

namespace {

constexpr int kUM = 128;     // rows per tile (UMMA M)
constexpr int kUN = 64;      // narrowest column tile (UMMA N); layers need N % 64 == 0
constexpr int kUK = 64;      // K per stage (one 128-byte swizzle row of bf16)
constexpr int kUSpins = 1 << 22;

__device__ __forceinline__ uint32_t su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void ubar_init(uint64_t* b, uint32_t n) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(b)), "r"(n) : "memory");
}
__device__ __forceinline__ void ubar_expect(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool ubar_try(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(su32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool ubar_wait(uint64_t* b, uint32_t parity) {
  for (int i = 0; i < kUSpins; ++i)
    if (ubar_try(b, parity)) return true;
  return false;
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFF) >> 4);  // start address
  d |= (uint64_t)1 << 16;                   // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;         // stride byte offset between 8-row groups
  d |= (uint64_t)1 << 46;                   // descriptor version
  d |= (uint64_t)2 << 61;                   // 128-byte swizzle
  return d;
}

__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(su32(bar))
               : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          su32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(su32(bar)), "r"(x), "r"(y)
      : "memory");
}

constexpr int kU2Threads = 192;
constexpr int kAStages = 3;
constexpr uint32_t kAHalf = kUM * kUK * 2;       // 16 KB: one bf16 half of an A tile
constexpr uint32_t kAStageBytes = 2 * kAHalf;    // hi + lo

template <int BN>
struct UCfg {
  static constexpr int kWStages = BN == 128 ? 6 : 8;
  static constexpr uint32_t kWBytes = BN * kUK * 2;
  static constexpr int kMaxMT = 512 / BN;  // row tiles held in TMEM at once
  // D fp32, A and B bf16, both K-major, M = 128, N = BN
  static constexpr uint32_t kIDesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                                     ((uint32_t)(kUM >> 4) << 24);
  static constexpr size_t kSmem = (size_t)kWStages * kWBytes + (size_t)kAStages * kAStageBytes +
                                  (size_t)(kMaxMT + 1) * kUM * 4 + (2 * kWStages + 2 * kAStages + 1) * 8 +
                                  16 + 1024;
};

template <int BN>
__device__ __forceinline__ void umma_n(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(UCfg<BN>::kIDesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void ubar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(b)) : "memory");
}
// bounded wait; once a wait of this thread has failed, later ones return at once
__device__ __forceinline__ void wait_or_fail(uint64_t* b, uint32_t parity, bool& failed) {
  if (failed) return;
  if (!ubar_wait(b, parity)) failed = true;
}
__device__ __forceinline__ void split_bf16(float x, uint16_t& hi, uint16_t& lo) {
  const __nv_bfloat16 h = __float2bfloat16_rn(x);
  const __nv_bfloat16 l = __float2bfloat16_rn(x - __bfloat162float(h));
  hi = *reinterpret_cast<const uint16_t*>(&h);
  lo = *reinterpret_cast<const uint16_t*>(&l);
}


__device__ __forceinline__ void tld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
        "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
        "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Epilogue of one 128 x BN accumulator tile for an epilogue warp: thread = TMEM lane = tile row,
// columns [n0, n0 + BN) of global row `grow`, scaled by `sc`. The operands of each 32-column chunk
// (residual pairs or RoPE factors) are loaded before the stores of the chunk before it, those of
// the first chunk before `wait()` (the accumulator's completion), so that the row walks its
// columns with about one memory latency per two chunks instead of one per column pair.
template <int BN, typename Wait>
__device__ __forceinline__ void tile_epilogue(const EpiArgs& e, uint32_t tbase, int grow, bool ok, int n0,
                                              const float* sc_ptr, float sc_val, Wait wait) {
  EpiRow q{0, 0, 0};
  float2 op0[16], op1[16];
  float sc = sc_val;
  if (ok) {
    q = epi_row(e, grow);
    if (sc_ptr) sc = *sc_ptr;
#pragma unroll
    for (int i = 0; i < 16; ++i) op0[i] = epi_operand(e, q, grow, n0 + 2 * i);
  }
  wait();
#pragma unroll
  for (int cb = 0; cb < BN; cb += 64) {
    uint32_t v[32];
    tld32(tbase + (uint32_t)cb, v);
    if (ok) {
#pragma unroll
      for (int i = 0; i < 16; ++i) op1[i] = epi_operand(e, q, grow, n0 + cb + 32 + 2 * i);
#pragma unroll
      for (int i = 0; i < 16; ++i)
        epi_out<__nv_bfloat16>(e, q, op0[i], grow, n0 + cb + 2 * i, __uint_as_float(v[2 * i]) * sc,
                               __uint_as_float(v[2 * i + 1]) * sc);
    }
    tld32(tbase + (uint32_t)(cb + 32), v);
    if (ok) {
      if (cb + 64 < BN) {
#pragma unroll
        for (int i = 0; i < 16; ++i) op0[i] = epi_operand(e, q, grow, n0 + cb + 64 + 2 * i);
      }
#pragma unroll
      for (int i = 0; i < 16; ++i)
        epi_out<__nv_bfloat16>(e, q, op1[i], grow, n0 + cb + 32 + 2 * i, __uint_as_float(v[2 * i]) * sc,
                               __uint_as_float(v[2 * i + 1]) * sc);
    }
  }
}

// Cluster split-K: rank `ks` adds rows [ks * 128 / KS, ...) of the KS partial tiles (each
// [128][BN + 1] in its CTA's shared memory) and applies the epilogue, four items per batch with
// all loads of a batch before its stores.
template <int BN, int NT>
__device__ __forceinline__ void cluster_epilogue(const EpiArgs& e, cooperative_groups::cluster_group& cl,
                                                 float* red, const float* ssred, int KS, int ks, int mrow0,
                                                 int rbase, int M, int n0, int Kd, float eps, const float* inv,
                                                 bool norm_ss, bool norm_inv) {
  const int RPC = kUM / KS;
  const int items = RPC * (BN / 2);
  constexpr int U = 4;
  for (int base = threadIdx.x; base < items; base += U * NT) {
    float s0[U], s1[U], sc[U];
    float2 op[U];
    EpiRow q[U];
    int gr[U], col[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int idx = base + u * NT;
      const int rl = idx / (BN / 2), c = (idx - rl * (BN / 2)) * 2;
      const int rt = ks * RPC + rl;
      ok[u] = idx < items && mrow0 + rt < M;
      gr[u] = rbase + mrow0 + rt;
      col[u] = n0 + c;
      s0[u] = s1[u] = 0.f;
      sc[u] = 1.f;
      if (ok[u]) {
        float sq = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (k < KS) {
            const float* pr = cl.map_shared_rank(red, k) + rt * (BN + 1) + c;
            s0[u] += pr[0];
            s1[u] += pr[1];
            if (norm_ss) sq += *cl.map_shared_rank(ssred + rt, k);
          }
        }
        if (norm_ss) sc[u] = rsqrtf(sq / (float)Kd + eps);
        if (norm_inv) sc[u] = inv[gr[u]];
        q[u] = epi_row(e, gr[u]);
        op[u] = epi_operand(e, q[u], gr[u], col[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (ok[u]) epi_out<__nv_bfloat16>(e, q[u], op[u], gr[u], col[u], s0[u] * sc[u], s1[u] * sc[u]);
  }
}

template <int BN, bool NORM>
__global__ void __launch_bounds__(kU2Threads, 1)
k_umma(LinearArgs a, const __grid_constant__ CUtensorMap tmW, int MG, int KS, int tcols) {
  using C = UCfg<BN>;
  namespace cgr = cooperative_groups;
  TraceScope _trace(TT_UMMA);
  extern __shared__ __align__(1024) unsigned char usm_raw[];
  unsigned char* base =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(usm_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* Ws = base;                                         // [kWStages][BN x 64 bf16]
  unsigned char* As = Ws + C::kWStages * C::kWBytes;                // [kAStages][hi | lo]
  float* ss_s = reinterpret_cast<float*>(As + kAStages * kAStageBytes);  // [kMaxMT][128]
  float* ssred = ss_s + C::kMaxMT * kUM;                             // [128]
  uint64_t* wfull = reinterpret_cast<uint64_t*>(ssred + kUM);
  uint64_t* wempty = wfull + C::kWStages;
  uint64_t* afull = wempty + C::kWStages;
  uint64_t* aempty = afull + kAStages;
  uint64_t* accdone = aempty + kAStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accdone + 1);
  float* red = reinterpret_cast<float*>(As);  // [128][BN + 1], reuses the A ring after the MMAs

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * BN;
  const int ks = blockIdx.y;
  const int grp = blockIdx.z / MG, mg0 = blockIdx.z % MG;
  const int rbase = grp * a.Mg_stride;
  const int nkb = a.Kd / kUK / KS;
  const int kb0 = ks * nkb;
  const int wrow = grp * a.N + n0;

  if (tid == 0) {
    for (int i = 0; i < C::kWStages; ++i) {
      ubar_init(&wfull[i], 1);
      ubar_init(&wempty[i], 1);
    }
    for (int i = 0; i < kAStages; ++i) {
      ubar_init(&afull[i], 128);
      ubar_init(&aempty[i], 1);
    }
    ubar_init(accdone, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
  }
  __syncthreads();
  // weights never change: the first ring of W tiles streams before the grid-dependency wait
  const int pre = nkb < C::kWStages ? nkb : C::kWStages;
  uint32_t issued = 0;  // W copies this CTA has issued (thread 0)
  if (tid == 0) {
    issued = pre;
    for (int i = 0; i < pre; ++i) {
      ubar_expect(&wfull[i], C::kWBytes);
#pragma unroll
      for (int h = 0; h < BN / 64; ++h)
        tma_load_2d(Ws + (size_t)i * C::kWBytes + h * 8192, &tmW, (kb0 + i) * kUK, wrow + h * 64, &wfull[i]);
    }
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                 "r"(tcols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  const int ntm = (M + kUM - 1) / kUM;
  const int npass = (ntm + C::kMaxMT - 1) / C::kMaxMT;
  int my_passes = (npass - mg0 + MG - 1) / MG;
  if (my_passes < 1) my_passes = 1;  // the pre-issued W tiles are consumed by a first (possibly empty) pass
  bool failed = false;
  uint32_t wit = 0, ait = 0;
  const int r = ((warp & 3) << 5) | lane;  // converter/epilogue row = TMEM lane of this warp quarter
  const int RPC = kUM / KS;                // rows each cluster rank reduces

  for (int ps = 0; ps < my_passes; ++ps) {
    const int mt_lo = (mg0 + ps * MG) * C::kMaxMT;
    int nmt = ntm - mt_lo;
    nmt = nmt < 0 ? 0 : (nmt > C::kMaxMT ? C::kMaxMT : nmt);
    if (warp == 0) {
      if (lane == 0) {
        for (int kb = (ps == 0 ? pre : 0); kb < nkb; ++kb) {
          const uint32_t it = wit + kb;
          const int s = it % C::kWStages;
          if (it >= (uint32_t)C::kWStages) wait_or_fail(&wempty[s], ((it / C::kWStages) - 1) & 1, failed);
          if (failed) break;
          ++issued;
          ubar_expect(&wfull[s], C::kWBytes);
#pragma unroll
          for (int h = 0; h < BN / 64; ++h)
            tma_load_2d(Ws + (size_t)s * C::kWBytes + h * 8192, &tmW, (kb0 + kb) * kUK, wrow + h * 64, &wfull[s]);
        }
      }
    } else if (warp == 1) {
      if (lane == 0) {
        for (int kb = 0; kb < nkb; ++kb) {
          const uint32_t it = wit + kb;
          const int s = it % C::kWStages;
          wait_or_fail(&wfull[s], (it / C::kWStages) & 1, failed);
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t bbase = su32(Ws + (size_t)s * C::kWBytes);
          for (int j = 0; j < nmt; ++j) {
            const uint32_t at = ait + kb * nmt + j;
            const int sa = at % kAStages;
            wait_or_fail(&afull[sa], (at / kAStages) & 1, failed);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t ahi = su32(As + (size_t)sa * kAStageBytes), alo = ahi + kAHalf;
            const uint32_t d = tmem + (uint32_t)(j * BN);
            if (!failed) {
#pragma unroll
              for (int k = 0; k < kUK / 16; ++k) {
                umma_n<BN>(d, sdesc(ahi + k * 32), sdesc(bbase + k * 32), (kb > 0 || k > 0) ? 1u : 0u);
                umma_n<BN>(d, sdesc(alo + k * 32), sdesc(bbase + k * 32), 1u);
              }
            }
            umma_commit(&aempty[sa]);
          }
          if (nmt > 0) umma_commit(&wempty[s]);
          else ubar_arrive(&wempty[s]);
        }
        if (nmt > 0) umma_commit(accdone);
        else ubar_arrive(accdone);
      }
    } else {
      // converters: step st = (kb, j) in the MMA thread's order. A half-warp reads one row's
      // 64-element block (16 lanes x 16 bytes, coalesced); a warp instruction covers two rows.
      const int cw = warp - 2, half = lane >> 4, q = lane & 15;
      if (NORM && q == 0)
        for (int j = 0; j < nmt; ++j)
#pragma unroll
          for (int it = 0; it < 16; ++it) ss_s[j * kUM + 2 * (cw + 4 * it) + half] = 0.f;
      const int steps = nkb * nmt;
      float4 cur[16];
      auto load_step = [&](int st, float4 (&v)[16]) {
        const int kb = st / nmt, j = st - kb * nmt;
        const float* xb = a.x + (size_t)(kb0 + kb) * kUK + q * 4;
#pragma unroll
        for (int it = 0; it < 16; ++it) {
          const int row = (mt_lo + j) * kUM + 2 * (cw + 4 * it) + half;
          v[it] = row < M ? *reinterpret_cast<const float4*>(xb + (size_t)(rbase + row) * a.ldx)
                          : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      };
      auto convert_step = [&](int st, const float4 (&v)[16]) {
        const int kb = st / nmt, j = st - kb * nmt;
        const uint32_t at = ait + st;
        const int sa = at % kAStages;
        if (at >= (uint32_t)kAStages) wait_or_fail(&aempty[sa], ((at / kAStages) - 1) & 1, failed);
        unsigned char* ahi = As + (size_t)sa * kAStageBytes;
        unsigned char* alo = ahi + kAHalf;
        const int k0 = (kb0 + kb) * kUK;
        float4 g = make_float4(1.f, 1.f, 1.f, 1.f);
        if (NORM) g = *reinterpret_cast<const float4*>(a.norm + k0 + q * 4);
#pragma unroll
        for (int it = 0; it < 16; ++it) {
          const int rr = 2 * (cw + 4 * it) + half;  // row within the tile
          float e[4] = {v[it].x, v[it].y, v[it].z, v[it].w};
          if (NORM) {
            float ss = e[0] * e[0] + e[1] * e[1] + e[2] * e[2] + e[3] * e[3];
#pragma unroll
            for (int o = 8; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
            if (q == 0) ss_s[j * kUM + rr] += ss;
            e[0] *= g.x; e[1] *= g.y; e[2] *= g.z; e[3] *= g.w;
          }
          uint16_t h[4], l[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) split_bf16(e[u], h[u], l[u]);
          const int off = (rr >> 3) * 1024 + (rr & 7) * 128 + (((q >> 1) ^ (rr & 7)) * 16) + (q & 1) * 8;
          *reinterpret_cast<uint2*>(ahi + off) = make_uint2(h[0] | ((uint32_t)h[1] << 16), h[2] | ((uint32_t)h[3] << 16));
          *reinterpret_cast<uint2*>(alo + off) = make_uint2(l[0] | ((uint32_t)l[1] << 16), l[2] | ((uint32_t)l[3] << 16));
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        ubar_arrive(&afull[sa]);
      };
      // two register buffers in turn: the loads of the next step are in flight while this one
      // is converted (no register copies that would wait for them)
      float4 nxt[16];
      if (steps > 0) load_step(0, cur);
      for (int st = 0; st < steps; st += 2) {
        if (st + 1 < steps) load_step(st + 1, nxt);
        convert_step(st, cur);
        if (st + 2 < steps) load_step(st + 2, cur);
        if (st + 1 < steps) convert_step(st + 1, nxt);
      }
      // the row sums of squares were written by other converter threads than the epilogue's
      asm volatile("bar.sync 1, 128;" ::: "memory");
      wait_or_fail(accdone, ps & 1, failed);
    }
    __syncwarp();
    wit += nkb;
    ait += nkb * nmt;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    // ---- epilogue of this pass
    for (int j = 0; j < nmt; ++j) {
      const int mrow0 = (mt_lo + j) * kUM;
      if (KS == 1) {
        if (warp >= 2) {
          const int row = mrow0 + r;
          const float inv = NORM ? rsqrtf(ss_s[j * kUM + r] / (float)a.Kd + a.eps) : 1.f;
          tile_epilogue<BN>(a.epi, tmem + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)(j * BN), rbase + row,
                            row < M, n0, nullptr, inv, [] {});
        }
      } else {
        cgr::cluster_group cl = cgr::this_cluster();
        if (warp >= 2) {
#pragma unroll
          for (int cb = 0; cb < BN; cb += 32) {
            uint32_t v[32];
            tld32(tmem + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)(j * BN + cb), v);
#pragma unroll
            for (int q = 0; q < 32; ++q) red[r * (BN + 1) + cb + q] = __uint_as_float(v[q]);
          }
          ssred[r] = NORM ? ss_s[j * kUM + r] : 0.f;
        }
        cl.sync();
        cluster_epilogue<BN, kU2Threads>(a.epi, cl, red, ssred, KS, ks, mrow0, rbase, M, n0, a.Kd, a.eps, nullptr,
                                         NORM, false);
        cl.sync();
      }
    }
    // TMEM reads of this pass are done before the next pass's MMAs overwrite the accumulators
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  }
  // after a failed wait, W copies may still be in flight: wait (bounded) for the last one issued
  // into each stage before the CTA's shared memory is released
  const bool any_failed = __syncthreads_or(failed);
  if (tid == 0 && any_failed) {
    for (uint32_t s = 0; s < (uint32_t)C::kWStages && s < issued; ++s) {
      const uint32_t last = issued - 1 - ((issued - 1 - s) % C::kWStages);
      ubar_wait(&wfull[last % C::kWStages], (last / C::kWStages) & 1);
    }
    atomicOr(a.epi.err, kErrTimeout);
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tcols) : "memory");
}

template <int BN, bool NORM>
void umma_go(const LinearArgs& a, const CUtensorMap& tm, dim3 grid, int MG, int KS, int tcols, cudaStream_t s) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kU2Threads);
  cfg.dynamicSmemBytes = UCfg<BN>::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = KS;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  cudaLaunchKernelEx(&cfg, k_umma<BN, NORM>, a, tm, MG, KS, tcols);
}

}  // namespace

// ---------------------------------------------------------------- split rows + TMA-fed GEMM
// For the decode step's many-row layers the activations are split once per layer by
// k_split_rows (one warp per row: x * g -> hi = bf16, lo = bf16(rest); the row's inverse RMS on
// the side), and k_tgemm then streams both operands by TMA: 2D output tiles of 128 rows x BN
// columns, the activation tiles' two halves and the weight tile sharing one stage of a ring,
// a split of K across a thread-block cluster when the grid would be thin.
template <bool NORM>
__global__ void __launch_bounds__(256)
k_split_rows(LinearArgs a, __nv_bfloat16* __restrict__ hi, __nv_bfloat16* __restrict__ lo,
             float* __restrict__ inv) {
  TraceScope _trace(TT_UMMA);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = gridDim.x * (blockDim.x >> 5);
  const int K = a.Kd;
  for (int rr = blockIdx.x * (blockDim.x >> 5) + warp; rr < a.groups * a.M_cap; rr += nw) {
    const int grp = rr / a.M_cap, r = rr - grp * a.M_cap;
    if (r >= M) continue;
    const size_t row = (size_t)grp * a.Mg_stride + r;
    const float4* xr = reinterpret_cast<const float4*>(a.x + row * a.ldx);
    float ss = 0.f;
    for (int k4 = lane; k4 < K / 4; k4 += 32) {
      float4 v = xr[k4];
      if (NORM) {
        ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        const float4 g = reinterpret_cast<const float4*>(a.norm)[k4];
        v.x *= g.x; v.y *= g.y; v.z *= g.z; v.w *= g.w;
      }
      uint16_t h0, h1, h2, h3, l0, l1, l2, l3;
      split_bf16(v.x, h0, l0);
      split_bf16(v.y, h1, l1);
      split_bf16(v.z, h2, l2);
      split_bf16(v.w, h3, l3);
      reinterpret_cast<uint2*>(hi + row * K)[k4] = make_uint2(h0 | ((uint32_t)h1 << 16), h2 | ((uint32_t)h3 << 16));
      reinterpret_cast<uint2*>(lo + row * K)[k4] = make_uint2(l0 | ((uint32_t)l1 << 16), l2 | ((uint32_t)l3 << 16));
    }
    if (NORM) {
#pragma unroll
      for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
      if (lane == 0) inv[row] = rsqrtf(ss / (float)K + a.eps);
    }
  }
}

constexpr int kTThreads = 192;
template <int BN>
struct TCfg {
  static constexpr int kStages = BN == 256 ? 3 : 4;
  static constexpr uint32_t kABytes = kUM * kUK * 2;          // one half (hi or lo) of an A tile
  static constexpr uint32_t kWBytes = BN * kUK * 2;
  static constexpr uint32_t kStageBytes = 2 * kABytes + kWBytes;
  static constexpr uint32_t kIDesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                                     ((uint32_t)(kUM >> 4) << 24);
  static constexpr size_t kSmem = (size_t)kStages * kStageBytes + (2 * kStages + 1) * 8 + 16 + 1024;
  static_assert((size_t)kUM * (BN + 1) * 4 <= (size_t)kStages * kStageBytes, "reduction buffer");
};

template <int BN>
__device__ __forceinline__ void tmma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(TCfg<BN>::kIDesc), "r"(accumulate)
      : "memory");
}

template <int BN>
__global__ void __launch_bounds__(kTThreads, 1)
k_tgemm(LinearArgs a, const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmAh,
        const __grid_constant__ CUtensorMap tmAl, const float* __restrict__ inv, int MT, int KS) {
  using C = TCfg<BN>;
  namespace cgr = cooperative_groups;
  TraceScope _trace(TT_UMMA);
  extern __shared__ __align__(1024) unsigned char tsm_raw[];
  unsigned char* ring =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(tsm_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + C::kStages * C::kStageBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* accdone = empty + C::kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accdone + 1);
  float* red = reinterpret_cast<float*>(ring);  // [128][BN + 1] after the MMAs

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * BN;
  const int ks = blockIdx.y;
  const int grp = blockIdx.z / MT, mt = blockIdx.z % MT;
  const int rbase = grp * a.Mg_stride;
  const int nkb = a.Kd / kUK / KS;
  const int kb0 = ks * nkb;
  const int wrow = grp * a.N + n0;
  const int arow = rbase + mt * kUM;

  if (tid == 0) {
    for (int i = 0; i < C::kStages; ++i) {
      ubar_init(&full[i], 1);
      ubar_init(&empty[i], 1);
    }
    ubar_init(accdone, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
  }
  __syncthreads();
  // weights never change: the W part of the first stages is copied before the dependency wait
  const int pre = nkb < C::kStages ? nkb : C::kStages;
  if (tid == 0) {
    for (int i = 0; i < pre; ++i) {
      ubar_expect(&full[i], C::kStageBytes);
      unsigned char* st = ring + (size_t)i * C::kStageBytes;
#pragma unroll
      for (int h = 0; h < BN / 64; ++h)
        tma_load_2d(st + 2 * C::kABytes + h * 8192, &tmW, (kb0 + i) * kUK, wrow + h * 64, &full[i]);
    }
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  const bool live = mt * kUM < M;  // the same for every CTA of a cluster
  bool failed = false;
  uint32_t issued = pre;
  if (tid == 0) {
    // the activation halves of the first stages (written by the previous kernel)
    for (int i = 0; i < pre; ++i) {
      unsigned char* st = ring + (size_t)i * C::kStageBytes;
      tma_load_2d(st, &tmAh, (kb0 + i) * kUK, arow, &full[i]);
      tma_load_2d(st + C::kABytes, &tmAl, (kb0 + i) * kUK, arow, &full[i]);
    }
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                 "r"(BN < 32 ? 32 : BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      for (int kb = pre; kb < nkb; ++kb) {
        const int s = kb % C::kStages;
        wait_or_fail(&empty[s], ((kb / C::kStages) - 1) & 1, failed);
        if (failed) break;
        ++issued;
        unsigned char* st = ring + (size_t)s * C::kStageBytes;
        ubar_expect(&full[s], C::kStageBytes);
        tma_load_2d(st, &tmAh, (kb0 + kb) * kUK, arow, &full[s]);
        tma_load_2d(st + C::kABytes, &tmAl, (kb0 + kb) * kUK, arow, &full[s]);
#pragma unroll
        for (int h = 0; h < BN / 64; ++h)
          tma_load_2d(st + 2 * C::kABytes + h * 8192, &tmW, (kb0 + kb) * kUK, wrow + h * 64, &full[s]);
      }
      // traced launches mark the end of the main loop
      if (g_trace) {
        wait_or_fail(accdone, 0, failed);
        _trace.mark();
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % C::kStages;
        wait_or_fail(&full[s], (kb / C::kStages) & 1, failed);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t ahi = su32(ring + (size_t)s * C::kStageBytes);
        const uint32_t alo = ahi + C::kABytes, wb = ahi + 2 * C::kABytes;
        if (live && !failed) {
#pragma unroll
          for (int k = 0; k < kUK / 16; ++k) {
            tmma<BN>(tmem, sdesc(ahi + k * 32), sdesc(wb + k * 32), (kb > 0 || k > 0) ? 1u : 0u);
            tmma<BN>(tmem, sdesc(alo + k * 32), sdesc(wb + k * 32), 1u);
          }
          umma_commit(&empty[s]);
        } else {
          ubar_arrive(&empty[s]);
        }
      }
      if (live) umma_commit(accdone);
      else ubar_arrive(accdone);
    }
  } else if (!live || KS > 1) {
    wait_or_fail(accdone, 0, failed);
  }
  __syncwarp();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const int r = ((warp & 3) << 5) | lane;  // epilogue row = TMEM lane
  if (live) {
    if (KS == 1) {
      if (warp >= 2) {
        const int row = mt * kUM + r;
        // the accumulator wait sits inside, after the first chunk's operand loads
        tile_epilogue<BN>(a.epi, tmem + ((uint32_t)((warp & 3) * 32) << 16), rbase + row, row < M, n0,
                          a.norm ? inv + rbase + row : nullptr, 1.f, [&] {
                            wait_or_fail(accdone, 0, failed);
                            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                          });
      }
    } else {
      cgr::cluster_group cl = cgr::this_cluster();
      if (warp >= 2) {
#pragma unroll
        for (int cb = 0; cb < BN; cb += 32) {
          uint32_t v[32];
          tld32(tmem + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)cb, v);
#pragma unroll
          for (int q = 0; q < 32; ++q) red[r * (BN + 1) + cb + q] = __uint_as_float(v[q]);
        }
      }
      cl.sync();
      cluster_epilogue<BN, kTThreads>(a.epi, cl, red, nullptr, KS, ks, mt * kUM, rbase, M, n0, a.Kd, a.eps, inv,
                                      false, a.norm != nullptr);
      cl.sync();
    }
  }
  const bool any_failed = __syncthreads_or(failed);
  if (tid == 0 && any_failed) {
    for (uint32_t s = 0; s < (uint32_t)C::kStages && s < issued; ++s) {
      const uint32_t last = issued - 1 - ((issued - 1 - s) % C::kStages);
      ubar_wait(&full[last % C::kStages], (last / C::kStages) & 1);
    }
    atomicOr(a.epi.err, kErrTimeout);
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(BN < 32 ? 32 : BN)
                 : "memory");
}

template <int BN>
void tgemm_go(const LinearArgs& a, const CUtensorMap& tw, const CUtensorMap& th, const CUtensorMap& tl,
              const float* inv, int MT, int KS, cudaStream_t s) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(a.N / BN, KS, a.groups * MT);
  cfg.blockDim = dim3(kTThreads);
  cfg.dynamicSmemBytes = TCfg<BN>::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = KS;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  cudaLaunchKernelEx(&cfg, k_tgemm<BN>, a, tw, th, tl, inv, MT, KS);
}

// Split rows, then the TMA-fed GEMM. Tile width BN (256, 128 or 64, dividing N) and K split KS
// (power of two, at most 8, at least two 64-deep blocks per CTA, while the grid fits one wave)
// minimise a simple cost: waves x (BN x K blocks per CTA + a fixed part) + a cluster-reduction
// term proportional to BN; ties go to the wider tile.
void split_gemm(const Dev& D, const LinearArgs& a, const void* amap, __nv_bfloat16* hi, __nv_bfloat16* lo,
                float* inv, cudaStream_t s) {
  const int sms = D.num_sms > 0 ? D.num_sms : 148;
  {
    const int need = a.groups * a.M_cap;
    const int blocks = std::min((need + 7) / 8, 4 * sms);
    ++g_launches;
    if (a.norm) launch_pdl(k_split_rows<true>, dim3(blocks), dim3(256), 0, s, a, hi, lo, inv);
    else launch_pdl(k_split_rows<false>, dim3(blocks), dim3(256), 0, s, a, hi, lo, inv);
  }
  const int MT = (a.M_cap + kUM - 1) / kUM;
  const int kb = a.Kd / kUK;
  int best_bn = 64, best_ks = 1;
  long long best = -1;
  for (int bn : {256, 128, 64}) {
    if (a.N % bn) continue;
    const long long base = (long long)(a.N / bn) * a.groups * MT;
    int ks = 1;
    while (ks < 8 && kb % (2 * ks) == 0 && kb / (2 * ks) >= 2 && base * 2 * ks <= sms) ks *= 2;
    const long long tot = base * ks;
    const long long waves = (tot + sms - 1) / sms;
    const long long cost = waves * ((long long)bn * (kb / ks) + 512) + (ks > 1 ? 2LL * bn : 0);
    if (best < 0 || cost < best) {
      best = cost;
      best_bn = bn;
      best_ks = ks;
    }
  }
  CUtensorMap tw, th, tl;
  memcpy(&tw, a.tmap, sizeof(tw));
  memcpy(&th, amap, sizeof(th));
  memcpy(&tl, static_cast<const unsigned char*>(amap) + 128, sizeof(tl));
  if (best_bn == 256) tgemm_go<256>(a, tw, th, tl, inv, MT, best_ks, s);
  else if (best_bn == 128) tgemm_go<128>(a, tw, th, tl, inv, MT, best_ks, s);
  else tgemm_go<64>(a, tw, th, tl, inv, MT, best_ks, s);
}

// Tensor map of a bf16 weight [rows][K] (K innermost) with 64 x 64 boxes and the 128-byte swizzle.
int make_weight_tmap(void* out, const void* W, long long rows, long long K) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return LCA_E_CUDA;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  if (K % kUK || rows % kUN) return LCA_E_ARG;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kUK, (cuuint32_t)kUN};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = encode(reinterpret_cast<CUtensorMap*>(out), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                            const_cast<void*>(W), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LCA_OK : LCA_E_CUDA;
}

// Tensor maps (hi, lo) of the split activations [rows][K] bf16 with 64 x 128 boxes, 128-byte swizzle.
int make_split_tmaps(void* out, const void* hi, const void* lo, long long rows, long long K) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return LCA_E_CUDA;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  if (K % kUK || rows < 1) return LCA_E_ARG;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kUK, (cuuint32_t)kUM};
  const cuuint32_t estr[2] = {1, 1};
  for (int h = 0; h < 2; ++h) {
    const CUresult r = encode(reinterpret_cast<CUtensorMap*>(static_cast<unsigned char*>(out) + 128 * h),
                              CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(h ? lo : hi), dims, strides,
                              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return LCA_E_CUDA;
  }
  return LCA_OK;
}

void kernel_attrs_umma() {
  cudaFuncSetAttribute(k_tgemm<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TCfg<64>::kSmem);
  cudaFuncSetAttribute(k_tgemm<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TCfg<128>::kSmem);
  cudaFuncSetAttribute(k_tgemm<256>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TCfg<256>::kSmem);
  cudaFuncSetAttribute(k_umma<64, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)UCfg<64>::kSmem);
  cudaFuncSetAttribute(k_umma<64, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)UCfg<64>::kSmem);
  cudaFuncSetAttribute(k_umma<128, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)UCfg<128>::kSmem);
  cudaFuncSetAttribute(k_umma<128, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)UCfg<128>::kSmem);
}

// Launch on the tensor cores when the layer fits the tile shapes; false otherwise.
// Shape choice: 128-column tiles when at most four row tiles are typical and the layer is wide
// enough to fill the GPU with them, else 64; then split K (power of two, at most 8, at least two
// 64-deep blocks per CTA) while the grid still fits one wave of one CTA per SM.
bool linear_umma(const Dev& D, const LinearArgs& a, cudaStream_t s) {
  if (!a.tmap || D.dtype != LCA_BF16 || a.N % kUN || a.Kd % kUK) return false;
  if (a.amap && a.groups * a.M_cap <= D.as_rows) {
    split_gemm(D, a, a.amap, D.as_hi, D.as_lo, D.as_inv, s);
    return true;
  }
  const int mt_cap = (a.M_cap + kUM - 1) / kUM;
  const int rows_typ = a.rows_typ > 0 ? a.rows_typ : a.M_cap;
  int mt_typ = (rows_typ + kUM - 1) / kUM;
  mt_typ = mt_typ < 1 ? 1 : (mt_typ > mt_cap ? mt_cap : mt_typ);
  const int sms = D.num_sms > 0 ? D.num_sms : 148;
  const bool wide = mt_typ <= 4 && a.N % 128 == 0 && (long long)(a.N / 128) * a.groups * 8 >= sms;
  const int BN = wide ? 128 : 64;
  const int max_mt = 512 / BN;
  const int ncol = a.N / BN;
  const int mt_pass_cap = mt_cap < max_mt ? mt_cap : max_mt;
  int tcols = 32;
  while (tcols < mt_pass_cap * BN) tcols <<= 1;
  int MG = (mt_typ + max_mt - 1) / max_mt;
  const int MG_cap = (mt_cap + max_mt - 1) / max_mt;
  MG = MG < 1 ? 1 : (MG > MG_cap ? MG_cap : MG);
  const int kb = a.Kd / kUK;
  int KS = 1;
  while (KS < 8 && kb % (2 * KS) == 0 && kb / (2 * KS) >= 2 &&
         (long long)ncol * a.groups * MG * (2 * KS) <= sms)
    KS *= 2;
  CUtensorMap tm;
  memcpy(&tm, a.tmap, sizeof(tm));
  const dim3 grid(ncol, KS, a.groups * MG);
  if (BN == 128) {
    if (a.norm) umma_go<128, true>(a, tm, grid, MG, KS, tcols, s);
    else umma_go<128, false>(a, tm, grid, MG, KS, tcols, s);
  } else {
    if (a.norm) umma_go<64, true>(a, tm, grid, MG, KS, tcols, s);
    else umma_go<64, false>(a, tm, grid, MG, KS, tcols, s);
  }
  return true;
}

LCA_TRACE_SETTER(trace_set_umma)

}  // namespace lca

using namespace lca;

extern "C" size_t lca_debug_gemm_scratch_bytes(int32_t M, int32_t K) {
  if (M < 1 || K < 1) return 0;
  return (size_t)M * K * 2 * 2 + (size_t)M * 4 + 512;
}

extern "C" int lca_debug_gemm(const float* x, const void* W, float* y, int32_t M, int32_t N, int32_t K,
                              const int32_t* M_dev, int32_t rows_typ, int32_t* err_dev, void* scratch,
                              void* stream) {
  if (!x || !W || !y || !M_dev || !err_dev || M < 1 || N < 1 || K < 1 || rows_typ < 0 || rows_typ > M)
    return LCA_E_ARG;
  CUtensorMap tm;
  int st = make_weight_tmap(&tm, W, N, K);
  if (st != LCA_OK) return st;
  Dev D{};
  D.dtype = LCA_BF16;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  D.num_sms = sms;
  D.use_umma = 1;
  kernel_attrs_umma();
  int* err = err_dev;
  LinearArgs a{};
  a.x = x;
  a.ldx = K;
  a.W = W;
  a.N = N;
  a.Kd = K;
  a.groups = 1;
  a.M = M_dev;
  a.M_cap = M;
  a.rows_typ = rows_typ > 0 ? rows_typ : M;
  a.tmap = &tm;
  a.epi.mode = EPI_STORE;
  a.epi.y = y;
  a.epi.ldy = N;
  a.epi.err = err;
  if (scratch) {
    if (N % kUN || K % kUK) return LCA_E_ARG;
    char* p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(scratch) + 255) & ~uintptr_t(255));
    __nv_bfloat16* hi = reinterpret_cast<__nv_bfloat16*>(p);
    __nv_bfloat16* lo = hi + (size_t)M * K;
    float* inv = reinterpret_cast<float*>(lo + (size_t)M * K);
    alignas(64) unsigned char maps[256];
    st = make_split_tmaps(maps, hi, lo, M, K);
    if (st != LCA_OK) return st;
    split_gemm(D, a, maps, hi, lo, inv, reinterpret_cast<cudaStream_t>(stream));
    return cudaGetLastError() == cudaSuccess ? LCA_OK : LCA_E_CUDA;
  }
  if (!linear_umma(D, a, reinterpret_cast<cudaStream_t>(stream))) return LCA_E_ARG;
  return cudaGetLastError() == cudaSuccess ? LCA_OK : LCA_E_CUDA;
}
