// Tensor-core linear layer for many rows (batched decode, prefill): y = epi(norm?(x) . W^T) with
// tcgen05 (5th-generation tensor cores) on sm_103a.
//
// Two launches per layer:
//   * k_split_rows turns the layer's fp32 activations into two bf16 matrices, hi = bf16(x * g) and
//     lo = bf16(x * g - hi) (g: the RMSNorm gain, if the layer has one), plus each row's inverse
//     RMS. Both halves are multiplied below, so the product keeps about 16 bits of each activation
//     instead of 8; the weights are exactly bf16.
//   * k_tgemm streams both operands by TMA (tensor maps, 128-byte swizzle): output tiles of 128 rows
//     x BN columns, the two activation halves and the weight tile of one 64-deep K block sharing a
//     stage of a ring. Warp 0 issues the copies (the weight part of the first stages before the
//     grid-dependency wait, since weights never change), warp 1 owns TMEM and issues
//     tcgen05.mma (M=128, N=BN, K=16, bf16 x bf16 -> fp32), warps 2-5 run the epilogue from TMEM.
//     The grid covers the typical row count; a CTA walks further row tiles when a launch has more
//     rows. When the grid would be thin, K is split across a thread-block cluster and the partial
//     tiles are added through distributed shared memory.
// Every wait is bounded; a wait that runs out sets the timeout bit of the device error word and
// the kernel finishes without further waiting.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cooperative_groups.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>

#include "common.cuh"
#include "epilogue.cuh"

namespace lca {

namespace {

constexpr int kUM = 128;  // rows per tile (UMMA M)
constexpr int kUN = 64;   // narrowest column tile; layers need N % 64 == 0
constexpr int kUK = 64;   // K per stage (one 128-byte swizzle row of bf16)
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
__device__ __forceinline__ void ubar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(b)) : "memory");
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
// bounded wait; once a wait of this thread has failed, later ones return at once
__device__ __forceinline__ void wait_or_fail(uint64_t* b, uint32_t parity, bool& failed) {
  if (failed) return;
  if (!ubar_wait(b, parity)) failed = true;
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
__device__ __forceinline__ void split_bf16(float x, uint16_t& hi, uint16_t& lo) {
  const __nv_bfloat16 h = __float2bfloat16_rn(x);
  const __nv_bfloat16 l = __float2bfloat16_rn(x - __bfloat162float(h));
  hi = *reinterpret_cast<const uint16_t*>(&h);
  lo = *reinterpret_cast<const uint16_t*>(&l);
}
__device__ __forceinline__ uint32_t bf2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// Split on write: bf16 halves of NV output values (times the consumer's RMSNorm gain, if any) at
// columns [c0, c0 + NV) of row r, as 16-byte vectors.
template <int NV>
__device__ __forceinline__ void split_store(const EpiArgs& e, int r, int c0, const float (&y)[NV]) {
  uint32_t h[NV / 2], l[NV / 2];
#pragma unroll
  for (int i = 0; i < NV / 4; ++i) {
    const float4 g = e.sg ? reinterpret_cast<const float4*>(e.sg + c0)[i] : make_float4(1.f, 1.f, 1.f, 1.f);
    uint16_t h0, h1, h2, h3, l0, l1, l2, l3;
    split_bf16(y[4 * i] * g.x, h0, l0);
    split_bf16(y[4 * i + 1] * g.y, h1, l1);
    split_bf16(y[4 * i + 2] * g.z, h2, l2);
    split_bf16(y[4 * i + 3] * g.w, h3, l3);
    h[2 * i] = h0 | ((uint32_t)h1 << 16);
    h[2 * i + 1] = h2 | ((uint32_t)h3 << 16);
    l[2 * i] = l0 | ((uint32_t)l1 << 16);
    l[2 * i + 1] = l2 | ((uint32_t)l3 << 16);
  }
  uint4* ph = reinterpret_cast<uint4*>(e.sp_hi + (size_t)r * e.ldsp + c0);
  uint4* pl = reinterpret_cast<uint4*>(e.sp_lo + (size_t)r * e.ldsp + c0);
#pragma unroll
  for (int j = 0; j < NV / 8; ++j) {
    ph[j] = make_uint4(h[4 * j], h[4 * j + 1], h[4 * j + 2], h[4 * j + 3]);
    pl[j] = make_uint4(l[4 * j], l[4 * j + 1], l[4 * j + 2], l[4 * j + 3]);
  }
}

// ---------------------------------------------------------------- epilogue of 32-column chunks
// A thread owns one row of the tile and walks its columns in chunks of 32 (a chunk lies inside one
// head and one of Q/K/V, since d and head_dim are multiples of 32). Operands of a chunk: 32 residual
// values, or 16 RoPE (cos, sin) pairs; outputs go out as 16-byte vectors.
__device__ __forceinline__ void chunk_ops(const EpiArgs& e, const EpiRow& q, int r, int c0, float4 (&op)[8]) {
  if (e.mode == EPI_RESID || e.mode == EPI_RESID_SILU) {
    const float4* p = reinterpret_cast<const float4*>(e.res + (size_t)r * e.ldres + c0);
#pragma unroll
    for (int i = 0; i < 8; ++i) op[i] = p[i];
  } else if (e.mode == EPI_QKV) {
    const int part = c0 / e.d;
    if (part < 2) {
      const int dd0 = (c0 - part * e.d) % e.hd;
      const float4* p = reinterpret_cast<const float4*>(e.rope + (size_t)q.pos * (e.hd >> 1) + (dd0 >> 1));
#pragma unroll
      for (int i = 0; i < 8; ++i) op[i] = p[i];
    }
  }
}

template <typename TC>
__device__ __forceinline__ void chunk_out(const EpiArgs& e, const EpiRow& q, const float4 (&op)[8], int r, int c0,
                                          const uint32_t (&v)[32], float sc) {
  float x[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) x[i] = __uint_as_float(v[i]) * sc;
  switch (e.mode) {
    case EPI_STORE: {
      float4* y = reinterpret_cast<float4*>(e.y + (size_t)r * e.ldy + c0);
#pragma unroll
      for (int i = 0; i < 8; ++i) y[i] = make_float4(x[4 * i], x[4 * i + 1], x[4 * i + 2], x[4 * i + 3]);
      break;
    }
    case EPI_RESID:
    case EPI_RESID_SILU: {
      const bool sl = e.mode == EPI_RESID_SILU;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        x[4 * i] = op[i].x + (sl ? silu_f(x[4 * i]) : x[4 * i]);
        x[4 * i + 1] = op[i].y + (sl ? silu_f(x[4 * i + 1]) : x[4 * i + 1]);
        x[4 * i + 2] = op[i].z + (sl ? silu_f(x[4 * i + 2]) : x[4 * i + 2]);
        x[4 * i + 3] = op[i].w + (sl ? silu_f(x[4 * i + 3]) : x[4 * i + 3]);
      }
      if (!e.sp_only) {
        float4* y = reinterpret_cast<float4*>(e.y + (size_t)r * e.ldy + c0);
#pragma unroll
        for (int i = 0; i < 8; ++i) y[i] = make_float4(x[4 * i], x[4 * i + 1], x[4 * i + 2], x[4 * i + 3]);
      }
      if (e.sp_hi) {
        split_store<32>(e, r, c0, x);
        if (e.ss) {
          float q2 = 0.f;
#pragma unroll
          for (int i = 0; i < 32; ++i) q2 += x[i] * x[i];
          e.ss[(size_t)r * e.ss_ld + (c0 >> 5)] = q2;
        }
      }
      break;
    }
    case EPI_SWIGLU: {
      // interleaved (gate, up) columns -> silu(gate) * up at column c / 2
      float m[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) m[i] = silu_f(x[2 * i]) * x[2 * i + 1];
      if (!e.sp_only) {
        float4* y = reinterpret_cast<float4*>(e.y + (size_t)r * e.ldy + (c0 >> 1));
#pragma unroll
        for (int i = 0; i < 4; ++i) y[i] = make_float4(m[4 * i], m[4 * i + 1], m[4 * i + 2], m[4 * i + 3]);
      }
      if (e.sp_hi) split_store<16>(e, r, c0 >> 1, m);
      break;
    }
    case EPI_QKV: {
      const int part = c0 / e.d;
      const int cc0 = c0 - part * e.d;
      const int h = cc0 / e.hd;
      const int dd0 = cc0 - h * e.hd;
      if (part < 2) {
        // interleaved rotary pairs (2i, 2i + 1) with this chunk's 16 (cos, sin) factors
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float c = (j & 1) ? op[j >> 1].z : op[j >> 1].x;
          const float s = (j & 1) ? op[j >> 1].w : op[j >> 1].y;
          const float a0 = x[2 * j], a1 = x[2 * j + 1];
          x[2 * j] = a0 * c - a1 * s;
          x[2 * j + 1] = a0 * s + a1 * c;
        }
      }
      if (part == 0) {
        float4* y = reinterpret_cast<float4*>(e.y + (size_t)r * e.ldy + cc0);
#pragma unroll
        for (int i = 0; i < 8; ++i) y[i] = make_float4(x[4 * i], x[4 * i + 1], x[4 * i + 2], x[4 * i + 3]);
      } else {
        if (!kv_write_ok(e.kv, q.slot, q.pg)) {
          atomicOr(e.err, kErrIndex);
          return;
        }
        TC* base = reinterpret_cast<TC*>(part == 1 ? e.kv.k : e.kv.v);
        TC* p = base + kv_addr(e.kv, e.H, e.hd, q.b, h, q.slot, q.pg) + dd0;
        if (sizeof(TC) == 2) {
          uint4* d4 = reinterpret_cast<uint4*>(p);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            d4[i] = make_uint4(bf2(x[8 * i], x[8 * i + 1]), bf2(x[8 * i + 2], x[8 * i + 3]),
                               bf2(x[8 * i + 4], x[8 * i + 5]), bf2(x[8 * i + 6], x[8 * i + 7]));
        } else {
          float4* d4 = reinterpret_cast<float4*>(p);
#pragma unroll
          for (int i = 0; i < 8; ++i) d4[i] = make_float4(x[4 * i], x[4 * i + 1], x[4 * i + 2], x[4 * i + 3]);
        }
      }
      break;
    }
  }
}

// Epilogue of one 128 x BN accumulator tile for an epilogue warp: thread = TMEM lane = tile row,
// columns [n0, n0 + BN) of global row `grow`, scaled by sc. The operands of a chunk are loaded
// before the stores of the chunk before it, those of the first chunk before `wait()` (the
// accumulator's completion), so a row costs about one memory latency per two chunks.
template <int BN, typename Wait>
__device__ __forceinline__ void tile_epilogue(const EpiArgs& e, uint32_t tbase, int grow, bool ok, int n0,
                                              float sc, Wait wait, unsigned long long* t_first = nullptr) {
  EpiRow q{0, 0, 0};
  float4 opA[8], opB[8];
  if (ok) {
    q = epi_row(e, grow);
    chunk_ops(e, q, grow, n0, opA);
  }
  wait();
#pragma unroll
  for (int cb = 0; cb < BN; cb += 64) {
    uint32_t v[32];
    tld32(tbase + (uint32_t)cb, v);
    if (ok) {
      chunk_ops(e, q, grow, n0 + cb + 32, opB);
      chunk_out<__nv_bfloat16>(e, q, opA, grow, n0 + cb, v, sc);
    }
    if (t_first && cb == 0) *t_first = gtimer();
    tld32(tbase + (uint32_t)(cb + 32), v);
    if (ok) {
      if (cb + 64 < BN) chunk_ops(e, q, grow, n0 + cb + 64, opA);
      chunk_out<__nv_bfloat16>(e, q, opB, grow, n0 + cb + 32, v, sc);
    }
  }
}

// Split on write of one output pair (c even) of the residual and SwiGLU epilogues; returns the
// pair's contribution to the row's sum of squares (residual add only).
__device__ __forceinline__ float pair_split(const EpiArgs& e, float2 op, int r, int c, float a0, float a1) {
  if (e.mode == EPI_SWIGLU) {
    const float m = silu_f(a0) * a1;
    const int cm = c >> 1;
    if (!e.sp_only) e.y[(size_t)r * e.ldy + cm] = m;
    uint16_t h, l;
    split_bf16(e.sg ? m * e.sg[cm] : m, h, l);
    reinterpret_cast<uint16_t*>(e.sp_hi)[(size_t)r * e.ldsp + cm] = h;
    reinterpret_cast<uint16_t*>(e.sp_lo)[(size_t)r * e.ldsp + cm] = l;
    return 0.f;
  }
  const bool sl = e.mode == EPI_RESID_SILU;
  const float v0 = op.x + (sl ? silu_f(a0) : a0), v1 = op.y + (sl ? silu_f(a1) : a1);
  if (!e.sp_only) *reinterpret_cast<float2*>(e.y + (size_t)r * e.ldy + c) = make_float2(v0, v1);
  const float2 g = e.sg ? *reinterpret_cast<const float2*>(e.sg + c) : make_float2(1.f, 1.f);
  uint16_t h0, h1, l0, l1;
  split_bf16(v0 * g.x, h0, l0);
  split_bf16(v1 * g.y, h1, l1);
  *reinterpret_cast<uint32_t*>(e.sp_hi + (size_t)r * e.ldsp + c) = h0 | ((uint32_t)h1 << 16);
  *reinterpret_cast<uint32_t*>(e.sp_lo + (size_t)r * e.ldsp + c) = l0 | ((uint32_t)l1 << 16);
  return v0 * v0 + v1 * v1;
}

// Cluster split-K: rank `ks` adds rows [ks * 128 / KS, ...) of the KS partial tiles (each
// [128][BN + 1] in its CTA's shared memory) and applies the pair epilogue, four items per batch
// with all loads of a batch before its stores. inv_s: the tile rows' inverse RMS (nullptr: 1);
// meta_s: the tile rows' Q/K/V metadata (position, sequence, cache slot), staged in shared memory.
// The 32 lanes of a warp hold 32 consecutive pairs of one row (BN / 2 and the thread count are
// multiples of 32), so a 32-column block's sum of squares is a reduction over 16 lanes.
template <int BN, int NT>
__device__ __forceinline__ void cluster_epilogue(const EpiArgs& e, cooperative_groups::cluster_group& cl,
                                                 float* red, int KS, int ks, int mrow0, int rbase, int M, int n0,
                                                 const float* inv_s, const EpiRow* meta_s) {
  const int RPC = kUM / KS;
  const int items = RPC * (BN / 2);
  constexpr int U = 4;
  const int lane = threadIdx.x & 31;
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
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (k < KS) {
            const float* pr = cl.map_shared_rank(red, k) + rt * (BN + 1) + c;
            s0[u] += pr[0];
            s1[u] += pr[1];
          }
        }
        if (inv_s) sc[u] = inv_s[rt];
        q[u] = meta_s[rt];
        op[u] = epi_operand(e, q[u], gr[u], col[u]);
      }
    }
    if (e.sp_hi) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        float q2 = ok[u] ? pair_split(e, op[u], gr[u], col[u], s0[u] * sc[u], s1[u] * sc[u]) : 0.f;
        if (e.ss) {  // ok[u] is the same across the warp
#pragma unroll
          for (int o = 8; o; o >>= 1) q2 += __shfl_xor_sync(0xffffffffu, q2, o);
          if (ok[u] && (lane & 15) == 0) e.ss[(size_t)gr[u] * e.ss_ld + (col[u] >> 5)] = q2;
        }
      }
    } else {
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (ok[u]) epi_out<__nv_bfloat16>(e, q[u], op[u], gr[u], col[u], s0[u] * sc[u], s1[u] * sc[u]);
    }
  }
}

// ---------------------------------------------------------------- split rows
template <bool NORM>
__global__ void __launch_bounds__(256)
k_split_rows(LinearArgs a, __nv_bfloat16* __restrict__ hi, __nv_bfloat16* __restrict__ lo,
             float* __restrict__ ss, int ss_ld) {
  TraceScope _trace(TT_SPLIT);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = gridDim.x * (blockDim.x >> 5);
  const int K = a.Kd;
  for (int rr = blockIdx.x * (blockDim.x >> 5) + warp; rr < a.groups * M; rr += nw) {
    const int grp = rr / M, r = rr - grp * M;
    const size_t row = (size_t)grp * a.Mg_stride + r;
    const float4* xr = reinterpret_cast<const float4*>(a.x + row * a.ldx);
    float sq = 0.f;
    // four 16-byte loads per lane in flight before the first conversion
    for (int k0 = 0; k0 < K / 4; k0 += 128) {
      float4 v[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int k4 = k0 + j * 32 + lane;
        v[j] = k4 < K / 4 ? xr[k4] : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int k4 = k0 + j * 32 + lane;
        if (k4 >= K / 4) continue;
        float4 w = v[j];
        if (NORM) {
          sq += w.x * w.x + w.y * w.y + w.z * w.z + w.w * w.w;
          const float4 g = reinterpret_cast<const float4*>(a.norm)[k4];
          w.x *= g.x; w.y *= g.y; w.z *= g.z; w.w *= g.w;
        }
        uint16_t h0, h1, h2, h3, l0, l1, l2, l3;
        split_bf16(w.x, h0, l0);
        split_bf16(w.y, h1, l1);
        split_bf16(w.z, h2, l2);
        split_bf16(w.w, h3, l3);
        reinterpret_cast<uint2*>(hi + row * K)[k4] = make_uint2(h0 | ((uint32_t)h1 << 16), h2 | ((uint32_t)h3 << 16));
        reinterpret_cast<uint2*>(lo + row * K)[k4] = make_uint2(l0 | ((uint32_t)l1 << 16), l2 | ((uint32_t)l3 << 16));
      }
    }
    if (NORM) {
#pragma unroll
      for (int o = 16; o; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
      if (lane == 0) ss[row * ss_ld] = sq;
    }
  }
}

// Inverse RMS of a row from its sums of squares (n slots, summed in order): one slot, or up to 32
// slots read as 16-byte vectors that are all in flight at once (n a multiple of 4).
__device__ __forceinline__ float row_inv(const float* ss, int n, int ld, size_t row, int K, float eps) {
  const float* p = ss + row * ld;
  float t = 0.f;
  if (n == 1) {
    t = p[0];
  } else {
    float4 v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = 4 * i < n ? reinterpret_cast<const float4*>(p)[i] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int i = 0; i < 8; ++i) t += (v[i].x + v[i].y) + (v[i].z + v[i].w);
    for (int i = 32; i < n; ++i) t += p[i];
  }
  return rsqrtf(t / (float)K + eps);
}

// ---------------------------------------------------------------- TMA-fed tensor-core GEMM
constexpr int kTThreads = 192;
template <int BN>
struct TCfg {
  static constexpr int kStages = BN == 256 ? 3 : 4;
  static constexpr uint32_t kABytes = kUM * kUK * 2;  // one half (hi or lo) of an A tile
  static constexpr uint32_t kWBytes = BN * kUK * 2;
  static constexpr uint32_t kStageBytes = 2 * kABytes + kWBytes;
  // D fp32, A and B bf16, both K-major, M = 128, N = BN
  static constexpr uint32_t kIDesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                                     ((uint32_t)(kUM >> 4) << 24);
  // ring, barriers, TMEM address, the tile rows' inverse RMS, alignment slack
  static constexpr size_t kSmem =
      (size_t)kStages * kStageBytes + (2 * kStages + 1) * 8 + 16 + kUM * 4 + 32 + kUM * sizeof(EpiRow) + 1024;
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
        const __grid_constant__ CUtensorMap tmAl, const float* __restrict__ ss, int ss_n, int ss_ld, int MT,
        int KS) {
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
  float* inv_s = reinterpret_cast<float*>(accdone + 1) + 4;  // [128]
  // traced launches (one epilogue thread, first row tile): epilogue done, accumulator ready
  unsigned long long* tmk = reinterpret_cast<unsigned long long*>(inv_s + kUM);
  EpiRow* meta_s = reinterpret_cast<EpiRow*>(tmk + 4);  // [128]
  float* red = reinterpret_cast<float*>(ring);  // [128][BN + 1] after the MMAs of a pass

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * BN;
  const int ks = blockIdx.y;
  const int grp = blockIdx.z / MT, mt0 = blockIdx.z % MT;
  const int rbase = grp * a.Mg_stride;
  const int nkb = a.Kd / kUK / KS;
  const int kb0 = ks * nkb;
  const int wrow = grp * a.N + n0;

  if (tid == 0) {
    for (int i = 0; i < C::kStages; ++i) {
      ubar_init(&full[i], 1);
      ubar_init(&empty[i], 1);
    }
    tmk[0] = tmk[1] = tmk[2] = 0;
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
  const int ntm = (M + kUM - 1) / kUM;
  // row tiles mt0, mt0 + MT, ...; a first pass always runs (it consumes the copies issued above)
  int npass = (ntm - mt0 + MT - 1) / MT;
  if (npass < 1) npass = 1;
  bool failed = false;
  uint32_t issued = pre;
  if (tid == 0) {
    const int arow = rbase + mt0 * kUM;
    for (int i = 0; i < pre; ++i) {
      unsigned char* st = ring + (size_t)i * C::kStageBytes;
      tma_load_2d(st, &tmAh, (kb0 + i) * kUK, arow, &full[i]);
      tma_load_2d(st + C::kABytes, &tmAl, (kb0 + i) * kUK, arow, &full[i]);
    }
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                 "r"(BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  const int r = ((warp & 3) << 5) | lane;  // epilogue row = TMEM lane

  for (int ps = 0; ps < npass; ++ps) {
    const int mt = mt0 + ps * MT;
    const bool live = mt * kUM < M;  // the same for every CTA of a cluster
    const int arow = rbase + mt * kUM;
    const uint32_t kbase = (uint32_t)ps * nkb;  // K blocks of earlier passes (ring phases)
    if (warp == 0) {
      if (lane == 0) {
        for (int kb = (ps == 0 ? pre : 0); kb < nkb; ++kb) {
          const uint32_t it = kbase + kb;
          const int s = it % C::kStages;
          if (it >= (uint32_t)C::kStages) wait_or_fail(&empty[s], ((it / C::kStages) - 1) & 1, failed);
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
        // traced launches mark the end of the first main loop
        if (g_trace && ps == 0) {
          wait_or_fail(accdone, 0, failed);
          _trace.mark();
        }
      }
    } else if (warp == 1) {
      if (lane == 0) {
        for (int kb = 0; kb < nkb; ++kb) {
          const uint32_t it = kbase + kb;
          const int s = it % C::kStages;
          wait_or_fail(&full[s], (it / C::kStages) & 1, failed);
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
    } else if (!live) {
      wait_or_fail(accdone, ps & 1, failed);
    }
    __syncwarp();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (live) {
      // the row's inverse RMS, read while the main loop runs
      float sc = 1.f;
      if (warp >= 2 && a.norm && mt * kUM + r < M) sc = row_inv(ss, ss_n, ss_ld, rbase + mt * kUM + r, a.Kd, a.eps);
      if (KS == 1) {
        if (warp >= 2) {
          const int row = mt * kUM + r;
          // the accumulator wait sits inside, after the first chunk's operand loads
          tile_epilogue<BN>(a.epi, tmem + ((uint32_t)((warp & 3) * 32) << 16), rbase + row, row < M, n0, sc, [&] {
                              wait_or_fail(accdone, ps & 1, failed);
                              asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                              if (g_trace && ps == 0 && warp == 2 && lane == 0) tmk[1] = gtimer();
                            },
                            (g_trace && ps == 0 && warp == 2 && lane == 0) ? &tmk[2] : nullptr);
          if (g_trace && ps == 0 && warp == 2 && lane == 0) tmk[0] = gtimer();
        }
      } else {
        cgr::cluster_group cl = cgr::this_cluster();
        if (warp >= 2) {
          // the rows' metadata is read while the main loop runs; then the accumulator
          inv_s[r] = sc;
          meta_s[r] = mt * kUM + r < M ? epi_row(a.epi, rbase + mt * kUM + r) : EpiRow{0, 0, 0, 0};
          wait_or_fail(accdone, ps & 1, failed);
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          if (g_trace && ps == 0 && warp == 2 && lane == 0) tmk[1] = gtimer();
#pragma unroll
          for (int cb = 0; cb < BN; cb += 32) {
            uint32_t v[32];
            tld32(tmem + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)cb, v);
#pragma unroll
            for (int q = 0; q < 32; ++q) red[r * (BN + 1) + cb + q] = __uint_as_float(v[q]);
          }
        }
        cl.sync();
        cluster_epilogue<BN, kTThreads>(a.epi, cl, red, KS, ks, mt * kUM, rbase, M, n0, a.norm ? inv_s : nullptr,
                                        meta_s);
        if (g_trace && ps == 0 && warp == 2 && lane == 0) tmk[0] = gtimer();
        cl.sync();
      }
    }
    // this pass's TMEM reads and reduction-buffer use end before the next pass's MMAs and copies
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  }
  // after a failed wait, copies may still be in flight: wait (bounded) for the last one issued
  // into each stage before the CTA's shared memory is released
  if (g_trace) {
    _trace.mark_at(0, tmk[2] ? tmk[2] : tmk[1]);
    _trace.mark_at(1, tmk[1]);
    _trace.mark_at(2, tmk[0]);
  }
  const bool any_failed = __syncthreads_or(failed);
  if (tid == 0 && any_failed) {
    for (uint32_t s = 0; s < (uint32_t)C::kStages && s < issued; ++s) {
      const uint32_t last = issued - 1 - ((issued - 1 - s) % C::kStages);
      ubar_wait(&full[last % C::kStages], (last / C::kStages) & 1);
    }
    atomicOr(a.epi.err, kErrTimeout | kErrWaitGemm);
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(BN) : "memory");
}

// ---------------------------------------------------------------- skinny GEMM (few rows)
// For a few rows the roles swap: the tile computes Y^T [128 output columns][NR rows] =
// W [128][K] . X [NR][K]^T, with the weights as the MMA's A operand (M = 128) and the split
// activations as its B operand (N = NR). A stage then moves 16 KB of weights and only NR rows of
// activations, K is split across a cluster of up to 16 CTAs so that every CTA's weight slice fits
// its ring (all of it copied before the grid-dependency wait), and the epilogue sees one output
// column per thread (TMEM lane) and the rows along the TMEM columns: warp-wide stores per row, and
// the rotary and SwiGLU pairs are adjacent lanes.
constexpr int kSW = 128;  // output columns per tile (UMMA M)

template <int NR>
struct SCfg {
  static constexpr uint32_t kWBytes = kSW * kUK * 2;  // 16 KB
  static constexpr uint32_t kXBytes = NR * kUK * 2;   // one half (hi or lo) of an activation tile
  static constexpr uint32_t kStageBytes = kWBytes + 2 * kXBytes;
  // split-K partials pushed to the rank that finishes them: [KS source ranks][NR / KS rows][128]
  static constexpr uint32_t kRecvBytes = NR * kSW * 4;
  // about 104 KB in all, so that a CTA of the next layer's kernel fits beside one of this kernel
  // on an SM and copies its weights while this one finishes: 3 stages (NR 32), 2 (NR 64)
  static constexpr int kStages = (104 * 1024 - kRecvBytes) / kStageBytes;
  // D fp32, A and B bf16, both K-major, M = 128, N = NR
  static constexpr uint32_t kIDesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(NR >> 3) << 17) |
                                     ((uint32_t)(kSW >> 4) << 24);
  static constexpr uint32_t kTmemCols = NR < 32 ? 32 : NR;
  // ring, receive buffer, barriers (full, empty, accumulator, receive), TMEM address, per-row
  // inverse RMS / position / sequence / cache slot / its page, two trace times, alignment slack
  static constexpr size_t kSmem =
      (size_t)kStages * kStageBytes + kRecvBytes + (2 * kStages + 2) * 8 + 16 + NR * 20 + 16 + 1024;
  static_assert(NR == 32 || NR == 64, "tile rows");
  static_assert(kStages >= 2, "ring");
  static_assert(kStageBytes % 1024 == 0 && kXBytes % 1024 == 0, "swizzle atoms");
  static_assert(kSmem <= 112 * 1024, "two CTAs per SM");
};

template <int NR>
__device__ __forceinline__ void smma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(SCfg<NR>::kIDesc), "r"(accumulate)
      : "memory");
}

// Per-row tile metadata in shared memory.
struct SRowMeta {
  float* inv;
  int* pos;
  int* b;
  int* slot;
  int* pg;
};

// Output of value x (accumulator times the row's scale) at global row gr, column c, for one lane
// of a warp whose 32 lanes hold 32 consecutive columns of the same row; op is the residual value
// (residual modes), gc the consumer's RMSNorm gain of column c (split on write of a residual
// output). Every lane of the warp calls it (shuffles).
__device__ __forceinline__ void scol_out(const EpiArgs& e, size_t gr, int c, int lane, float x, float op,
                                         float gc, const SRowMeta& m, int rt) {
  switch (e.mode) {
    case EPI_STORE:
      e.y[gr * e.ldy + c] = x;
      break;
    case EPI_RESID:
    case EPI_RESID_SILU: {
      const float y = op + (e.mode == EPI_RESID_SILU ? silu_f(x) : x);
      if (!e.sp_only) e.y[gr * e.ldy + c] = y;
      if (e.sp_hi) {
        uint16_t h, l;
        split_bf16(y * gc, h, l);
        reinterpret_cast<uint16_t*>(e.sp_hi)[gr * e.ldsp + c] = h;
        reinterpret_cast<uint16_t*>(e.sp_lo)[gr * e.ldsp + c] = l;
        if (e.ss) {
          float q2 = y * y;
#pragma unroll
          for (int o = 16; o; o >>= 1) q2 += __shfl_xor_sync(0xffffffffu, q2, o);
          if (lane == 0) e.ss[gr * e.ss_ld + (c >> 5)] = q2;
        }
      }
      break;
    }
    case EPI_SWIGLU: {
      // interleaved (gate, up) columns: the even lane of a pair holds the gate
      const float u = __shfl_xor_sync(0xffffffffu, x, 1);
      if (!(lane & 1)) {
        const float mv = silu_f(x) * u;
        const int cm = c >> 1;
        if (!e.sp_only) e.y[gr * e.ldy + cm] = mv;
        if (e.sp_hi) {
          uint16_t h, l;
          split_bf16(e.sg ? mv * e.sg[cm] : mv, h, l);
          reinterpret_cast<uint16_t*>(e.sp_hi)[gr * e.ldsp + cm] = h;
          reinterpret_cast<uint16_t*>(e.sp_lo)[gr * e.ldsp + cm] = l;
        }
      }
      break;
    }
    case EPI_QKV: {
      const int part = c / e.d;  // the same across the warp (d is a multiple of 32)
      const int cc = c - part * e.d;
      const int h = cc / e.hd;
      const int dd = cc - h * e.hd;
      if (part < 2) {
        // interleaved rotary pairs (2i, 2i + 1) in adjacent lanes
        const float p = __shfl_xor_sync(0xffffffffu, x, 1);
        const float2 cs = e.rope[(size_t)m.pos[rt] * (e.hd >> 1) + (dd >> 1)];
        x = (lane & 1) ? p * cs.y + x * cs.x : x * cs.x - p * cs.y;
      }
      if (part == 0) {
        e.y[gr * e.ldy + cc] = x;
      } else {
        const int slot = m.slot[rt], pg = m.pg[rt];
        if (!kv_write_ok(e.kv, slot, pg)) {
          if (lane == 0) atomicOr(e.err, kErrIndex);
        } else {
          __nv_bfloat16* base = reinterpret_cast<__nv_bfloat16*>(part == 1 ? e.kv.k : e.kv.v);
          base[kv_addr(e.kv, e.H, e.hd, m.b[rt], h, slot, pg) + dd] = __float2bfloat16_rn(x);
        }
      }
      break;
    }
  }
}

__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait;" ::: "memory"); }

__device__ __forceinline__ uint32_t mapa_u32(uint32_t saddr, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}

// Cluster split-K of the skinny tile, push side: rank ks owns tile rows [ks * RPC, (ks + 1) * RPC)
// (RPC = NR / KS). An epilogue thread (one output column) reads its column of the accumulator and
// stores each row's partial into the owning rank's receive buffer, slot ks (its own rows into its
// own buffer with plain stores).
template <int NR, int KS>
__device__ __forceinline__ void spush(float* recv, int ks, uint32_t tlane, int col) {
  constexpr int RPC = NR / KS;
  const uint32_t lbase = su32(recv);
#pragma unroll 1
  for (int j0 = 0; j0 < NR; j0 += 32) {
    uint32_t v[32];
    tld32(tlane + (uint32_t)j0, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int rt = j0 + i, k = rt / RPC, r = rt - k * RPC;
      const uint32_t off = (uint32_t)(((ks * RPC + r) * kSW + col) * 4);
      if (k == ks) recv[(ks * RPC + r) * kSW + col] = __uint_as_float(v[i]);
      else st_cluster_f32(mapa_u32(lbase + off, k), __uint_as_float(v[i]));
    }
  }
}

// Finish side: the rank's rows, each the sum of the KS slots of the receive buffer (in rank
// order). Once every sum is in registers the thread arrives (relaxed: its reads of the buffer have
// returned, the sums use them) on the cluster barrier that closes the pass, then writes the rows.
template <int NR, int KS>
__device__ __forceinline__ void sfinish(const LinearArgs& a, const float* recv, const SRowMeta& meta, int ks, int mt,
                                        int rbase, int M, int c, int col, int lane) {
  constexpr int RPC = NR / KS;
  const bool resid = a.epi.mode == EPI_RESID || a.epi.mode == EPI_RESID_SILU;
  const float gc = (resid && a.epi.sp_hi && a.epi.sg) ? a.epi.sg[c] : 1.f;
  const int nrow = min(RPC, M - (mt * NR + ks * RPC));  // rows of this rank (may be <= 0)
  float op[RPC], acc[RPC];
#pragma unroll
  for (int i = 0; i < RPC; ++i) {
    const int row = mt * NR + ks * RPC + i;
    op[i] = resid && i < nrow ? a.epi.res[(size_t)(rbase + row) * a.epi.ldres + c] : 0.f;
    acc[i] = 0.f;
#pragma unroll
    for (int k = 0; k < KS; ++k) acc[i] += recv[(k * RPC + i) * kSW + col];
  }
  float dep = 0.f;
#pragma unroll
  for (int i = 0; i < RPC; ++i) dep += acc[i];
  asm volatile("barrier.cluster.arrive.relaxed;" ::"f"(dep) : "memory");
#pragma unroll
  for (int i = 0; i < RPC; ++i) {
    if (i >= nrow) break;  // the same across the warp
    const int rt = ks * RPC + i;
    scol_out(a.epi, (size_t)(rbase + mt * NR + rt), c, lane, acc[i] * meta.inv[rt], op[i], gc, meta, rt);
  }
}

template <int NR>
__global__ void __launch_bounds__(kTThreads, 2)
k_sgemm(LinearArgs a, const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmXh,
        const __grid_constant__ CUtensorMap tmXl, const float* __restrict__ ss, int ss_n, int ss_ld, int MT,
        int KS) {
  using C = SCfg<NR>;
  namespace cgr = cooperative_groups;
  TraceScope _trace(TT_SGEMM);
  extern __shared__ __align__(1024) unsigned char ssm_raw[];
  unsigned char* ring =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(ssm_raw) + 1023) & ~uintptr_t(1023));
  float* recv = reinterpret_cast<float*>(ring + C::kStages * C::kStageBytes);
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + C::kStages * C::kStageBytes + C::kRecvBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* accdone = empty + C::kStages;
  uint64_t* rbar = accdone + 1;  // the rank's rows: one arrival per peer
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rbar + 1);
  SRowMeta meta;
  meta.inv = reinterpret_cast<float*>(rbar + 1) + 4;
  meta.pos = reinterpret_cast<int*>(meta.inv + NR);
  meta.b = meta.pos + NR;
  meta.slot = meta.b + NR;
  meta.pg = meta.slot + NR;
  // traced launches: partials pushed, peers' partials received
  unsigned long long* tmk = reinterpret_cast<unsigned long long*>(meta.pg + NR);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * kSW;
  const int ks = blockIdx.y;
  const int grp = blockIdx.z / MT, mt0 = blockIdx.z % MT;
  const int rbase = grp * a.Mg_stride;
  const int nkb = a.Kd / kUK / KS;
  const int kb0 = ks * nkb;
  const int wrow = grp * a.N + n0;

  if (tid == 0) {
    for (int i = 0; i < C::kStages; ++i) {
      ubar_init(&full[i], 1);
      ubar_init(&empty[i], 1);
    }
    ubar_init(accdone, 1);
    ubar_init(rbar, KS > 1 ? KS - 1 : 1);
    tmk[0] = tmk[1] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
  }
  __syncthreads();
  // the peers' receive barriers are initialised before anyone pushes (before the dependency
  // wait, so this overlaps the previous kernel)
  if (KS > 1) cooperative_groups::this_cluster().sync();
  // weights never change: the weight part of the first stages (all of them when the slice fits
  // the ring) is copied before the dependency wait
  const int pre = nkb < C::kStages ? nkb : C::kStages;
  if (tid == 0) {
    for (int i = 0; i < pre; ++i) {
      ubar_expect(&full[i], C::kStageBytes);
      unsigned char* st = ring + (size_t)i * C::kStageBytes;
      tma_load_2d(st, &tmW, (kb0 + i) * kUK, wrow, &full[i]);
      tma_load_2d(st + 8192, &tmW, (kb0 + i) * kUK, wrow + 64, &full[i]);
    }
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  int M = *a.M;
  M = M < a.M_cap ? M : a.M_cap;
  const int ntm = (M + NR - 1) / NR;
  int npass = (ntm - mt0 + MT - 1) / MT;
  if (npass < 1) npass = 1;
  bool failed = false;
  uint32_t issued = pre;
  if (tid == 0) {
    const int xrow = rbase + mt0 * NR;
    for (int i = 0; i < pre; ++i) {
      unsigned char* st = ring + (size_t)i * C::kStageBytes;
      tma_load_2d(st + C::kWBytes, &tmXh, (kb0 + i) * kUK, xrow, &full[i]);
      tma_load_2d(st + C::kWBytes + C::kXBytes, &tmXl, (kb0 + i) * kUK, xrow, &full[i]);
    }
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                 "r"(C::kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  const int eq = warp & 3;                 // TMEM lane quarter of an epilogue warp
  const int c = n0 + eq * 32 + lane;       // output column of an epilogue thread
  const uint32_t tlane = tmem + ((uint32_t)(eq * 32) << 16);
  const int et = (warp - 2) * 32 + lane;   // epilogue thread 0..127

  for (int ps = 0; ps < npass; ++ps) {
    const int mt = mt0 + ps * MT;
    const bool live = mt * NR < M;  // the same for every CTA of a cluster
    const int xrow = rbase + mt * NR;
    const uint32_t kbase = (uint32_t)ps * nkb;
    if (warp == 0) {
      if (lane == 0) {
        for (int kb = (ps == 0 ? pre : 0); kb < nkb; ++kb) {
          const uint32_t it = kbase + kb;
          const int s = it % C::kStages;
          if (it >= (uint32_t)C::kStages) wait_or_fail(&empty[s], ((it / C::kStages) - 1) & 1, failed);
          if (failed) break;
          ++issued;
          unsigned char* st = ring + (size_t)s * C::kStageBytes;
          ubar_expect(&full[s], C::kStageBytes);
          tma_load_2d(st + C::kWBytes, &tmXh, (kb0 + kb) * kUK, xrow, &full[s]);
          tma_load_2d(st + C::kWBytes + C::kXBytes, &tmXl, (kb0 + kb) * kUK, xrow, &full[s]);
          tma_load_2d(st, &tmW, (kb0 + kb) * kUK, wrow, &full[s]);
          tma_load_2d(st + 8192, &tmW, (kb0 + kb) * kUK, wrow + 64, &full[s]);
        }
        if (g_trace && ps == 0) {
          wait_or_fail(accdone, 0, failed);
          _trace.mark();
        }
      }
    } else if (warp == 1) {
      if (lane == 0) {
        for (int kb = 0; kb < nkb; ++kb) {
          const uint32_t it = kbase + kb;
          const int s = it % C::kStages;
          wait_or_fail(&full[s], (it / C::kStages) & 1, failed);
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t wb = su32(ring + (size_t)s * C::kStageBytes);
          const uint32_t xh = wb + C::kWBytes, xl = xh + C::kXBytes;
          if (live && !failed) {
#pragma unroll
            for (int k = 0; k < kUK / 16; ++k) {
              smma<NR>(tmem, sdesc(wb + k * 32), sdesc(xh + k * 32), (kb > 0 || k > 0) ? 1u : 0u);
              smma<NR>(tmem, sdesc(wb + k * 32), sdesc(xl + k * 32), 1u);
            }
            umma_commit(&empty[s]);
          } else {
            ubar_arrive(&empty[s]);
          }
        }
        if (live) umma_commit(accdone);
        else ubar_arrive(accdone);
      }
    } else {
      // rows' metadata of this tile: inverse RMS, and for Q/K/V the position, sequence and slot
      if (et < NR) {
        const int row = mt * NR + et;
        float inv = 1.f;
        if (row < M) {
          if (a.norm) inv = row_inv(ss, ss_n, ss_ld, rbase + row, a.Kd, a.eps);
          if (a.epi.mode == EPI_QKV) {
            meta.pos[et] = a.epi.rows.pos[rbase + row];
            meta.b[et] = a.epi.rows.b[rbase + row];
            meta.slot[et] = a.epi.rows.slot[rbase + row];
            meta.pg[et] = a.epi.kv.pt ? a.epi.rows.page[rbase + row] : 0;
          }
        }
        meta.inv[et] = inv;
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (live && KS == 1) {
        const bool resid = a.epi.mode == EPI_RESID || a.epi.mode == EPI_RESID_SILU;
        const float gc = (resid && a.epi.sp_hi && a.epi.sg) ? a.epi.sg[c] : 1.f;
        for (int j0 = 0; j0 < NR; j0 += 32) {
          if (mt * NR + j0 >= M) break;
          float op[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int row = mt * NR + j0 + i;
            op[i] = resid && row < M ? a.epi.res[(size_t)(rbase + row) * a.epi.ldres + c] : 0.f;
          }
          if (j0 == 0) {
            wait_or_fail(accdone, ps & 1, failed);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          }
          uint32_t v[32];
          tld32(tlane + (uint32_t)j0, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int rt = j0 + i;
            if (mt * NR + rt >= M) break;  // the same across the warp
            scol_out(a.epi, (size_t)(rbase + mt * NR + rt), c, lane, __uint_as_float(v[i]) * meta.inv[rt], op[i],
                     gc, meta, rt);
          }
        }
      }
    }
    __syncwarp();
    if (live && KS > 1) {
      // push the partials to their owners; the owner waits for its KS - 1 peers and finishes its
      // rows; a cluster barrier closes the pass (no CTA refills a receive buffer, or exits while a
      // peer may still write to it, before every CTA has read its rows)
      if (warp >= 2) {
        wait_or_fail(accdone, ps & 1, failed);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        switch (KS) {
          case 2: spush<NR, 2>(recv, ks, tlane, eq * 32 + lane); break;
          case 4: spush<NR, 4>(recv, ks, tlane, eq * 32 + lane); break;
          case 8: spush<NR, 8>(recv, ks, tlane, eq * 32 + lane); break;
          default: spush<NR, 16>(recv, ks, tlane, eq * 32 + lane); break;
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (g_trace && et == 0 && ps == 0) tmk[0] = gtimer();
        if (et == 0) {
          // one cluster-scope fence orders every epilogue thread's pushes (they precede the barrier)
          // before the relaxed arrivals on the owners' barriers
          asm volatile("fence.acq_rel.cluster;" ::: "memory");
          for (int k = 1; k < KS; ++k) {
            const int peer = (ks + k) % KS;
            asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(
                             mapa_u32(su32(rbar), peer))
                         : "memory");
          }
          bool ok = false;
          for (int it = 0; it < kUSpins && !ok; ++it) {
            uint32_t done;
            asm volatile(
                "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
                " selp.u32 %0, 1, 0, p;\n}"
                : "=r"(done)
                : "r"(su32(rbar)), "r"((uint32_t)(ps & 1))
                : "memory");
            ok = done != 0;
          }
          if (!ok) failed = true;
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (g_trace && et == 0 && ps == 0) tmk[1] = gtimer();
        switch (KS) {
          case 2: sfinish<NR, 2>(a, recv, meta, ks, mt, rbase, M, c, eq * 32 + lane, lane); break;
          case 4: sfinish<NR, 4>(a, recv, meta, ks, mt, rbase, M, c, eq * 32 + lane, lane); break;
          case 8: sfinish<NR, 8>(a, recv, meta, ks, mt, rbase, M, c, eq * 32 + lane, lane); break;
          default: sfinish<NR, 16>(a, recv, meta, ks, mt, rbase, M, c, eq * 32 + lane, lane); break;
        }
      } else {
        asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory");
      }
      cluster_wait();
    }
    // this pass's TMEM reads, reduction-buffer and metadata use end before the next pass
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  }
  if (g_trace) {
    _trace.mark_at(1, tmk[0]);
    _trace.mark_at(2, tmk[1]);
  }
  const bool any_failed = __syncthreads_or(failed);
  if (tid == 0 && any_failed) {
    for (uint32_t s = 0; s < (uint32_t)C::kStages && s < issued; ++s) {
      const uint32_t last = issued - 1 - ((issued - 1 - s) % C::kStages);
      ubar_wait(&full[last % C::kStages], (last / C::kStages) & 1);
    }
    atomicOr(a.epi.err, kErrTimeout | kErrWaitGemm);
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::kTmemCols)
                 : "memory");
}

template <int NR>
void sgemm_go(const LinearArgs& a, const CUtensorMap& tw, const CUtensorMap& th, const CUtensorMap& tl,
              const float* ss, int ss_n, int ss_ld, int MT, int KS, cudaStream_t s) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(a.N / kSW, KS, a.groups * MT);
  cfg.blockDim = dim3(kTThreads);
  cfg.dynamicSmemBytes = SCfg<NR>::kSmem;
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
  cudaLaunchKernelEx(&cfg, k_sgemm<NR>, a, tw, th, tl, ss, ss_n, ss_ld, MT, KS);
}

template <int BN>
void tgemm_go(const LinearArgs& a, const CUtensorMap& tw, const CUtensorMap& th, const CUtensorMap& tl,
              const float* ss, int ss_n, int ss_ld, int MT, int KS, cudaStream_t s) {
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
  cudaLaunchKernelEx(&cfg, k_tgemm<BN>, a, tw, th, tl, ss, ss_n, ss_ld, MT, KS);
}

PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess && fn)
      encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  return encode;
}

int encode_bf16_2d(void* out, const void* base, long long rows, long long K, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
  if (!encode) return LCA_E_CUDA;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kUK, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = encode(reinterpret_cast<CUtensorMap*>(out), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                            const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LCA_OK : LCA_E_CUDA;
}

}  // namespace

// Split rows (unless the producing layer's epilogue already did), then the TMA-fed GEMM. The rows'
// sums of squares (for the RMSNorm) sit in ss[row * ss_ld + i]: one slot from k_split_rows, Kd / 32
// per-block slots from a producing epilogue. The grid covers the typical row count (rows_typ). Tile width
// BN (256, 128 or 64, dividing N) and K split KS (power of two, at most 8, at least two 64-deep
// blocks per CTA, while the grid fits one wave) minimise a simple cost: waves x (BN x K blocks
// per CTA + a fixed part) + a cluster-reduction term proportional to BN; ties go to the wider tile.
void split_gemm(const Dev& D, const LinearArgs& a, const void* amap, __nv_bfloat16* hi, __nv_bfloat16* lo,
                float* ss, int ss_ld, cudaStream_t s) {
  const int sms = D.num_sms > 0 ? D.num_sms : 148;
  const int ss_n = a.presplit ? a.Kd / 32 : 1;
  if (!a.presplit) {
    // a warp per row; the grid covers the typical rows and its warps walk any further ones
    const int need = a.groups * (a.rows_typ > 0 ? std::min(a.rows_typ, a.M_cap) : a.M_cap);
    const int blocks = std::max(1, std::min((need + 7) / 8, 4 * sms));
    ++g_launches;
    if (a.norm) launch_pdl(k_split_rows<true>, dim3(blocks), dim3(256), 0, s, a, hi, lo, ss, ss_ld);
    else launch_pdl(k_split_rows<false>, dim3(blocks), dim3(256), 0, s, a, hi, lo, ss, ss_ld);
  }
  const int rows_typ = a.rows_typ > 0 ? a.rows_typ : a.M_cap;
  if (rows_typ <= D.sgemm_max_rows && a.N % kSW == 0) {
    // skinny: NR rows per tile; K split (power of two, at most sgemm_max_ks, dividing the K
    // blocks and NR) as far as the grid fits one wave of two CTAs per SM
    const int NR = rows_typ <= 32 ? 32 : 64;
    const int mtc = (a.M_cap + NR - 1) / NR;
    const int MT = std::max(1, std::min((rows_typ + NR - 1) / NR, mtc));
    const int kb = a.Kd / kUK;
    const long long base = (long long)(a.N / kSW) * a.groups * MT;
    int KS = 1;
    // two CTAs fit an SM (about 96 KB of ring each)
    while (2 * KS <= D.sgemm_max_ks && kb % (2 * KS) == 0 && NR % (2 * KS) == 0 && base * 2 * KS <= 2 * sms)
      KS *= 2;
    CUtensorMap tw, th, tl;
    const int mo = NR == 32 ? 256 : 512;
    memcpy(&tw, a.tmap, sizeof(tw));
    memcpy(&th, static_cast<const unsigned char*>(amap) + mo, sizeof(th));
    memcpy(&tl, static_cast<const unsigned char*>(amap) + mo + 128, sizeof(tl));
    if (NR == 32) sgemm_go<32>(a, tw, th, tl, ss, ss_n, ss_ld, MT, KS, s);
    else sgemm_go<64>(a, tw, th, tl, ss, ss_n, ss_ld, MT, KS, s);
    return;
  }
  const int mt_cap = (a.M_cap + kUM - 1) / kUM;
  int MT = (rows_typ + kUM - 1) / kUM;
  MT = MT < 1 ? 1 : (MT > mt_cap ? mt_cap : MT);
  const int kb = a.Kd / kUK;
  int best_bn = 64, best_ks = 1;
  long long best = -1;
  static const int bn_only = [] {
    const char* e = getenv("LCA_TGEMM_BN");
    return e ? atoi(e) : 0;
  }();
  for (int bn : {256, 128, 64}) {
    if (a.N % bn || (bn_only && bn != bn_only)) continue;
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
  if (best_bn == 256) tgemm_go<256>(a, tw, th, tl, ss, ss_n, ss_ld, MT, best_ks, s);
  else if (best_bn == 128) tgemm_go<128>(a, tw, th, tl, ss, ss_n, ss_ld, MT, best_ks, s);
  else tgemm_go<64>(a, tw, th, tl, ss, ss_n, ss_ld, MT, best_ks, s);
}

// Tensor map of a bf16 weight [rows][K] (K innermost) with 64 x 64 boxes and the 128-byte swizzle.
int make_weight_tmap(void* out, const void* W, long long rows, long long K) {
  if (K % kUK || rows % kUN) return LCA_E_ARG;
  return encode_bf16_2d(out, W, rows, K, kUN);
}

// Tensor maps (hi, lo) of the split activations [rows][K] bf16 with 128-byte swizzle and K boxes of
// 64: 128-row boxes (at 0), 32-row boxes (at 256) and 64-row boxes (at 512).
int make_split_tmaps(void* out, const void* hi, const void* lo, long long rows, long long K) {
  if (K % kUK || rows < 1) return LCA_E_ARG;
  unsigned char* o = static_cast<unsigned char*>(out);
  const int boxes[3] = {kUM, 32, 64};
  for (int i = 0; i < 3; ++i) {
    int st = encode_bf16_2d(o + 256 * i, hi, rows, K, boxes[i]);
    if (st == LCA_OK) st = encode_bf16_2d(o + 256 * i + 128, lo, rows, K, boxes[i]);
    if (st != LCA_OK) return st;
  }
  return LCA_OK;
}

template <int NR>
int sgemm_attrs() {
  cudaFuncSetAttribute(k_sgemm<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SCfg<NR>::kSmem);
  cudaFuncSetAttribute(k_sgemm<NR>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  // can the GPU hold a 16-CTA cluster of this kernel at all?
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(8, 16, 1);
  cfg.blockDim = dim3(kTThreads);
  cfg.dynamicSmemBytes = SCfg<NR>::kSmem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 16;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int nc = 0;
  if (cudaOccupancyMaxActiveClusters(&nc, k_sgemm<NR>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    nc = 0;
  }
  return nc;
}

// Kernel attributes; with D, the skinny GEMM's largest K split (16 only if 16-CTA clusters of
// every tile height fit; environment LCA_SGEMM_MAX_KS lowers it) and its row limit (environment
// LCA_SGEMM_MAX_ROWS, default 64).
void kernel_attrs_umma(Dev* D) {
  cudaFuncSetAttribute(k_tgemm<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TCfg<64>::kSmem);
  cudaFuncSetAttribute(k_tgemm<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TCfg<128>::kSmem);
  cudaFuncSetAttribute(k_tgemm<256>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TCfg<256>::kSmem);
  const int c32 = sgemm_attrs<32>(), c64 = sgemm_attrs<64>();
  if (D) {
    D->sgemm_max_ks = (c32 > 0 && c64 > 0) ? 16 : 8;
    const char* k = getenv("LCA_SGEMM_MAX_KS");
    if (k) D->sgemm_max_ks = std::max(1, std::min(D->sgemm_max_ks, atoi(k)));
    const char* e = getenv("LCA_SGEMM_MAX_ROWS");
    D->sgemm_max_rows = e ? std::max(0, std::min(256, atoi(e))) : 64;
  }
}

// The tensor cores take a layer that has a weight tensor map and split-activation maps for its K,
// whose rows fit the split buffers and whose shape fits the tiles.
bool umma_ready(const Dev& D, const LinearArgs& a) {
  if (!D.use_umma || !a.tmap || !a.amap || D.dtype != LCA_BF16 || a.N % kUN || a.Kd % kUK) return false;
  if (a.abuf < 0 || a.abuf > 1 || (a.presplit && a.norm && a.Kd / 32 > D.as_ss_ld)) return false;
  return (long long)a.groups * a.M_cap <= D.as_rows;
}

// Launch on the tensor cores if umma_ready; false otherwise.
bool linear_umma(const Dev& D, const LinearArgs& a, cudaStream_t s) {
  if (!umma_ready(D, a)) return false;
  split_gemm(D, a, a.amap, D.as_hi[a.abuf], D.as_lo[a.abuf], D.as_ss, D.as_ss_ld, s);
  return true;
}

LCA_TRACE_SETTER(trace_set_umma)

}  // namespace lca

using namespace lca;

extern "C" size_t lca_debug_gemm_scratch_bytes(int32_t M, int32_t K) {
  if (M < 1 || K < 1) return 0;
  return (size_t)M * K * 2 * 2 + (size_t)M * 4 + 512;  // hi, lo, one sum-of-squares slot per row
}

extern "C" int lca_debug_gemm(const float* x, const void* W, float* y, int32_t M, int32_t N, int32_t K,
                              const int32_t* M_dev, int32_t rows_typ, int32_t* err_dev, void* scratch,
                              void* stream) {
  if (!x || !W || !y || !M_dev || !err_dev || !scratch || M < 1 || N < 1 || K < 1 || rows_typ < 0 ||
      rows_typ > M || N % kUN || K % kUK)
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
  kernel_attrs_umma(&D);
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
  a.epi.err = err_dev;
  char* p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(scratch) + 255) & ~uintptr_t(255));
  __nv_bfloat16* hi = reinterpret_cast<__nv_bfloat16*>(p);
  __nv_bfloat16* lo = hi + (size_t)M * K;
  float* ss = reinterpret_cast<float*>(lo + (size_t)M * K);
  alignas(64) unsigned char maps[kSplitMapBytes];
  st = make_split_tmaps(maps, hi, lo, M, K);
  if (st != LCA_OK) return st;
  split_gemm(D, a, maps, hi, lo, ss, 1, reinterpret_cast<cudaStream_t>(stream));
  return cudaGetLastError() == cudaSuccess ? LCA_OK : LCA_E_CUDA;
}
