// Epilogues of the linear layers, shared by the CUDA-core and tensor-core kernels: residual add,
// SwiGLU, residual SiLU (MLP head), and Q/K/V with rotary embedding and the KV-cache append.
#pragma once
#include "common.cuh"

namespace lca {

// SiLU with the fast exponential and division intrinsics (a few ulp; for x -> -inf the divisor
// overflows to inf and the quotient is 0)
static __device__ __forceinline__ float silu_f(float x) { return __fdividef(x, 1.0f + __expf(-x)); }

static __device__ __forceinline__ void store_cache(float* p, float v) { *p = v; }
static __device__ __forceinline__ void store_cache(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

// Epilogue of one pair of adjacent output columns (c even) of row r.
template <typename TC>
static __device__ __forceinline__ void epi_pair(const EpiArgs& e, int r, int c, float a0, float a1) {
  switch (e.mode) {
    case EPI_STORE: {
      float* y = e.y + (size_t)r * e.ldy + c;
      y[0] = a0;
      y[1] = a1;
      break;
    }
    case EPI_RESID: {
      const float* rr = e.res + (size_t)r * e.ldres + c;
      float r0 = rr[0], r1 = rr[1];
      float* y = e.y + (size_t)r * e.ldy + c;
      y[0] = r0 + a0;
      y[1] = r1 + a1;
      break;
    }
    case EPI_RESID_SILU: {
      const float* rr = e.res + (size_t)r * e.ldres + c;
      float r0 = rr[0], r1 = rr[1];
      float* y = e.y + (size_t)r * e.ldy + c;
      y[0] = r0 + silu_f(a0);
      y[1] = r1 + silu_f(a1);
      break;
    }
    case EPI_SWIGLU: {
      e.y[(size_t)r * e.ldy + (c >> 1)] = silu_f(a0) * a1;
      break;
    }
    case EPI_QKV: {
      const int part = c / e.d;
      const int cc = c - part * e.d;
      const int h = cc / e.hd;
      const int dd = cc - h * e.hd;
      if (part < 2) {
        const int pos = e.rows.pos[r];
        const float2 cs = e.rope[(size_t)pos * (e.hd >> 1) + (dd >> 1)];
        const float r0 = a0 * cs.x - a1 * cs.y;
        const float r1 = a0 * cs.y + a1 * cs.x;
        a0 = r0;
        a1 = r1;
      }
      if (part == 0) {
        float* y = e.y + (size_t)r * e.ldy + cc;
        y[0] = a0;
        y[1] = a1;
      } else {
        const int b = e.rows.b[r];
        const int slot = e.rows.slot[r];
        const int pg = e.kv.pt ? e.rows.page[r] : 0;
        if (!kv_write_ok(e.kv, slot, pg)) {
          atomicOr(e.err, kErrIndex);
          return;
        }
        TC* base = reinterpret_cast<TC*>(part == 1 ? e.kv.k : e.kv.v);
        TC* p = base + kv_addr(e.kv, e.H, e.hd, b, h, slot, pg) + dd;
        store_cache(p, a0);
        store_cache(p + 1, a1);
      }
      break;
    }
  }
}

// Epilogue operands that do not depend on the dot products (residual values, RoPE angle,
// cache slot), loaded early so that their latency overlaps the main loop.
struct EpiPre {
  float r0, r1;  // residual pair
  float2 cs;     // RoPE cos/sin
  int b, slot, pg;  // cache sequence, slot and its page
  int pos;       // RoPE position (epi_load_early; the angle follows in epi_load_late)
};

static __device__ __forceinline__ EpiPre epi_load(const EpiArgs& e, int r, int c) {
  EpiPre p;
  p.r0 = p.r1 = 0.f;
  p.cs = make_float2(1.f, 0.f);
  p.b = p.slot = p.pg = 0;
  if (e.mode == EPI_RESID || e.mode == EPI_RESID_SILU) {
    const float2 q = *reinterpret_cast<const float2*>(e.res + (size_t)r * e.ldres + c);
    p.r0 = q.x;
    p.r1 = q.y;
  } else if (e.mode == EPI_QKV) {
    const int part = c / e.d;
    const int cc = c - part * e.d;
    const int dd = cc % e.hd;
    if (part < 2) {
      const int pos = e.rows.pos[r];
      p.cs = e.rope[(size_t)pos * (e.hd >> 1) + (dd >> 1)];
    }
    if (part > 0) {
      p.b = e.rows.b[r];
      p.slot = e.rows.slot[r];
      if (e.kv.pt) p.pg = e.rows.page[r];
    }
  }
  return p;
}

// epi_load in two halves, so that no load waits on another before the caller's own loads are
// issued: the first loads everything but the RoPE angle (the row's position instead), the second
// loads the angle at that position.
static __device__ __forceinline__ EpiPre epi_load_early(const EpiArgs& e, int r, int c) {
  EpiPre p;
  p.r0 = p.r1 = 0.f;
  p.cs = make_float2(1.f, 0.f);
  p.b = p.slot = p.pg = 0;
  p.pos = 0;
  if (e.mode == EPI_RESID || e.mode == EPI_RESID_SILU) {
    const float2 q = *reinterpret_cast<const float2*>(e.res + (size_t)r * e.ldres + c);
    p.r0 = q.x;
    p.r1 = q.y;
  } else if (e.mode == EPI_QKV) {
    const int part = c / e.d;
    if (part < 2) p.pos = e.rows.pos[r];
    if (part > 0) {
      p.b = e.rows.b[r];
      p.slot = e.rows.slot[r];
      if (e.kv.pt) p.pg = e.rows.page[r];
    }
  }
  return p;
}
static __device__ __forceinline__ void epi_load_late(const EpiArgs& e, EpiPre& p, int c) {
  if (e.mode == EPI_QKV) {
    const int part = c / e.d;
    if (part < 2) {
      const int dd = (c - part * e.d) % e.hd;
      p.cs = e.rope[(size_t)p.pos * (e.hd >> 1) + (dd >> 1)];
    }
  }
}

// The same epilogue split for row-wise batching (tensor-core tiles, where a thread owns a row and
// walks its columns): per-row metadata once, then per pair one float2 operand (the residual
// pair, or the RoPE cos/sin) that can be loaded a whole chunk of columns ahead of the stores.
struct EpiRow {
  int pos, b, slot, pg;
};
static __device__ __forceinline__ EpiRow epi_row(const EpiArgs& e, int r) {
  EpiRow q{0, 0, 0, 0};
  if (e.mode == EPI_QKV) {
    q.pos = e.rows.pos[r];
    q.b = e.rows.b[r];
    q.slot = e.rows.slot[r];
    if (e.kv.pt) q.pg = e.rows.page[r];
  }
  return q;
}
static __device__ __forceinline__ float2 epi_operand(const EpiArgs& e, const EpiRow& q, int r, int c) {
  if (e.mode == EPI_RESID || e.mode == EPI_RESID_SILU)
    return *reinterpret_cast<const float2*>(e.res + (size_t)r * e.ldres + c);
  if (e.mode == EPI_QKV) {
    const int part = c / e.d;
    if (part < 2) {
      const int dd = (c - part * e.d) % e.hd;
      return e.rope[(size_t)q.pos * (e.hd >> 1) + (dd >> 1)];
    }
  }
  return make_float2(0.f, 0.f);
}
template <typename TC>
static __device__ __forceinline__ void epi_store(const EpiArgs& e, const EpiPre& p, int r, int c, float a0, float a1) {
  switch (e.mode) {
    case EPI_STORE: {
      float* y = e.y + (size_t)r * e.ldy + c;
      *reinterpret_cast<float2*>(y) = make_float2(a0, a1);
      break;
    }
    case EPI_RESID: {
      float* y = e.y + (size_t)r * e.ldy + c;
      *reinterpret_cast<float2*>(y) = make_float2(p.r0 + a0, p.r1 + a1);
      break;
    }
    case EPI_RESID_SILU: {
      float* y = e.y + (size_t)r * e.ldy + c;
      *reinterpret_cast<float2*>(y) = make_float2(p.r0 + silu_f(a0), p.r1 + silu_f(a1));
      break;
    }
    case EPI_SWIGLU: {
      e.y[(size_t)r * e.ldy + (c >> 1)] = silu_f(a0) * a1;
      break;
    }
    case EPI_QKV: {
      const int part = c / e.d;
      const int cc = c - part * e.d;
      const int h = cc / e.hd;
      const int dd = cc - h * e.hd;
      if (part < 2) {
        const float x0 = a0 * p.cs.x - a1 * p.cs.y;
        const float x1 = a0 * p.cs.y + a1 * p.cs.x;
        a0 = x0;
        a1 = x1;
      }
      if (part == 0) {
        *reinterpret_cast<float2*>(e.y + (size_t)r * e.ldy + cc) = make_float2(a0, a1);
      } else {
        if (!kv_write_ok(e.kv, p.slot, p.pg)) {
          atomicOr(e.err, kErrIndex);
          return;
        }
        TC* base = reinterpret_cast<TC*>(part == 1 ? e.kv.k : e.kv.v);
        TC* q = base + kv_addr(e.kv, e.H, e.hd, p.b, h, p.slot, p.pg) + dd;
        store_cache(q, a0);
        store_cache(q + 1, a1);
      }
      break;
    }
  }
}


// Split on write by the weight-streaming GEMV: the final values of the column pair (c, c + 1) of row
// r (after the residual add, or the SwiGLU, which gives one value at column c / 2) as bf16 halves of
// v * g (g0, g1: the consumer's RMSNorm gain at those columns, or 1) at sp_hi / sp_lo[r * ldsp + c];
// returns the sum of the values' squares (before the gain).
static __device__ __forceinline__ float epi_split_pair(const EpiArgs& e, const EpiPre& p, int r, int c, float a0,
                                                       float a1, float g0, float g1) {
  float v0 = a0, v1 = a1;
  if (e.mode == EPI_RESID) {
    v0 = p.r0 + a0;
    v1 = p.r1 + a1;
  } else if (e.mode == EPI_RESID_SILU) {
    v0 = p.r0 + silu_f(a0);
    v1 = p.r1 + silu_f(a1);
  } else if (e.mode == EPI_SWIGLU) {
    const float m = silu_f(a0) * a1;
    const __nv_bfloat16 h = __float2bfloat16_rn(m * g0);
    const __nv_bfloat16 l = __float2bfloat16_rn(m * g0 - __bfloat162float(h));
    const size_t o = (size_t)r * e.ldsp + (c >> 1);
    e.sp_hi[o] = h;
    e.sp_lo[o] = l;
    return m * m;
  }
  const float x0 = v0 * g0, x1 = v1 * g1;
  const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
  const float2 hf = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
  const size_t o = (size_t)r * e.ldsp + c;
  *reinterpret_cast<__nv_bfloat162*>(e.sp_hi + o) = h;
  *reinterpret_cast<__nv_bfloat162*>(e.sp_lo + o) = l;
  return v0 * v0 + v1 * v1;
}

template <typename TC>
static __device__ __forceinline__ void epi_out(const EpiArgs& e, const EpiRow& q, float2 op, int r, int c,
                                               float a0, float a1) {
  EpiPre p;
  p.r0 = op.x;
  p.r1 = op.y;
  p.cs = op;
  p.b = q.b;
  p.slot = q.slot;
  p.pg = q.pg;
  p.pos = q.pos;
  epi_store<TC>(e, p, r, c, a0, a1);
}


}  // namespace lca
