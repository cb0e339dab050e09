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
#include "common.cuh"

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

__device__ __forceinline__ float silu_f(float x) { return x / (1.0f + expf(-x)); }

__device__ __forceinline__ void store_cache(float* p, float v) { *p = v; }
__device__ __forceinline__ void store_cache(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

// Epilogue of one pair of adjacent output columns (c even) of row r.
template <typename TC>
__device__ __forceinline__ void epi_pair(const EpiArgs& e, int r, int c, float a0, float a1) {
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
        if (slot < 0 || slot >= e.kv.S) {
          atomicOr(e.err, kErrIndex);
          return;
        }
        TC* base = reinterpret_cast<TC*>(part == 1 ? e.kv.k : e.kv.v);
        TC* p = base + (((size_t)b * e.H + h) * e.kv.S + slot) * e.hd + dd;
        store_cache(p, a0);
        store_cache(p + 1, a1);
      }
      break;
    }
  }
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

template <typename TW, bool NORM>
__global__ void __launch_bounds__(kWarps * 32)
k_gemv(LinearArgs a, int ksplit, float* __restrict__ part, int* __restrict__ cnt) {
  extern __shared__ float smem[];
  const int Kr = a.Kd / ksplit;
  float* xs = smem;                 // [kMC][Kr]
  float* inv = smem + kMC * Kr;     // [kMC]
  __shared__ int s_last;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tile = blockIdx.x;
  const int split = blockIdx.y;
  const int grp = blockIdx.z;
  const int k0 = split * Kr;
  const int col0 = tile * kColsPerCta + warp * kCPW;
  const TW* W = reinterpret_cast<const TW*>(a.W) + (size_t)grp * a.N * a.Kd;
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
        for (int k = lane; k < a.Kd; k += 32) ss += xr[k] * xr[k];
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
          const float s = inv[i];
          const float4 g = *reinterpret_cast<const float4*>(a.norm + k0 + kk);
          v.x *= s * g.x; v.y *= s * g.y; v.z *= s * g.z; v.w *= s * g.w;
        }
      }
      *reinterpret_cast<float4*>(xs + i * Kr + kk) = v;
    }
    __syncthreads();

    if (col0 < a.N) {
      float acc[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[j] = 0.f;
#pragma unroll 2
      for (int kk = lane * 8; kk < Kr; kk += 256) {
        float w[kCPW][8];
#pragma unroll
        for (int c = 0; c < kCPW; ++c) load_w8(W + (size_t)(col0 + c) * a.Kd + k0 + kk, w[c]);
#pragma unroll
        for (int i = 0; i < kMC; ++i) {
          const float4 xa = *reinterpret_cast<const float4*>(xs + i * Kr + kk);
          const float4 xb = *reinterpret_cast<const float4*>(xs + i * Kr + kk + 4);
#pragma unroll
          for (int c = 0; c < kCPW; ++c) {
            float s = acc[i * kCPW + c];
            s = fmaf(w[c][0], xa.x, s); s = fmaf(w[c][1], xa.y, s);
            s = fmaf(w[c][2], xa.z, s); s = fmaf(w[c][3], xa.w, s);
            s = fmaf(w[c][4], xb.x, s); s = fmaf(w[c][5], xb.y, s);
            s = fmaf(w[c][6], xb.z, s); s = fmaf(w[c][7], xb.w, s);
            acc[i * kCPW + c] = s;
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

// ---------------------------------------------------------------- tiled GEMM (many rows)
constexpr int kBM = 64, kBN = 64, kBK = 32;

__global__ void k_rowstats(const float* __restrict__ x, int ldx, int Kd, const int* Mp, int M_cap,
                           int groups, int Mg_stride, float eps, float* __restrict__ inv) {
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
  __shared__ float As[kBK][kBM + 4];
  __shared__ float Bs[kBK][kBN + 4];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int grp = blockIdx.z;
  const TW* W = reinterpret_cast<const TW*>(a.W) + (size_t)grp * a.N * a.Kd;
  const int rbase = grp * a.Mg_stride;
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

template <typename TW, bool NORM>
void launch_gemv(const Dev& D, const LinearArgs& a, cudaStream_t s) {
  int ksplit = 1;
  if (a.groups == 1 && a.N <= 2048 && D.lin_part) {
    ksplit = a.Kd >= 2048 ? 8 : 4;
    while (ksplit > 1 && ((a.Kd % ksplit) || ((a.Kd / ksplit) % 8) ||
                          (size_t)ksplit * a.M_cap * a.N > D.lin_part_floats))
      ksplit >>= 1;
  }
  const int Kr = a.Kd / ksplit;
  const size_t smem = (size_t)kMC * Kr * sizeof(float) + kMC * sizeof(float);
  dim3 grid((a.N + kColsPerCta - 1) / kColsPerCta, ksplit, a.groups);
  ++g_launches;
  k_gemv<TW, NORM><<<grid, kWarps * 32, smem, s>>>(a, ksplit, D.lin_part, D.lin_cnt);
}

template <typename TW, bool NORM>
void launch_gemm(const Dev& D, const LinearArgs& a, cudaStream_t s) {
  if (NORM) {
    ++g_launches;
    k_rowstats<<<256, 256, 0, s>>>(a.x, a.ldx, a.Kd, a.M, a.M_cap, a.groups, a.Mg_stride, a.eps,
                                   D.inv_rms);
  }
  const int ntm = (a.M_cap + kBM - 1) / kBM, ntn = (a.N + kBN - 1) / kBN;
  int tiles = ntm * ntn;
  int grid = tiles < 152 * 4 ? tiles : 152 * 4;
  ++g_launches;
  k_gemm<TW, NORM><<<dim3(grid, 1, a.groups), 256, 0, s>>>(a, D.inv_rms);
}

} // namespace

void kernel_attrs_linear() {
  const int mx = 200 * 1024;
  cudaFuncSetAttribute(k_gemv<__nv_bfloat16, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  cudaFuncSetAttribute(k_gemv<__nv_bfloat16, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  cudaFuncSetAttribute(k_gemv<float, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  cudaFuncSetAttribute(k_gemv<float, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
}

void linear(const Dev& D, const LinearArgs& a, bool tiled, cudaStream_t s) {
  const bool norm = a.norm != nullptr;
  ProfScope ps(PK_LINEAR, (double)a.N * a.Kd * a.groups * (D.dtype == LCA_BF16 ? 2 : 4), s);
  if (D.dtype == LCA_BF16) {
    if (tiled) norm ? launch_gemm<__nv_bfloat16, true>(D, a, s) : launch_gemm<__nv_bfloat16, false>(D, a, s);
    else norm ? launch_gemv<__nv_bfloat16, true>(D, a, s) : launch_gemv<__nv_bfloat16, false>(D, a, s);
  } else {
    if (tiled) norm ? launch_gemm<float, true>(D, a, s) : launch_gemm<float, false>(D, a, s);
    else norm ? launch_gemv<float, true>(D, a, s) : launch_gemv<float, false>(D, a, s);
  }
}

} // namespace lca
