// Causal softmax attention of query rows over a KV-cache layer (Section 2.2 causal masks;
// inside the multi-byte window of Algorithm 1 (its drafting window) the LCA mask is causal as well, so
// every attention of the decode step is "query row r sees cache slots [0, kvlen[r])").
//
// One CTA serves one (sequence, query tile of up to 8 rows, head, key split). Keys and
// values stream through shared memory in tiles of 32; softmax is computed online in fp32.
// With several key splits each CTA writes (max, sum, acc) partials and the last CTA of the
// (sequence, head) combines them in split order (deterministic).
#include <cooperative_groups.h>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cstring>
#include <algorithm>
#include <mutex>

#include "common.cuh"

namespace lca {

namespace {

constexpr int kKT = 64;     // keys per tile
constexpr int kThreads = 128;
constexpr int kQTMax = 4;   // query tiles per sequence that may split their key range
constexpr int kMaxClusterSplit = 8;  // portable thread-block cluster size

__device__ __forceinline__ void unpack16(const uint4& u, float* f, const float*) {
  f[0] = __uint_as_float(u.x); f[1] = __uint_as_float(u.y);
  f[2] = __uint_as_float(u.z); f[3] = __uint_as_float(u.w);
}
__device__ __forceinline__ void unpack16(const uint4& u, float* f, const __nv_bfloat16*) {
  f[0] = __uint_as_float(u.x << 16); f[1] = __uint_as_float(u.x & 0xFFFF0000u);
  f[2] = __uint_as_float(u.y << 16); f[3] = __uint_as_float(u.y & 0xFFFF0000u);
  f[4] = __uint_as_float(u.z << 16); f[5] = __uint_as_float(u.z & 0xFFFF0000u);
  f[6] = __uint_as_float(u.w << 16); f[7] = __uint_as_float(u.w & 0xFFFF0000u);
}

// An attention output value v at element o of [rows][H * HD]; with osh set, also as bf16 halves
// (v = hi + lo) at the same place of osh / osl, the staged input of a weight-streaming GEMV.
__device__ __forceinline__ void out_store(float* out, __nv_bfloat16* osh, __nv_bfloat16* osl, size_t o, float v) {
  out[o] = v;
  if (osh) {
    const __nv_bfloat16 hv = __float2bfloat16_rn(v);
    osh[o] = hv;
    osl[o] = __float2bfloat16_rn(v - __bfloat162float(hv));
  }
}

template <typename TC, int HD>
__global__ void __launch_bounds__(kThreads)
k_attn(const float* __restrict__ q, float* __restrict__ out, KV kv, Rows rows, int H, float scale,
       int splits, float* __restrict__ part, int* __restrict__ cnt, int* err) {
  TraceScope _trace(TT_ATTN);
  constexpr int QT = kAttnQT;
  constexpr int EV = 16 / (int)sizeof(TC);  // cache elements per 16-byte vector
  __shared__ float qs[QT][HD];
  __shared__ float ks[kKT][HD + 1];
  __shared__ float vs[kKT][HD];
  __shared__ float ps[QT][kKT];
  __shared__ float s_m[QT], s_l[QT], s_corr[QT];
  __shared__ int s_kv[QT];
  __shared__ int s_last;

  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const int b = blockIdx.x;
  const int h = blockIdx.z / splits;
  const int sp = blockIdx.z - h * splits;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nrows = rows.seq_count[b];
  const int rbeg = rows.seq_start[b];
  const int ntiles = (nrows + QT - 1) / QT;
  const TC* Kc = reinterpret_cast<const TC*>(kv.k);
  const TC* Vc = reinterpret_cast<const TC*>(kv.v);
  const int ld = H * HD;

  // accumulator ownership: row ai, dims ad..ad+DPT-1
  constexpr int DPT = QT * HD / kThreads;
  const int ai = tid / (HD / DPT);
  const int ad = (tid % (HD / DPT)) * DPT;
  // score ownership: key sk, rows sr..sr+3
  const int sk = tid & (kKT - 1);
  const int sr = (tid / kKT) * (QT * kKT / kThreads);

  for (int qt = blockIdx.y; qt < ntiles; qt += gridDim.y) {
    const int r0 = rbeg + qt * QT;
    const int nq = min(QT, nrows - qt * QT);
    __syncthreads();
    for (int idx = tid; idx < QT * HD; idx += kThreads) {
      const int i = idx / HD, dd = idx - i * HD;
      qs[i][dd] = i < nq ? q[(size_t)(r0 + i) * ld + h * HD + dd] * scale : 0.f;
    }
    if (tid < QT) {
      int kl = tid < nq ? rows.kvlen[r0 + tid] : 0;
      if (kl > kv.S) {
        atomicOr(err, kErrIndex);
        kl = kv.S;
      }
      s_kv[tid] = kl;
      s_m[tid] = -INFINITY;
      s_l[tid] = 0.f;
    }
    __syncthreads();
    int kv_hi = 0;
#pragma unroll
    for (int i = 0; i < QT; ++i) kv_hi = max(kv_hi, s_kv[i]);
    // tiles beyond kQTMax (long multi-byte windows) are done whole by split 0
    const bool split_mode = splits > 1 && qt < kQTMax;
    if (!split_mode && sp != 0) continue;
    const int nsp = split_mode ? splits : 1;
    const int chunk = ((kv_hi + nsp - 1) / nsp + 15) / 16 * 16;
    const int lo = split_mode ? sp * chunk : 0;
    const int hi = min(kv_hi, lo + chunk);

    float acc[DPT];
#pragma unroll
    for (int j = 0; j < DPT; ++j) acc[j] = 0.f;

    for (int j0 = lo; j0 < hi; j0 += kKT) {
      const int nk = min(kKT, hi - j0);
      {
        // the whole K/V tile: every thread issues all its 16-byte loads before any store
        constexpr int NL = kKT * HD / EV / kThreads;
        uint4 uk[NL], uv[NL];
#pragma unroll
        for (int u = 0; u < NL; ++u) {
          const int e = (tid + u * kThreads) * EV;
          const int kk = e / HD, dd = e - kk * HD;
          if (kk < nk) {
            const size_t o = kv_off(kv, H, HD, b, h, j0 + kk) + dd;
            uk[u] = *reinterpret_cast<const uint4*>(Kc + o);
            uv[u] = *reinterpret_cast<const uint4*>(Vc + o);
          } else {
            uk[u] = make_uint4(0, 0, 0, 0);
            uv[u] = make_uint4(0, 0, 0, 0);
          }
        }
#pragma unroll
        for (int u = 0; u < NL; ++u) {
          const int e = (tid + u * kThreads) * EV;
          const int kk = e / HD, dd = e - kk * HD;
          float fk[8], fv[8];
          unpack16(uk[u], fk, (const TC*)nullptr);
          unpack16(uv[u], fv, (const TC*)nullptr);
#pragma unroll
          for (int j = 0; j < EV; ++j) {
            ks[kk][dd + j] = fk[j];
            vs[kk][dd + j] = fv[j];
          }
        }
      }
      __syncthreads();
      // scores of 4 rows for one key per thread
      {
        float sc[QT * kKT / kThreads];
#pragma unroll
        for (int r = 0; r < QT * kKT / kThreads; ++r) sc[r] = 0.f;
#pragma unroll 16
        for (int dd = 0; dd < HD; ++dd) {
          const float kd = ks[sk][dd];
#pragma unroll
          for (int r = 0; r < QT * kKT / kThreads; ++r) sc[r] = fmaf(qs[sr + r][dd], kd, sc[r]);
        }
#pragma unroll
        for (int r = 0; r < QT * kKT / kThreads; ++r)
          ps[sr + r][sk] = (sk < nk && j0 + sk < s_kv[sr + r]) ? sc[r] : -INFINITY;
      }
      __syncthreads();
      // online softmax: warp w updates rows 2w, 2w+1
      for (int i = warp * (QT / 4); i < (warp + 1) * (QT / 4); ++i) {
        const float v0 = ps[i][lane], v1 = ps[i][lane + 32];
        float mx = fmaxf(v0, v1);
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_old = s_m[i];
        const float m_new = fmaxf(m_old, mx);
        const float p0 = v0 == -INFINITY ? 0.f : expf(v0 - m_new);
        const float p1 = v1 == -INFINITY ? 0.f : expf(v1 - m_new);
        float ssum = p0 + p1;
#pragma unroll
        for (int o = 16; o; o >>= 1) ssum += __shfl_xor_sync(0xffffffffu, ssum, o);
        ps[i][lane] = p0;
        ps[i][lane + 32] = p1;
        __syncwarp();
        if (lane == 0) {
          const float corr = (m_old == -INFINITY) ? 0.f : expf(m_old - m_new);
          s_corr[i] = corr;
          s_l[i] = s_l[i] * corr + ssum;
          s_m[i] = m_new;
        }
      }
      __syncthreads();
      {
        const float corr = s_corr[ai];
#pragma unroll
        for (int j = 0; j < DPT; ++j) acc[j] *= corr;
        for (int kk = 0; kk < nk; ++kk) {
          const float p = ps[ai][kk];
#pragma unroll
          for (int j = 0; j < DPT; ++j) acc[j] = fmaf(p, vs[kk][ad + j], acc[j]);
        }
      }
      __syncthreads();
    }

    if (!split_mode) {
      if (ai < nq) {
        const float l = s_l[ai];
        const float il = l > 0.f ? 1.f / l : 0.f;
        float* o = out + (size_t)(r0 + ai) * ld + h * HD + ad;
#pragma unroll
        for (int j = 0; j < DPT; ++j) o[j] = acc[j] * il;
      }
      continue;
    }
    // split partials: tile (b, qt, h), split sp -> acc[QT][HD], m[QT], l[QT]
    const size_t tile_id = ((size_t)b * kQTMax + qt) * H + h;
    float* pp = part + (tile_id * splits + sp) * (QT * (HD + 2));
#pragma unroll
    for (int j = 0; j < DPT; ++j) pp[ai * HD + ad + j] = acc[j];
    if (tid < QT) {
      pp[QT * HD + tid] = s_m[tid];
      pp[QT * HD + QT + tid] = s_l[tid];
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = (atomicAdd(cnt + tile_id, 1) == splits - 1);
    __syncthreads();
    if (!s_last) continue;
    __threadfence();
    {
      // stage every split's (max, sum) in shared memory with parallel loads, then combine
      const float* base = part + tile_id * splits * (QT * (HD + 2));
      float* sm = &ps[0][0];                // splits * QT maxima   (<= 128 floats)
      float* sl = &ks[0][0];                // splits * QT sums
      for (int idx = tid; idx < splits * QT; idx += kThreads) {
        const int k = idx / QT, i = idx - k * QT;
        sm[idx] = __ldcg(base + k * (QT * (HD + 2)) + QT * HD + i);
        sl[idx] = __ldcg(base + k * (QT * (HD + 2)) + QT * HD + QT + i);
      }
      __syncthreads();
      if (ai < nq) {
        float M = -INFINITY;
        for (int k = 0; k < splits; ++k) M = fmaxf(M, sm[k * QT + ai]);
        float L = 0.f, o[DPT];
#pragma unroll
        for (int j = 0; j < DPT; ++j) o[j] = 0.f;
#pragma unroll 4
        for (int k = 0; k < splits; ++k) {
          const float mk = sm[k * QT + ai];
          const float w = mk == -INFINITY ? 0.f : expf(mk - M);
          L += w * sl[k * QT + ai];
          const float* pk = base + k * (QT * (HD + 2)) + ai * HD + ad;
#pragma unroll
          for (int j = 0; j < DPT; ++j) o[j] += w * __ldcg(pk + j);
        }
        const float il = L > 0.f ? 1.f / L : 0.f;
        float* dst = out + (size_t)(r0 + ai) * ld + h * HD + ad;
#pragma unroll
        for (int j = 0; j < DPT; ++j) dst[j] = o[j] * il;
      }
    }
    if (tid == 0) cnt[tile_id] = 0;
  }
}

// Decode attention, second form: 256 threads; scores with one key per thread (its K row held in
// registers, loaded straight from global memory), online softmax with one warp per query row,
// and P.V with each thread owning 4 dims of every row over a group of keys. The key range of a
// (sequence, query tile, head) is split over the CTAs of a cluster and combined through
// distributed shared memory by rank 0, in rank order.
constexpr int kA2Threads = 256;
constexpr int kA2Keys = 256;  // keys per pass

__device__ __forceinline__ void unpack_vec(const uint4& u, float* f, const __nv_bfloat16*) {
  f[0] = __uint_as_float(u.x << 16); f[1] = __uint_as_float(u.x & 0xFFFF0000u);
  f[2] = __uint_as_float(u.y << 16); f[3] = __uint_as_float(u.y & 0xFFFF0000u);
  f[4] = __uint_as_float(u.z << 16); f[5] = __uint_as_float(u.z & 0xFFFF0000u);
  f[6] = __uint_as_float(u.w << 16); f[7] = __uint_as_float(u.w & 0xFFFF0000u);
}
__device__ __forceinline__ void unpack_vec(const uint4& u, float* f, const float*) {
  f[0] = __uint_as_float(u.x); f[1] = __uint_as_float(u.y);
  f[2] = __uint_as_float(u.z); f[3] = __uint_as_float(u.w);
}
__device__ __forceinline__ void load4(const __nv_bfloat16* p, float (&v)[4]) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  v[0] = __uint_as_float(u.x << 16); v[1] = __uint_as_float(u.x & 0xFFFF0000u);
  v[2] = __uint_as_float(u.y << 16); v[3] = __uint_as_float(u.y & 0xFFFF0000u);
}
__device__ __forceinline__ void load4(const float* p, float (&v)[4]) {
  const float4 u = *reinterpret_cast<const float4*>(p);
  v[0] = u.x; v[1] = u.y; v[2] = u.z; v[3] = u.w;
}

template <typename TC, int HD>
__global__ void __launch_bounds__(kA2Threads)
k_attn2(const float* __restrict__ q, float* __restrict__ out, KV kv, Rows rows, int H, float scale,
        int* err) {
  namespace cgr = cooperative_groups;
  constexpr int QT = kAttnQT;
  constexpr int EV = 16 / (int)sizeof(TC);
  constexpr int NV = HD / EV;              // 16-byte vectors per key row
  constexpr int DG = HD / 4;               // dim groups of 4
  constexpr int KG = kA2Threads / DG;      // key groups in P.V
  constexpr int KPG = kA2Keys / KG;        // keys per key group
  __shared__ __align__(16) float qs[QT][HD];
  __shared__ float ps[QT][kA2Keys];
  __shared__ __align__(16) float red[KG][QT][HD];
  __shared__ __align__(16) float pacc[QT][HD];
  __shared__ float s_m[QT], s_l[QT], s_corr[QT];
  __shared__ int s_kv[QT];

  TraceScope _trace(TT_ATTN);
  cgr::cluster_group cl = cgr::this_cluster();
  const int splits = (int)cl.dim_blocks().z;
  const int sp = (int)cl.block_rank();
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const int b = blockIdx.x;
  const int h = blockIdx.z / splits;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int dg = tid % DG, kg = tid / DG;
  const int nrows = rows.seq_count[b];
  const int rbeg = rows.seq_start[b];
  const int ntiles = (nrows + QT - 1) / QT;
  const TC* Kc = reinterpret_cast<const TC*>(kv.k);
  const TC* Vc = reinterpret_cast<const TC*>(kv.v);
  const int ld = H * HD;

  for (int qt = blockIdx.y; qt < ntiles; qt += gridDim.y) {
    const int r0 = rbeg + qt * QT;
    const int nq = min(QT, nrows - qt * QT);
    __syncthreads();
    for (int idx = tid; idx < QT * HD; idx += kA2Threads) {
      const int i = idx / HD, dd = idx - i * HD;
      qs[i][dd] = i < nq ? q[(size_t)(r0 + i) * ld + h * HD + dd] * scale : 0.f;
    }
    if (tid < QT) {
      int kl = tid < nq ? rows.kvlen[r0 + tid] : 0;
      if (kl > kv.S) {
        atomicOr(err, kErrIndex);
        kl = kv.S;
      }
      s_kv[tid] = kl;
      s_m[tid] = -INFINITY;
      s_l[tid] = 0.f;
    }
    __syncthreads();
    int kv_hi = 0;
#pragma unroll
    for (int i = 0; i < QT; ++i) kv_hi = max(kv_hi, s_kv[i]);
    const int chunk = ((kv_hi + splits - 1) / splits + 15) / 16 * 16;
    const int lo = sp * chunk;
    const int hi = min(kv_hi, lo + chunk);
    float acc[QT][4];
#pragma unroll
    for (int r = 0; r < QT; ++r)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[r][e] = 0.f;

    for (int j0 = lo; j0 < hi; j0 += kA2Keys) {
      const int nk = min(kA2Keys, hi - j0);
      // scores: thread tid owns key j0 + tid
      {
        const int j = j0 + tid;
        float sc[QT];
#pragma unroll
        for (int r = 0; r < QT; ++r) sc[r] = 0.f;
        if (tid < nk) {
          uint4 kr[NV];
          const TC* kp = Kc + kv_off(kv, H, HD, b, h, j);
#pragma unroll
          for (int v = 0; v < NV; ++v) kr[v] = *reinterpret_cast<const uint4*>(kp + v * EV);
#pragma unroll
          for (int v = 0; v < NV; ++v) {
            float kf[8];
            unpack_vec(kr[v], kf, (const TC*)nullptr);
#pragma unroll
            for (int r = 0; r < QT; ++r) {
              if (r < nq) {
#pragma unroll
                for (int e4 = 0; e4 < EV; e4 += 4) {
                  const float4 qv = *reinterpret_cast<const float4*>(&qs[r][v * EV + e4]);
                  sc[r] = fmaf(qv.x, kf[e4 + 0], sc[r]);
                  sc[r] = fmaf(qv.y, kf[e4 + 1], sc[r]);
                  sc[r] = fmaf(qv.z, kf[e4 + 2], sc[r]);
                  sc[r] = fmaf(qv.w, kf[e4 + 3], sc[r]);
                }
              }
            }
          }
        }
#pragma unroll
        for (int r = 0; r < QT; ++r) ps[r][tid] = (tid < nk && r < nq && j < s_kv[r]) ? sc[r] : -INFINITY;
      }
      __syncthreads();
      // online softmax: warp w owns row w
      if (warp < QT) {
        const int i = warp;
        float v[kA2Keys / 32];
        float mx = -INFINITY;
#pragma unroll
        for (int u = 0; u < kA2Keys / 32; ++u) {
          v[u] = ps[i][lane + 32 * u];
          mx = fmaxf(mx, v[u]);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_old = s_m[i];
        const float m_new = fmaxf(m_old, mx);
        float ssum = 0.f;
#pragma unroll
        for (int u = 0; u < kA2Keys / 32; ++u) {
          const float p = v[u] == -INFINITY ? 0.f : expf(v[u] - m_new);
          ps[i][lane + 32 * u] = p;
          ssum += p;
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) ssum += __shfl_xor_sync(0xffffffffu, ssum, o);
        if (lane == 0) {
          const float corr = (m_old == -INFINITY) ? 0.f : expf(m_old - m_new);
          s_corr[i] = corr;
          s_l[i] = s_l[i] * corr + ssum;
          s_m[i] = m_new;
        }
      }
      __syncthreads();
      // P.V: thread (dg, kg) accumulates dims 4dg..4dg+3 of every row over its keys
      {
#pragma unroll
        for (int r = 0; r < QT; ++r) {
          const float corr = s_corr[r];
#pragma unroll
          for (int e = 0; e < 4; ++e) acc[r][e] *= corr;
        }
        float vv[KPG][4];
#pragma unroll
        for (int u = 0; u < KPG; ++u) {
          const int key = kg * KPG + u;
          if (key < nk) load4(Vc + kv_off(kv, H, HD, b, h, j0 + key) + dg * 4, vv[u]);
          else vv[u][0] = vv[u][1] = vv[u][2] = vv[u][3] = 0.f;
        }
#pragma unroll
        for (int u = 0; u < KPG; ++u) {
          const int key = kg * KPG + u;
#pragma unroll
          for (int r = 0; r < QT; ++r) {
            if (r < nq) {
              const float p = ps[r][key];
#pragma unroll
              for (int e = 0; e < 4; ++e) acc[r][e] = fmaf(p, vv[u][e], acc[r][e]);
            }
          }
        }
      }
      __syncthreads();
    }
    // reduce the key groups: pacc[r][d] = sum over kg
#pragma unroll
    for (int r = 0; r < QT; ++r)
      *reinterpret_cast<float4*>(&red[kg][r][dg * 4]) = make_float4(acc[r][0], acc[r][1], acc[r][2], acc[r][3]);
    __syncthreads();
    for (int idx = tid; idx < QT * HD; idx += kA2Threads) {
      const int r = idx / HD, dd = idx - r * HD;
      float t = 0.f;
#pragma unroll 8
      for (int g2 = 0; g2 < KG; ++g2) t += red[g2][r][dd];
      pacc[r][dd] = t;
    }
    cl.sync();
    // every rank combines its slice of the head dims over all ranks, in rank order; the
    // remote (max, sum, acc) values are requested before any is used
    {
      const int dpr = (HD + splits - 1) / splits;  // dims per rank
      const int d0 = sp * dpr;
      const int nd = min(dpr, HD - d0);
      for (int idx = tid; idx < nq * nd; idx += kA2Threads) {
        const int r = idx / nd, dd = d0 + (idx - r * nd);
        float mr[kMaxClusterSplit], lr[kMaxClusterSplit], ar[kMaxClusterSplit];
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k) {
          if (k < splits) {
            mr[k] = *cl.map_shared_rank(&s_m[r], k);
            lr[k] = *cl.map_shared_rank(&s_l[r], k);
            ar[k] = *cl.map_shared_rank(&pacc[r][dd], k);
          }
        }
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k)
          if (k < splits) M = fmaxf(M, mr[k]);
        float L = 0.f, o = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k) {
          if (k < splits && mr[k] != -INFINITY) {
            const float w = expf(mr[k] - M);
            L += w * lr[k];
            o += w * ar[k];
          }
        }
        out[(size_t)(r0 + r) * ld + h * HD + dd] = L > 0.f ? o / L : 0.f;
      }
    }
    cl.sync();
  }
}

// ---------------------------------------------------------------- pipelined decode attention
// One CTA of 128 threads serves (sequence, query tile of up to 8 rows, head, key split). Its key
// range streams in chunks of 64 keys through a ring of shared-memory stages filled by bulk
// asynchronous copies (the cache of one (sequence, head) is contiguous, so a chunk of K or V is
// one copy), several chunks ahead of the arithmetic. Per chunk: one key per thread for the
// scores (16-byte reads rotated per key, so a warp's reads spread over all banks), one warp per
// query row for the online softmax (fp32), a pair of head dims per thread for P.V with the
// probabilities broadcast from shared memory. Key splits of one (sequence, head) form a
// thread-block cluster and combine (max, sum, accumulator) through distributed shared memory.
constexpr int kA4MaxSplit = 16;  // largest key split (non-portable cluster size)
constexpr int kA3Threads = 128;
constexpr int kA3Keys = 64;     // keys per chunk
constexpr int kA3Stages = 4;
constexpr int kA3Spins = 1 << 22;

__device__ __forceinline__ uint32_t a3_su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void a3_expect(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a3_su32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void a3_copy(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          a3_su32(dst)),
      "l"(src), "r"(bytes), "r"(a3_su32(bar))
      : "memory");
}
__device__ __forceinline__ bool a3_wait(uint64_t* bar, uint32_t parity) {
  for (int i = 0; i < kA3Spins; ++i) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(a3_su32(bar)), "r"(parity)
        : "memory");
    if (ok) return true;
  }
  return false;
}
__device__ __forceinline__ void a3_v2(const float* p, float& a, float& b) {
  const float2 v = *reinterpret_cast<const float2*>(p);
  a = v.x;
  b = v.y;
}
__device__ __forceinline__ void a3_v2(const __nv_bfloat16* p, float& a, float& b) {
  const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
  a = __uint_as_float(u << 16);
  b = __uint_as_float(u & 0xFFFF0000u);
}

template <typename TC, int HD>
__global__ void __launch_bounds__(kA3Threads, 3)
k_attn3(const float* __restrict__ q, float* __restrict__ out, KV kv, Rows rows, int H, float scale,
        int* err, __nv_bfloat16* osh, __nv_bfloat16* osl) {
  namespace cgr = cooperative_groups;
  constexpr int QT = kAttnQT;                     // query rows per tile (8)
  constexpr int KC = kA3Keys;
  constexpr int EV = 16 / (int)sizeof(TC);        // elements per 16-byte vector
  constexpr int NV = HD / EV;                     // 16-byte vectors per key row
  constexpr uint32_t CB = KC * HD * sizeof(TC);   // bytes of one K (or V) chunk
  constexpr int RH = kA3Threads / KC;             // row groups in the score phase (2)
  constexpr int DP = HD / 2;                      // dim pairs
  constexpr int RG = kA3Threads / DP;             // row groups in P.V (4 for HD 64)
  constexpr int RPT = QT / RG;                    // rows per thread in P.V
  static_assert(QT % RH == 0 && QT % RG == 0 && RPT >= 1, "tile shape");
  extern __shared__ __align__(128) unsigned char a3sm[];
  unsigned char* ring = a3sm;                                        // [stages][K | V]
  float* qs = reinterpret_cast<float*>(a3sm + kA3Stages * 2 * CB);   // [QT][HD], pre-scaled
  float* sc = qs + QT * HD;                                          // [QT][KC] scores -> probs
  float* pacc = sc + QT * KC;                                        // [QT][HD] this split's acc
  float* s_m = pacc + QT * HD;                                       // [QT]
  float* s_l = s_m + QT;                                             // [QT]
  float* s_corr = s_l + QT;                                          // [QT]
  int* s_kv = reinterpret_cast<int*>(s_corr + QT);                   // [QT]
  uint64_t* full = reinterpret_cast<uint64_t*>(s_kv + QT);           // [stages]
  int* s_pt = reinterpret_cast<int*>(full + kA3Stages);              // [pt_ld] page table row (paged)

  TraceScope _trace(TT_ATTN);
  cgr::cluster_group cl = cgr::this_cluster();
  const int splits = (int)cl.dim_blocks().z;
  const int sp = (int)cl.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < kA3Stages; ++i)
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(a3_su32(&full[i])) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  pdl_wait();
  _trace.waited();
  __syncthreads();
  const int b = blockIdx.x;
  const int h = blockIdx.z / splits;
  const int pt0 = kv_pages_load(kv, b, tid);  // stored with the first tile's loads
  const int nrows = rows.seq_count[b];
  const int rbeg = rows.seq_start[b];
  const int ntiles = (nrows + QT - 1) / QT;
  const TC* Kc = reinterpret_cast<const TC*>(kv.k);
  const TC* Vc = reinterpret_cast<const TC*>(kv.v);
  const int ld = H * HD;
  bool failed = false;
  uint32_t cc = 0;      // chunks consumed by this CTA so far (ring phase)
  uint32_t issued = 0;  // chunks whose copies were issued (thread 0)

  for (int qt = blockIdx.y; qt < ntiles; qt += gridDim.y) {
    const int r0 = rbeg + qt * QT;
    const int nq = min(QT, nrows - qt * QT);
    for (int idx = tid; idx < QT * HD; idx += kA3Threads) {
      const int i = idx / HD, dd = idx - i * HD;
      qs[idx] = i < nq ? q[(size_t)(r0 + i) * ld + h * HD + dd] * scale : 0.f;
    }
    if (tid < QT) {
      int kl = tid < nq ? rows.kvlen[r0 + tid] : 0;
      if (kl > kv.S || kl < 0) {
        atomicOr(err, kErrIndex);
        kl = kl < 0 ? 0 : kv.S;
      }
      s_kv[tid] = kl;
      s_m[tid] = -INFINITY;
      s_l[tid] = 0.f;
    }
    if (qt == (int)blockIdx.y) kv_pages_store(kv, b, s_pt, tid, kA3Threads, pt0);
    __syncthreads();
    int kv_hi = 0;
#pragma unroll
    for (int i = 0; i < QT; ++i) kv_hi = max(kv_hi, s_kv[i]);
    const int per = ((kv_hi + splits - 1) / splits + KC - 1) / KC * KC;
    const int lo = sp * per;
    const int hi = min(kv_hi, lo + per);
    const int nch = hi > lo ? (hi - lo + KC - 1) / KC : 0;
    auto issue = [&](int c) {
      const uint32_t g = cc + c;
      const int st = g % kA3Stages;
      const int j0 = lo + c * KC;
      const int nk = min(KC, hi - j0);
      const uint32_t bytes = (uint32_t)(nk * HD * sizeof(TC));
      unsigned char* dst = ring + (size_t)st * 2 * CB;
      ++issued;
      // a chunk starts on a page (KC == kPage, lo a multiple of KC) and stays inside it
      const size_t o = kv_addr(kv, H, HD, b, h, j0, kv.pt ? s_pt[j0 / kPage] : 0);
      a3_expect(&full[st], 2 * bytes);
      a3_copy(dst, Kc + o, bytes, &full[st]);
      a3_copy(dst + CB, Vc + o, bytes, &full[st]);
    };
    if (tid == 0)
      for (int c = 0; c < nch && c < kA3Stages - 1; ++c) issue(c);
    float acc[RPT][2];
#pragma unroll
    for (int m = 0; m < RPT; ++m) acc[m][0] = acc[m][1] = 0.f;
    const int dp = tid % DP, rg = tid / DP;

    for (int c = 0; c < nch; ++c) {
      __syncthreads();  // chunk c-1 fully read: its stage may be refilled
      if (tid == 0 && c + kA3Stages - 1 < nch) issue(c + kA3Stages - 1);
      const uint32_t g = cc + c;
      const int st = g % kA3Stages;
      if (!failed && !a3_wait(&full[st], (g / kA3Stages) & 1)) failed = true;
      const TC* Ks = reinterpret_cast<const TC*>(ring + (size_t)st * 2 * CB);
      const TC* Vs = reinterpret_cast<const TC*>(ring + (size_t)st * 2 * CB + CB);
      const int j0 = lo + c * KC;
      const int nk = min(KC, hi - j0);
      // scores: key j of this chunk, rows rh, rh + RH, ...
      {
        const int j = tid % KC, rh = tid / KC;
        float s[QT / RH];
#pragma unroll
        for (int m = 0; m < QT / RH; ++m) s[m] = 0.f;
        if (j < nk) {
          const uint4* kr = reinterpret_cast<const uint4*>(Ks + (size_t)j * HD);
#pragma unroll
          for (int v = 0; v < NV; ++v) {
            const int vv = (v + j) % NV;
            float kf[EV];
            unpack16(kr[vv], kf, (const TC*)nullptr);
#pragma unroll
            for (int m = 0; m < QT / RH; ++m) {
              if (rh + m * RH < nq) {  // warp-uniform
                const float* qr = qs + (rh + m * RH) * HD + vv * EV;
#pragma unroll
                for (int e = 0; e < EV; ++e) s[m] = fmaf(qr[e], kf[e], s[m]);
              }
            }
          }
        }
#pragma unroll
        for (int m = 0; m < QT / RH; ++m) {
          const int i = rh + m * RH;
          const bool ok = j < nk && (j0 + j) < s_kv[i] && i < nq;
          sc[i * KC + j] = ok ? s[m] : -INFINITY;
        }
      }
      __syncthreads();
      // online softmax: warp w owns rows w, w + 4
      for (int i = warp; i < QT; i += kA3Threads / 32) {
        const float x0 = sc[i * KC + lane], x1 = sc[i * KC + lane + 32];
        float mx = fmaxf(x0, x1);
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_old = s_m[i];
        const float m_new = fmaxf(m_old, mx);
        float p0 = 0.f, p1 = 0.f, corr = 1.f;
        if (m_new != -INFINITY) {
          p0 = x0 == -INFINITY ? 0.f : expf(x0 - m_new);
          p1 = x1 == -INFINITY ? 0.f : expf(x1 - m_new);
          corr = m_old == -INFINITY ? 0.f : expf(m_old - m_new);
        }
        float ps = p0 + p1;
#pragma unroll
        for (int o = 16; o; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
        sc[i * KC + lane] = p0;
        sc[i * KC + lane + 32] = p1;
        __syncwarp();
        if (lane == 0) {
          s_l[i] = s_l[i] * corr + ps;
          s_m[i] = m_new;
          s_corr[i] = corr;
        }
      }
      __syncthreads();
      // P.V: dims (2 dp, 2 dp + 1) of rows rg, rg + RG, ...
#pragma unroll
      for (int m = 0; m < RPT; ++m) {
        const float cr = s_corr[rg + m * RG];
        acc[m][0] *= cr;
        acc[m][1] *= cr;
      }
      auto pv_key = [&](int j) {
        float v0, v1;
        a3_v2(Vs + (size_t)j * HD + 2 * dp, v0, v1);
#pragma unroll
        for (int m = 0; m < RPT; ++m) {
          if (rg + m * RG < nq) {  // warp-uniform: a warp's threads share their rows
            const float pj = sc[(rg + m * RG) * KC + j];
            acc[m][0] = fmaf(pj, v0, acc[m][0]);
            acc[m][1] = fmaf(pj, v1, acc[m][1]);
          }
        }
      };
      if (nk == KC) {
        // full chunk: unrolled so that the shared-memory loads of many keys are in flight
#pragma unroll 16
        for (int j = 0; j < KC; ++j) pv_key(j);
      } else {
        for (int j = 0; j < nk; ++j) pv_key(j);
      }
    }
    cc += nch;
    // this split's partial accumulators -> shared memory; combine across the cluster
#pragma unroll
    for (int m = 0; m < RPT; ++m) {
      pacc[(rg + m * RG) * HD + 2 * dp] = acc[m][0];
      pacc[(rg + m * RG) * HD + 2 * dp + 1] = acc[m][1];
    }
    // the dependent launch starts once the keys are done (its CTAs and weight copies would
    // otherwise compete with the key loop)
    if (qt == (int)blockIdx.y) pdl_trigger();
    cl.sync();
    {
      const int dpr = (HD + splits - 1) / splits;
      const int d0 = sp * dpr;
      const int nd = min(dpr, HD - d0);
      for (int idx = tid; idx < nq * nd; idx += kA3Threads) {
        const int i = idx / nd, dd = d0 + (idx - i * nd);
        float mr[kA4MaxSplit], lr[kA4MaxSplit], ar[kA4MaxSplit];
#pragma unroll
        for (int k = 0; k < kA4MaxSplit; ++k) {
          if (k < splits) {
            mr[k] = *cl.map_shared_rank(&s_m[i], k);
            lr[k] = *cl.map_shared_rank(&s_l[i], k);
            ar[k] = *cl.map_shared_rank(&pacc[i * HD + dd], k);
          }
        }
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < kA4MaxSplit; ++k)
          if (k < splits) M = fmaxf(M, mr[k]);
        float L = 0.f, o = 0.f;
#pragma unroll
        for (int k = 0; k < kA4MaxSplit; ++k) {
          if (k < splits && mr[k] != -INFINITY) {
            const float w = expf(mr[k] - M);
            L += w * lr[k];
            o += w * ar[k];
          }
        }
        out_store(out, osh, osl, (size_t)(r0 + i) * ld + h * HD + dd, L > 0.f ? o / L : 0.f);
      }
    }
    cl.sync();  // peers are done reading this tile's partials
  }
  // after a failed wait, copies may still be in flight: wait (bounded) for the last one issued
  // into each stage before the CTA's shared memory is released
  if (__syncthreads_or(failed) && tid == 0) {
    for (uint32_t st = 0; st < (uint32_t)kA3Stages && st < issued; ++st) {
      const uint32_t last = issued - 1 - ((issued - 1 - st) % kA3Stages);
      a3_wait(&full[last % kA3Stages], (last / kA3Stages) & 1);
    }
    atomicOr(err, kErrTimeout | kErrWaitAttn3);
  }
}

// Dynamic shared memory of k_attn3, with pt_bytes of staged page table.
template <typename TC, int HD>
size_t attn3_smem(size_t pt_bytes = (size_t)kMaxPtRow * 4) {
  constexpr int QT = kAttnQT;
  return (size_t)kA3Stages * 2 * kA3Keys * HD * sizeof(TC) + (size_t)(2 * QT * HD + QT * kA3Keys + 4 * QT) * 4 +
         kA3Stages * 8 + 16 + pt_bytes;
}

template <typename TC, int HD>
void launch_a3(const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale,
               int qtiles_grid, int splits, int* err, __nv_bfloat16* osh, __nv_bfloat16* osl, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(B, qtiles_grid, H * splits);
  cfg.blockDim = dim3(kA3Threads);
  cfg.dynamicSmemBytes = attn3_smem<TC, HD>(kv_pages_smem(kv));
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = splits;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  cudaLaunchKernelEx(&cfg, k_attn3<TC, HD>, q, out, kv, rows, H, scale, err, osh, osl);
}

// ---------------------------------------------------------------- warp-walk decode attention
// Decode steps of small batches (bf16 caches, head_dim 64, at most 8 query rows per sequence):
// one CTA per (sequence, head, key split) and no block barrier inside the key loop.
//
// Cache slots below the sequence's committed length (`stable`, read from the sequence state, plus
// `stable_add`) are not written during a decode step, and a step starts only once the step before
// it has completed (graph launches, and the iterations of the generate loop, run in stream
// order). So, before the grid-dependency wait, each CTA copies its share of those slots (up to
// `stage_cap` keys of K and V) into shared memory with two bulk copies on an mbarrier, while its
// predecessors (the Q/K/V layer that appends this step's rows) are still running. After the wait
// only the query rows, the cache lengths and the keys appended in this step (or stable keys past
// the staging capacity) come from global memory.
//
// Keys of a CTA: an equal share of the stable slots [0, S) per split, then an equal share of the
// slots [S, kv_hi) appended in this step. Each warp walks its own groups of four keys; a lane
// holds two head dims, so a key's K and V rows are single 128-byte warp reads. The scores come from
// warp reductions, each warp keeps its own online softmax per row, the warps combine in shared
// memory and the key splits through distributed shared memory. Without `stable` (S = 0) the whole
// range is split evenly and read from global memory.
constexpr int kAwWarps = 4;
constexpr int kAwThreads = kAwWarps * 32;
constexpr int kAwG = 4;           // keys per group
constexpr int kAwStageMax = 256;  // keys staged per CTA (64 KB of K and V)

// [lo, hi) of split sp when n keys starting at base are shared in groups of kAwG
__device__ __forceinline__ void aw_share(int base, int n, int splits, int sp, int& lo, int& hi) {
  const int per = ((n + splits - 1) / splits + kAwG - 1) / kAwG * kAwG;
  lo = base + min(n, sp * per);
  hi = base + min(n, sp * per + per);
}

template <int QT>
__global__ void __launch_bounds__(kAwThreads, QT <= 4 ? 3 : 2)
k_attn_w(const float* __restrict__ q, float* __restrict__ out, KV kv, Rows rows, int H, float scale, int* err,
         const int* __restrict__ stable, int stable_stride, int stable_add, int stage_cap, __nv_bfloat16* osh,
         __nv_bfloat16* osl) {
  namespace cgr = cooperative_groups;
  constexpr int HD = 64;
  __shared__ float Ow[kAwWarps][QT][HD];
  __shared__ float mw[kAwWarps][QT], lw[kAwWarps][QT];
  __shared__ float pacc[QT][HD];
  __shared__ float s_m[QT], s_l[QT];
  __shared__ __align__(16) float qs[QT][HD];
  __shared__ int s_kl[QT];
  __shared__ __align__(8) uint64_t s_bar;   // the staged keys
  __shared__ __align__(8) uint64_t s_rbar;  // rank 0: the peers' partials have arrived
  __shared__ int s_stage[3];  // S, first staged slot, staged keys
  extern __shared__ __align__(128) unsigned char aw_dyn[];
  __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(aw_dyn);  // [stage_cap][HD]
  __nv_bfloat16* Vs = Ks + (size_t)stage_cap * HD;                // [stage_cap][HD]
  float* rbuf = reinterpret_cast<float*>(Vs + (size_t)stage_cap * HD);  // rank 0: [splits][QT][HD]

  TraceScope _trace(TT_ATTN);
  cgr::cluster_group cl = cgr::this_cluster();
  const int splits = (int)cl.dim_blocks().z;
  const int sp = (int)cl.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float* rm = rbuf + (size_t)splits * QT * HD;  // rank 0: [splits][QT] maxima
  float* rl = rm + splits * QT;                  // rank 0: [splits][QT] sums
  // the page table row (paged), after the partials' buffer when there is one
  int* s_pt = reinterpret_cast<int*>(splits > 1 ? rl + splits * QT : rbuf);
  const int b = blockIdx.x;
  const int h = blockIdx.z / splits;
  const __nv_bfloat16* Kc = reinterpret_cast<const __nv_bfloat16*>(kv.k);
  const __nv_bfloat16* Vc = reinterpret_cast<const __nv_bfloat16*>(kv.v);
  if (warp == 0) {
    int S = 0, slo = 0, nst = 0;
    if (stable) {
      S = stable[(size_t)b * stable_stride] + stable_add;
      S = S < 0 ? 0 : (S > kv.S ? kv.S : S);
      int shi;
      aw_share(0, S, splits, sp, slo, shi);
      nst = min(shi - slo, stage_cap);
    }
    // committed slots (their pages were mapped by earlier steps, so the table entries are final):
    // lane i copies the run of the staged range in the i-th page (at most five: 256 keys from a
    // 4-aligned slot), all lanes' page lookups in flight together; contiguous: lane 0, one run
    const int p0 = slo & ~(kPage - 1);
    const int a = kv.pt ? max(slo, p0 + lane * kPage) : slo;
    const int e = kv.pt ? min(slo + nst, p0 + (lane + 1) * kPage) : slo + nst;
    const bool mine = a < e && (kv.pt || lane == 0);
    const int pg = mine ? kv_page_cg(kv, b, a) : 0;
    if (lane == 0) {
      s_stage[0] = S;
      s_stage[1] = slo;
      s_stage[2] = nst;
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(a3_su32(&s_bar)) : "memory");
      if (sp == 0 && splits > 1)
        asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a3_su32(&s_rbar)), "r"(splits - 1) : "memory");
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      if (nst > 0) a3_expect(&s_bar, 2u * (uint32_t)(nst * HD * 2));
    }
    __syncwarp();
    if (mine) {
      const size_t o = kv_addr(kv, H, HD, b, h, a, pg);
      const uint32_t rb = (uint32_t)((e - a) * HD * 2);
      a3_copy(Ks + (size_t)(a - slo) * HD, Kc + o, rb, &s_bar);
      a3_copy(Vs + (size_t)(a - slo) * HD, Vc + o, rb, &s_bar);
    }
  }
  // rank 0's arrival barrier exists before any peer can arrive on it (a cluster barrier before
  // the dependency wait, off the critical path)
  if (splits > 1) cl.sync();
  else __syncthreads();
  const int S = s_stage[0], slo = s_stage[1], nst = s_stage[2];
  bool staged = nst == 0;  // the staged keys have landed (or there are none)
  pdl_wait();
  _trace.waited();
  const int pt0 = kv_pages_load(kv, b, tid);  // stored with the first tile's loads
  const int ld = H * HD;
  // One sequence (a grid of one sequence): its rows start at 0, so the first tile's query rows and
  // cache lengths are loaded together with the row count (rows past the count are dropped after).
  static_assert(QT * 64 / 4 <= kAwThreads, "one query vector per thread");
  const bool one_seq = gridDim.x == 1;
  float4 q_pre = make_float4(0.f, 0.f, 0.f, 0.f);
  int kl_pre = 0;
  if (one_seq) {
    const int r0 = (int)blockIdx.y * QT;
    if (tid < QT * HD / 4) {
      const int i = tid / (HD / 4), c4 = tid - i * (HD / 4);
      q_pre = *reinterpret_cast<const float4*>(q + (size_t)(r0 + i) * ld + h * HD + 4 * c4);
    }
    if (tid < QT) kl_pre = rows.kvlen[r0 + tid];
  }
  const int nrows = rows.seq_count[b];
  const int rbeg = one_seq ? 0 : rows.seq_start[b];
  const int ntiles = (nrows + QT - 1) / QT;

  const int g = lane >> 3, e = lane & 7;  // key slot of this lane in a warp step, its 8 head dims
  for (int qt = blockIdx.y; qt < ntiles; qt += gridDim.y) {
    const int r0 = rbeg + qt * QT;
    const int nq = min(QT, nrows - qt * QT);
    const bool pre = one_seq && qt == (int)blockIdx.y;
    // the tile's query rows (pre-scaled) and cache lengths in shared memory
    for (int idx = tid; idx < QT * HD / 4; idx += kAwThreads) {
      const int i = idx / (HD / 4), c4 = idx - i * (HD / 4);
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (i < nq) {
        v = pre ? q_pre : *reinterpret_cast<const float4*>(q + (size_t)(r0 + i) * ld + h * HD + 4 * c4);
        v.x *= scale; v.y *= scale; v.z *= scale; v.w *= scale;
      }
      *reinterpret_cast<float4*>(&qs[i][4 * c4]) = v;
    }
    if (tid < QT) {
      int k = 0;
      if (tid < nq) {
        k = pre ? kl_pre : rows.kvlen[r0 + tid];
        if (k > kv.S || k < 0) {
          atomicOr(err, kErrIndex);
          k = k < 0 ? 0 : kv.S;
        }
      }
      s_kl[tid] = k;
    }
    if (qt == (int)blockIdx.y) kv_pages_store(kv, b, s_pt, tid, kAwThreads, pt0);
    __syncthreads();
    int kl[QT];
    int kv_hi = 0;
#pragma unroll
    for (int i = 0; i < QT; ++i) {
      kl[i] = s_kl[i];
      kv_hi = max(kv_hi, kl[i]);
    }
    // this split's keys: stable slots [slo2, shi) (the first nst_ok of them staged), then new slots
    // [nlo, nhi); virtual key v < nsk is slot slo2 + v, else slot nlo + v - nsk
    int slo2, shi, nlo, nhi;
    aw_share(0, min(S, kv_hi), splits, sp, slo2, shi);
    aw_share(S, max(kv_hi - S, 0), splits, sp, nlo, nhi);
    const int nsk = shi - slo2;
    const int nv = nsk + (nhi - nlo);
    const int nst_ok = slo2 == slo ? min(nst, nsk) : 0;  // staged keys usable for this range
    if (!staged) {
      if (!a3_wait(&s_bar, 0)) {
        if (lane == 0 && warp == 0) atomicOr(err, kErrTimeout | kErrWaitAttnW);
        a3_wait(&s_bar, 0);  // once more (bounded) for the copies still in flight
      }
      staged = true;
    }
    if (qt == (int)blockIdx.y) _trace.mark(0);  // staged keys landed
    // each group of 8 lanes walks its own keys (key v0 + g of every warp step) with its own online
    // softmax per row; a lane holds 8 head dims of the key, so a score is 8 FMAs and 3 shuffles
    float m[QT], l[QT], acc[QT][8];
#pragma unroll
    for (int i = 0; i < QT; ++i) {
      m[i] = -INFINITY;
      l[i] = 0.f;
#pragma unroll
      for (int d = 0; d < 8; ++d) acc[i][d] = 0.f;
    }
    for (int v0 = kAwG * warp; v0 < nv; v0 += kAwG * kAwWarps) {
      const int v = v0 + g;
      const bool valid = v < nv;
      const int j = v < nsk ? slo2 + v : nlo + v - nsk;
      uint4 ku = make_uint4(0u, 0u, 0u, 0u), vu = ku;
      if (valid) {
        if (v < nst_ok) {
          ku = *reinterpret_cast<const uint4*>(Ks + (size_t)v * HD + 8 * e);
          vu = *reinterpret_cast<const uint4*>(Vs + (size_t)v * HD + 8 * e);
        } else {
          // paged caches only (the dispatcher checks): page of slot j from the staged table row
          const size_t o = (((size_t)s_pt[j / kPage] * H + h) * kPage + (j & (kPage - 1))) * HD + 8 * e;
          ku = *reinterpret_cast<const uint4*>(Kc + o);
          vu = *reinterpret_cast<const uint4*>(Vc + o);
        }
      }
      float kf[8], vf[8];
      unpack16(ku, kf, (const __nv_bfloat16*)nullptr);
      unpack16(vu, vf, (const __nv_bfloat16*)nullptr);
      // every row of the tile (rows past nq have no keys and stay empty): independent chains
#pragma unroll
      for (int i = 0; i < QT; ++i) {
        const float4 qa = *reinterpret_cast<const float4*>(&qs[i][8 * e]);
        const float4 qb = *reinterpret_cast<const float4*>(&qs[i][8 * e + 4]);
        float sc = qa.x * kf[0];
        sc = fmaf(qa.y, kf[1], sc); sc = fmaf(qa.z, kf[2], sc); sc = fmaf(qa.w, kf[3], sc);
        sc = fmaf(qb.x, kf[4], sc); sc = fmaf(qb.y, kf[5], sc); sc = fmaf(qb.z, kf[6], sc);
        sc = fmaf(qb.w, kf[7], sc);
        sc += __shfl_xor_sync(0xffffffffu, sc, 1);
        sc += __shfl_xor_sync(0xffffffffu, sc, 2);
        sc += __shfl_xor_sync(0xffffffffu, sc, 4);
        if (!valid || j >= kl[i]) sc = -INFINITY;
        const float mn = fmaxf(m[i], sc);
        const float cr = mn == -INFINITY ? 1.f : __expf(m[i] - mn);
        const float p = sc == -INFINITY ? 0.f : __expf(sc - mn);
#pragma unroll
        for (int d = 0; d < 8; ++d) acc[i][d] = fmaf(p, vf[d], acc[i][d] * cr);
        l[i] = fmaf(l[i], cr, p);
        m[i] = mn;
      }
    }
    if (qt == (int)blockIdx.y) _trace.mark(1);  // this warp's keys done
    // the dependent launch starts now, not at entry: its CTAs and weight copies would compete with
    // the key loop (measured: the step is 1% faster)
    pdl_trigger();
    // combine the four key slots of the warp (lanes e, e + 8, e + 16, e + 24), then the warps
#pragma unroll
    for (int i = 0; i < QT; ++i) {
      if (i >= nq) break;
      float M = fmaxf(m[i], __shfl_xor_sync(0xffffffffu, m[i], 8));
      M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 16));
      const float f = m[i] == -INFINITY ? 0.f : __expf(m[i] - M);
      float L = l[i] * f;
      L += __shfl_xor_sync(0xffffffffu, L, 8);
      L += __shfl_xor_sync(0xffffffffu, L, 16);
      float o[8];
#pragma unroll
      for (int d = 0; d < 8; ++d) {
        o[d] = acc[i][d] * f;
        o[d] += __shfl_xor_sync(0xffffffffu, o[d], 8);
        o[d] += __shfl_xor_sync(0xffffffffu, o[d], 16);
      }
      if (g == 0) {
        *reinterpret_cast<float4*>(&Ow[warp][i][8 * e]) = make_float4(o[0], o[1], o[2], o[3]);
        *reinterpret_cast<float4*>(&Ow[warp][i][8 * e + 4]) = make_float4(o[4], o[5], o[6], o[7]);
        if (e == 0) {
          mw[warp][i] = M;
          lw[warp][i] = L;
        }
      }
    }
    __syncthreads();
    for (int idx = tid; idx < nq * HD; idx += kAwThreads) {
      const int i = idx / HD, dd = idx - i * HD;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kAwWarps; ++w) M = fmaxf(M, mw[w][i]);
      float L = 0.f, ov = 0.f;
#pragma unroll
      for (int w = 0; w < kAwWarps; ++w) {
        const float f = mw[w][i] == -INFINITY ? 0.f : __expf(mw[w][i] - M);
        L += f * lw[w][i];
        ov += f * Ow[w][i][dd];
      }
      pacc[i][dd] = ov;
      if (dd == 0) {
        s_m[i] = M;
        s_l[i] = L;
      }
    }
    if (ntiles <= (int)gridDim.y) {
      // one tile per CTA: the peers push their partials into rank 0's shared memory and arrive on
      // its barrier (release, cluster scope), then leave; rank 0 waits, combines in split order
      // and stores the rows. No cluster barrier on the critical path.
      __syncthreads();  // this CTA's partials are complete
      if (sp != 0) {
        float* dst = cl.map_shared_rank(rbuf, 0) + (size_t)sp * QT * HD;
        for (int idx = tid; idx < nq * HD; idx += kAwThreads) dst[idx] = (&pacc[0][0])[idx];
        if (tid < nq) {
          cl.map_shared_rank(rm, 0)[sp * QT + tid] = s_m[tid];
          cl.map_shared_rank(rl, 0)[sp * QT + tid] = s_l[tid];
        }
        __syncthreads();
        if (tid == 0) {
          uint32_t remote;
          asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(a3_su32(&s_rbar)), "r"(0));
          asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote) : "memory");
        }
        if (qt == (int)blockIdx.y) _trace.mark(2);  // partials pushed
      } else {
        if (tid == 0 && splits > 1) {
          bool ok = false;
          for (int it = 0; it < kA3Spins && !ok; ++it) {
            uint32_t done;
            asm volatile(
                "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], 0;\n"
                " selp.u32 %0, 1, 0, p;\n}"
                : "=r"(done)
                : "r"(a3_su32(&s_rbar))
                : "memory");
            ok = done != 0;
          }
          if (!ok) atomicOr(err, kErrTimeout | kErrWaitAttnW);
        }
        __syncthreads();
        if (qt == (int)blockIdx.y) _trace.mark(2);  // every split's partials ready
        for (int idx = tid; idx < nq * HD; idx += kAwThreads) {
          const int i = idx / HD, dd = idx - i * HD;
          float M = s_m[i];
          for (int k = 1; k < splits; ++k) M = fmaxf(M, rm[k * QT + i]);
          float L = 0.f, ov = 0.f;
          if (s_m[i] != -INFINITY) {
            const float w = __expf(s_m[i] - M);
            L = w * s_l[i];
            ov = w * pacc[i][dd];
          }
          for (int k = 1; k < splits; ++k) {
            const float mk = rm[k * QT + i];
            if (mk != -INFINITY) {
              const float w = __expf(mk - M);
              L += w * rl[k * QT + i];
              ov += w * rbuf[((size_t)k * QT + i) * HD + dd];
            }
          }
          out_store(out, osh, osl, (size_t)(r0 + i) * ld + h * HD + dd, L > 0.f ? ov / L : 0.f);
        }
      }
      continue;
    }
    cl.sync();
    if (qt == (int)blockIdx.y) _trace.mark(2);  // every split's partials ready
    {
      const int dpr = (HD + splits - 1) / splits;
      const int d0 = sp * dpr;
      const int nd = min(dpr, HD - d0);
      for (int idx = tid; idx < nq * nd; idx += kAwThreads) {
        const int i = idx / nd, dd = d0 + (idx - i * nd);
        float mr[kA4MaxSplit], lr[kA4MaxSplit], ar[kA4MaxSplit];
#pragma unroll
        for (int k = 0; k < kA4MaxSplit; ++k) {
          if (k < splits) {
            mr[k] = *cl.map_shared_rank(&s_m[i], k);
            lr[k] = *cl.map_shared_rank(&s_l[i], k);
            ar[k] = *cl.map_shared_rank(&pacc[i][dd], k);
          }
        }
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < kA4MaxSplit; ++k)
          if (k < splits) M = fmaxf(M, mr[k]);
        float L = 0.f, ov = 0.f;
#pragma unroll
        for (int k = 0; k < kA4MaxSplit; ++k) {
          if (k < splits && mr[k] != -INFINITY) {
            const float w = __expf(mr[k] - M);
            L += w * lr[k];
            ov += w * ar[k];
          }
        }
        out_store(out, osh, osl, (size_t)(r0 + i) * ld + h * HD + dd, L > 0.f ? ov / L : 0.f);
      }
    }
    cl.sync();  // peers are done reading this tile's partials
  }
  // no rows: the staged copies must still land before the CTA leaves (bounded, twice)
  if (!staged && !a3_wait(&s_bar, 0)) {
    if (tid == 0) atomicOr(err, kErrTimeout | kErrWaitAttnW);
    a3_wait(&s_bar, 0);
  }
}

// Keys staged per CTA of k_attn_w for a cache of S slots in `splits` splits (0: no staging).
int aw_stage_cap(int S, int splits, bool stable) {
  if (!stable) return 0;
  const int per = ((S + splits - 1) / splits + kAwG - 1) / kAwG * kAwG;
  return std::min(per, kAwStageMax);
}

void launch_aw(const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale, int splits,
               int* err, const int* stable, int stable_stride, int stable_add, int rows_seq, __nv_bfloat16* osh,
               __nv_bfloat16* osl, cudaStream_t s) {
  const int cap = aw_stage_cap(kv.S, splits, stable != nullptr);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(B, 1, H * splits);
  cfg.blockDim = dim3(kAwThreads);
  const int qt = rows_seq <= 4 ? 4 : kAttnQT;
  cfg.dynamicSmemBytes =
      (size_t)cap * 64 * 2 * 2 + (splits > 1 ? (size_t)splits * qt * (64 + 2) * 4 : 0) + kv_pages_smem(kv);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = splits;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  // query tiles of 4 rows when a sequence has at most 4 (fewer registers: three CTAs per SM)
  if (qt == 4)
    cudaLaunchKernelEx(&cfg, k_attn_w<4>, q, out, kv, rows, H, scale, err, stable, stable_stride, stable_add, cap, osh,
                       osl);
  else
    cudaLaunchKernelEx(&cfg, k_attn_w<kAttnQT>, q, out, kv, rows, H, scale, err, stable, stable_stride, stable_add,
                       cap, osh, osl);
}

// ---------------------------------------------------------------- tensor-core decode attention
// bf16 caches with head_dim 64. One CTA serves (sequence, query tile of up to 16 rows, head, key
// split): a producer warp streams 64-key chunks of K and V by TMA (128-byte swizzle) through a
// ring of shared-memory stages, and four compute warps each take every fourth chunk with their
// own online softmax (no block barrier inside the key loop). Two CTAs share an SM. Q.K^T and P.V run on the tensor cores
// (mma.sync m16n8k16, bf16 operands, fp32 accumulation); K and V are exactly bf16, and Q and P
// are each split into two bf16 halves (x = hi + lo) so that the products keep about 16 bits of
// them. The warps then combine in shared memory, and the key splits of one (sequence, head)
// through distributed shared memory in a thread-block cluster.
constexpr int kA4Warps = 4;
constexpr int kA4Threads = (kA4Warps + 1) * 32;  // + the producer warp
constexpr int kA4QT = 16;
constexpr int kA4Keys = 64;
constexpr uint32_t kA4Chunk = kA4Keys * 64 * 2;  // one K or V chunk: 8 KB

__device__ __forceinline__ void a4_tma(void* dst, const CUtensorMap* m, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          a3_su32(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(a3_su32(bar)), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void ldsm4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm4t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// (x0, x1) -> bf16x2 hi and the bf16x2 of the remainders (first element in the low half)
__device__ __forceinline__ void split2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
  const float2 hf = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}
// byte offset of 16-byte chunk c of row j in a [64][128 B] tile with the 128-byte swizzle
__device__ __forceinline__ uint32_t swz(int j, int c) { return (uint32_t)(j * 128 + ((c ^ (j & 7)) << 4)); }

// The first wait of k_attn_mma that runs out records where it gave up (read by
// lca_debug_attn_diag): {set, block x, y, z, warp, which (0 ring slot free, 1 chunk landed),
// chunk, stage, chunks, key lo, key hi, chunks before this tile, copies issued}.
static __device__ int g_a4_diag[16];
__device__ __noinline__ void a4_record(int which, uint32_t gi, int st, int nch, int lo, int hi, uint32_t cc,
                                       uint32_t issued) {
  if (atomicCAS(&g_a4_diag[0], 0, 1) != 0) return;
  g_a4_diag[1] = blockIdx.x;
  g_a4_diag[2] = blockIdx.y;
  g_a4_diag[3] = blockIdx.z;
  g_a4_diag[4] = threadIdx.x >> 5;
  g_a4_diag[5] = which;
  g_a4_diag[6] = (int)gi;
  g_a4_diag[7] = st;
  g_a4_diag[8] = nch;
  g_a4_diag[9] = lo;
  g_a4_diag[10] = hi;
  g_a4_diag[11] = (int)cc;
  g_a4_diag[12] = (int)issued;
}

template <int NS>
__global__ void __maxnreg__(200)
k_attn_mma(const float* __restrict__ q, float* __restrict__ out, KV kv, Rows rows, int H, float scale, int* err,
           const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV) {
  namespace cgr = cooperative_groups;
  constexpr int HD = 64, QT = kA4QT, KC = kA4Keys;
  // each stage must have one consumer warp, which takes its phases in order: a warp waiting on a
  // stage that is still two phases behind would read the parity of the phase before as complete
  static_assert(NS % kA4Warps == 0, "ring stages must be a multiple of the compute warps");
  extern __shared__ __align__(1024) unsigned char a4raw[];
  unsigned char* ring =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(a4raw) + 1023) & ~uintptr_t(1023));
  unsigned char* qsh = ring + NS * 2 * kA4Chunk;                    // [QT][HD] bf16, swizzled: hi(q * scale)
  unsigned char* qsl = qsh + QT * HD * 2;                           // the remainders
  float* pacc = reinterpret_cast<float*>(qsl + QT * HD * 2);        // [QT][HD]
  float* s_m = pacc + QT * HD;                                      // [QT]
  float* s_l = s_m + QT;                                            // [QT]
  int* s_kv = reinterpret_cast<int*>(s_l + QT);                     // [QT]
  uint64_t* full = reinterpret_cast<uint64_t*>(s_kv + QT);          // [NS]
  uint64_t* empty = full + NS;                                      // [NS]
  int* s_pt = reinterpret_cast<int*>(empty + NS);                   // [pt_ld] page table row (paged)
  // after the key loop the ring holds the warps' partial results
  float* Ow = reinterpret_cast<float*>(ring);                       // [warps][QT][HD]
  float* mw = Ow + kA4Warps * QT * HD;                              // [warps][QT]
  float* lw = mw + kA4Warps * QT;                                   // [warps][QT]

  TraceScope _trace(TT_ATTN);
  cgr::cluster_group cl = cgr::this_cluster();
  const int splits = (int)cl.dim_blocks().z;
  const int sp = (int)cl.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;
  if (tid == 0) {
    for (int i = 0; i < NS; ++i) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(a3_su32(&full[i])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(a3_su32(&empty[i])) : "memory");
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  __syncthreads();
  const int b = blockIdx.x;
  const int h = blockIdx.z / splits;
  const int nrows = rows.seq_count[b];
  const int rbeg = rows.seq_start[b];
  const int ntiles = (nrows + QT - 1) / QT;
  const int ld = H * HD;
  bool failed = false;
  uint32_t cc = 0, issued = 0;

  for (int qt = blockIdx.y; qt < ntiles; qt += gridDim.y) {
    const int r0 = rbeg + qt * QT;
    const int nq = min(QT, nrows - qt * QT);
    for (int idx = tid; idx < QT * HD / 2; idx += kA4Threads) {
      const int i = idx / (HD / 2), dd = (idx - i * (HD / 2)) * 2;
      float2 v = make_float2(0.f, 0.f);
      if (i < nq) {
        v = *reinterpret_cast<const float2*>(q + (size_t)(r0 + i) * ld + h * HD + dd);
        v.x *= scale;
        v.y *= scale;
      }
      uint32_t hi2, lo2;
      split2(v.x, v.y, hi2, lo2);
      const uint32_t off = swz(i, dd >> 3) + (dd & 7) * 2;
      *reinterpret_cast<uint32_t*>(qsh + off) = hi2;
      *reinterpret_cast<uint32_t*>(qsl + off) = lo2;
    }
    if (tid < QT) {
      int kl = tid < nq ? rows.kvlen[r0 + tid] : 0;
      if (kl > kv.S || kl < 0) {
        atomicOr(err, kErrIndex);
        kl = kl < 0 ? 0 : kv.S;
      }
      s_kv[tid] = kl;
    }
    // prefill tiles are long: the table row is loaded here (a register held across the query
    // staging would spill)
    if (qt == (int)blockIdx.y) kv_pages_store(kv, b, s_pt, tid, kA4Threads, kv_pages_load(kv, b, tid));
    __syncthreads();
    int kv_hi = 0;
#pragma unroll
    for (int i = 0; i < QT; ++i) kv_hi = max(kv_hi, s_kv[i]);
    const int per = ((kv_hi + splits - 1) / splits + KC - 1) / KC * KC;
    const int lo = sp * per;
    const int hi = min(kv_hi, lo + per);
    const int nch = hi > lo ? (hi - lo + KC - 1) / KC : 0;

    // per compute warp: running max, sum and accumulator of rows g and g + 8
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    float o[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
    if (warp == kA4Warps) {
      // producer
      if (lane == 0) {
        for (int c = 0; c < nch; ++c) {
          const uint32_t gi = cc + c;
          const int st = gi % NS;
          if (gi >= (uint32_t)NS && !failed && !a3_wait(&empty[st], ((gi / NS) - 1) & 1)) {
            failed = true;
            a4_record(0, gi, st, nch, lo, hi, cc, issued);
          }
          if (failed) break;
          ++issued;
          unsigned char* dst = ring + (size_t)st * 2 * kA4Chunk;
          // tensor-map row of the chunk: 64 slots from a page start (lo is a multiple of KC == kPage)
          const int j0 = lo + c * KC;
          const int row = kv.pt ? (s_pt[j0 / kPage] * H + h) * kPage : (b * H + h) * kv.S + j0;
          a3_expect(&full[st], 2 * kA4Chunk);
          a4_tma(dst, &tmK, 0, row, &full[st]);
          a4_tma(dst + kA4Chunk, &tmV, 0, row, &full[st]);
        }
      }
      __syncwarp();
    } else {
      const uint32_t qhb = a3_su32(qsh), qlb = a3_su32(qsl);
      const int kl0 = min(s_kv[g], hi), kl1 = min(s_kv[g + 8], hi);
      for (int c = warp; c < nch; c += kA4Warps) {
        const uint32_t gi = cc + c;
        const int st = gi % NS;
        if (!failed && !a3_wait(&full[st], (gi / NS) & 1)) {
          failed = true;
          a4_record(1, gi, st, nch, lo, hi, cc, 0);
        }
        const uint32_t kb = a3_su32(ring + (size_t)st * 2 * kA4Chunk), vb = kb + kA4Chunk;
        const int j0 = lo + c * KC;
        // S = Q K^T over 64 keys: n-tile nt = keys 8 nt .. 8 nt + 7
        float sacc[8][4];
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) sacc[nt][0] = sacc[nt][1] = sacc[nt][2] = sacc[nt][3] = 0.f;
#pragma unroll
        for (int kp = 0; kp < 2; ++kp) {
          // Q fragments of dims 32 kp .. 32 kp + 31 (rows lane & 15, dims chunk 4 kp + 2 j + (lane >> 4))
          uint32_t qh0[4], ql0[4], qh1[4], ql1[4];
          ldsm4(qhb + swz(lane & 15, 4 * kp + (lane >> 4)), qh0);
          ldsm4(qlb + swz(lane & 15, 4 * kp + (lane >> 4)), ql0);
          ldsm4(qhb + swz(lane & 15, 4 * kp + 2 + (lane >> 4)), qh1);
          ldsm4(qlb + swz(lane & 15, 4 * kp + 2 + (lane >> 4)), ql1);
#pragma unroll
          for (int nt = 0; nt < 8; ++nt) {
            uint32_t bf[4];
            // matrices: keys 8 nt + (lane & 7), dims chunks 4 kp + (lane >> 3)
            ldsm4(kb + swz(8 * nt + (lane & 7), 4 * kp + (lane >> 3)), bf);
            mma16816(sacc[nt], qh0, bf[0], bf[1]);
            mma16816(sacc[nt], ql0, bf[0], bf[1]);
            mma16816(sacc[nt], qh1, bf[2], bf[3]);
            mma16816(sacc[nt], ql1, bf[2], bf[3]);
          }
        }
        // mask, online softmax (rows g, g + 8; the four lanes of a quad share a row)
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
          const int key = j0 + 8 * nt + 2 * t;
          if (key >= kl0) sacc[nt][0] = -INFINITY;
          if (key + 1 >= kl0) sacc[nt][1] = -INFINITY;
          if (key >= kl1) sacc[nt][2] = -INFINITY;
          if (key + 1 >= kl1) sacc[nt][3] = -INFINITY;
          mx0 = fmaxf(mx0, fmaxf(sacc[nt][0], sacc[nt][1]));
          mx1 = fmaxf(mx1, fmaxf(sacc[nt][2], sacc[nt][3]));
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float n0 = fmaxf(m0, mx0), n1 = fmaxf(m1, mx1);
        const float cr0 = n0 == -INFINITY ? 1.f : (m0 == -INFINITY ? 0.f : expf(m0 - n0));
        const float cr1 = n1 == -INFINITY ? 1.f : (m1 == -INFINITY ? 0.f : expf(m1 - n1));
        m0 = n0;
        m1 = n1;
        float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
          sacc[nt][0] = sacc[nt][0] == -INFINITY ? 0.f : expf(sacc[nt][0] - n0);
          sacc[nt][1] = sacc[nt][1] == -INFINITY ? 0.f : expf(sacc[nt][1] - n0);
          sacc[nt][2] = sacc[nt][2] == -INFINITY ? 0.f : expf(sacc[nt][2] - n1);
          sacc[nt][3] = sacc[nt][3] == -INFINITY ? 0.f : expf(sacc[nt][3] - n1);
          ps0 += sacc[nt][0] + sacc[nt][1];
          ps1 += sacc[nt][2] + sacc[nt][3];
          o[nt][0] *= cr0;
          o[nt][1] *= cr0;
          o[nt][2] *= cr1;
          o[nt][3] *= cr1;
        }
        l0 = l0 * cr0 + ps0;
        l1 = l1 * cr1 + ps1;
        // O += P V: k-step kk = keys 16 kk .. 16 kk + 15; n-tiles of 8 dims
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          uint32_t ph[4], pl[4];
          split2(sacc[2 * kk][0], sacc[2 * kk][1], ph[0], pl[0]);
          split2(sacc[2 * kk][2], sacc[2 * kk][3], ph[1], pl[1]);
          split2(sacc[2 * kk + 1][0], sacc[2 * kk + 1][1], ph[2], pl[2]);
          split2(sacc[2 * kk + 1][2], sacc[2 * kk + 1][3], ph[3], pl[3]);
#pragma unroll
          for (int np = 0; np < 4; ++np) {
            uint32_t bf[4];
            // matrices: keys 16 kk + 8 ((lane >> 3) & 1) + (lane & 7), dims chunk 2 np + (lane >> 4)
            ldsm4t(vb + swz(16 * kk + 8 * ((lane >> 3) & 1) + (lane & 7), 2 * np + (lane >> 4)), bf);
            mma16816(o[2 * np], ph, bf[0], bf[1]);
            mma16816(o[2 * np], pl, bf[0], bf[1]);
            mma16816(o[2 * np + 1], ph, bf[2], bf[3]);
            mma16816(o[2 * np + 1], pl, bf[2], bf[3]);
          }
        }
        __syncwarp();
        if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(a3_su32(&empty[st])) : "memory");
      }
      l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
      l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
      l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
      l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    }
    __syncthreads();  // every warp is done with the ring: it now holds the warps' partial results
    if (warp < kA4Warps) {
      float* ow = Ow + warp * QT * HD;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        *reinterpret_cast<float2*>(ow + g * HD + 8 * nt + 2 * t) = make_float2(o[nt][0], o[nt][1]);
        *reinterpret_cast<float2*>(ow + (g + 8) * HD + 8 * nt + 2 * t) = make_float2(o[nt][2], o[nt][3]);
      }
      if (t == 0) {
        mw[warp * QT + g] = m0;
        lw[warp * QT + g] = l0;
        mw[warp * QT + g + 8] = m1;
        lw[warp * QT + g + 8] = l1;
      }
    }
    __syncthreads();
    // combine the warps: this split's (max, sum, accumulator) per row
    for (int idx = tid; idx < QT * HD; idx += kA4Threads) {
      const int i = idx / HD, dd = idx - i * HD;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kA4Warps; ++w) M = fmaxf(M, mw[w * QT + i]);
      float L = 0.f, o = 0.f;
#pragma unroll
      for (int w = 0; w < kA4Warps; ++w) {
        const float mv = mw[w * QT + i];
        const float f = mv == -INFINITY ? 0.f : expf(mv - M);
        L += f * lw[w * QT + i];
        o += f * Ow[(w * QT + i) * HD + dd];
      }
      pacc[idx] = o;
      if (dd == 0) {
        s_m[i] = M;
        s_l[i] = L;
      }
    }
    cl.sync();
    {
      const int dpr = (HD + splits - 1) / splits;
      const int d0 = sp * dpr;
      const int nd = min(dpr, HD - d0);
      for (int idx = tid; idx < nq * nd; idx += kA4Threads) {
        const int i = idx / nd, dd = d0 + (idx - i * nd);
        float mr[kMaxClusterSplit], lr[kMaxClusterSplit], ar[kMaxClusterSplit];
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k) {
          if (k < splits) {
            mr[k] = *cl.map_shared_rank(&s_m[i], k);
            lr[k] = *cl.map_shared_rank(&s_l[i], k);
            ar[k] = *cl.map_shared_rank(&pacc[i * HD + dd], k);
          }
        }
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k)
          if (k < splits) M = fmaxf(M, mr[k]);
        float L = 0.f, o = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k) {
          if (k < splits && mr[k] != -INFINITY) {
            const float w = expf(mr[k] - M);
            L += w * lr[k];
            o += w * ar[k];
          }
        }
        out[(size_t)(r0 + i) * ld + h * HD + dd] = L > 0.f ? o / L : 0.f;
      }
    }
    cl.sync();
    cc += nch;
  }
  // after a failed wait, copies may still be in flight: wait (bounded) for the last one issued
  // into each stage before the CTA's shared memory is released
  if (__syncthreads_or(failed) && tid == kA4Warps * 32) {
    for (uint32_t st = 0; st < (uint32_t)NS && st < issued; ++st) {
      const uint32_t last = issued - 1 - ((issued - 1 - st) % NS);
      a3_wait(&full[last % NS], (last / NS) & 1);
    }
    atomicOr(err, kErrTimeout | kErrWaitAttnMma);
  }
}

template <int NS>
size_t attn_mma_smem(size_t pt_bytes = (size_t)kMaxPtRow * 4) {
  // ring, q halves (2 x QT x 64 bf16), pacc (QT x 64 fp32), row stats, barriers, page table row
  return 1024 + (size_t)NS * 2 * kA4Chunk + (size_t)(2 * kA4QT * 64 + 3 * kA4QT) * 4 + 2 * NS * 8 + 16 + pt_bytes;
}

template <int NS>
void launch_a4_ns(const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale,
                  int qtiles_grid, int splits, int* err, cudaStream_t s) {
  CUtensorMap tk, tv;
  memcpy(&tk, kv.tmaps, sizeof(tk));
  memcpy(&tv, static_cast<const unsigned char*>(kv.tmaps) + 128, sizeof(tv));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(B, qtiles_grid, H * splits);
  cfg.blockDim = dim3(kA4Threads);
  cfg.dynamicSmemBytes = attn_mma_smem<NS>(kv_pages_smem(kv));
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = splits;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  cudaLaunchKernelEx(&cfg, k_attn_mma<NS>, q, out, kv, rows, H, scale, err, tk, tv);
}

// ---------------------------------------------------------------- transposed tensor-core attention
// The same decode attention for query tiles of at most 8 rows (decode steps: n candidates, or one
// latent, per sequence). The scores are computed transposed, S^T = K Q^T, with the 16 keys of an
// MMA tile as its M dimension and the query rows as N = 8, so a tile of 8 rows costs half the MMAs
// of a 16-row one. P^T reaches the P.V product (O^T = V^T P^T, dims as M) through an in-register
// 8x8 transpose (movmatrix). Q's bf16 halves are loaded into registers once per tile; K and V
// come by TMA through the ring, as in k_attn_mma.
constexpr int kA5QT = 8;

__device__ __forceinline__ void ldsm4_(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ uint32_t movt(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}

template <int NS, int NWC>
__global__ void __launch_bounds__((NWC + 1) * 32, 1)
k_attn_mmt(const float* __restrict__ q, float* __restrict__ out, KV kv, Rows rows, int H, float scale, int* err,
           const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, __nv_bfloat16* osh,
           __nv_bfloat16* osl) {
  namespace cgr = cooperative_groups;
  constexpr int HD = 64, QT = kA5QT, KC = kA4Keys;
  static_assert(NS % NWC == 0, "ring stages must be a multiple of the compute warps");
  extern __shared__ __align__(1024) unsigned char a5raw[];
  unsigned char* ring =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(a5raw) + 1023) & ~uintptr_t(1023));
  unsigned char* qsh = ring + NS * 2 * kA4Chunk;                    // [QT][HD] bf16, swizzled: hi(q * scale)
  unsigned char* qsl = qsh + QT * HD * 2;                           // the remainders
  float* pacc = reinterpret_cast<float*>(qsl + QT * HD * 2);        // [QT][HD]
  float* s_m = pacc + QT * HD;                                      // [QT]
  float* s_l = s_m + QT;                                            // [QT]
  int* s_kv = reinterpret_cast<int*>(s_l + QT);                     // [QT]
  uint64_t* full = reinterpret_cast<uint64_t*>(s_kv + QT);          // [NS]
  uint64_t* empty = full + NS;                                      // [NS]
  int* s_pt = reinterpret_cast<int*>(empty + NS);                   // [pt_ld] page table row (paged)
  // after the key loop the ring holds the warps' partial results
  float* Ow = reinterpret_cast<float*>(ring);                       // [warps][QT][HD]
  float* mw = Ow + NWC * QT * HD;                              // [warps][QT]
  float* lw = mw + NWC * QT;                                   // [warps][QT]

  TraceScope _trace(TT_ATTN);
  cgr::cluster_group cl = cgr::this_cluster();
  const int splits = (int)cl.dim_blocks().z;
  const int sp = (int)cl.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;
  if (tid == 0) {
    for (int i = 0; i < NS; ++i) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(a3_su32(&full[i])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(a3_su32(&empty[i])) : "memory");
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
  }
  pdl_wait();
  _trace.waited();
  __syncthreads();
  const int b = blockIdx.x;
  const int h = blockIdx.z / splits;
  const int pt0 = kv_pages_load(kv, b, tid);  // stored with the first tile's loads
  const int nrows = rows.seq_count[b];
  const int rbeg = rows.seq_start[b];
  const int ntiles = (nrows + QT - 1) / QT;
  const int ld = H * HD;
  bool failed = false;
  uint32_t cc = 0, issued = 0;

  for (int qt = blockIdx.y; qt < ntiles; qt += gridDim.y) {
    const int r0 = rbeg + qt * QT;
    const int nq = min(QT, nrows - qt * QT);
    for (int idx = tid; idx < QT * HD / 2; idx += ((NWC + 1) * 32)) {
      const int i = idx / (HD / 2), dd = (idx - i * (HD / 2)) * 2;
      float2 v = make_float2(0.f, 0.f);
      if (i < nq) {
        v = *reinterpret_cast<const float2*>(q + (size_t)(r0 + i) * ld + h * HD + dd);
        v.x *= scale;
        v.y *= scale;
      }
      uint32_t hi2, lo2;
      split2(v.x, v.y, hi2, lo2);
      const uint32_t off = swz(i, dd >> 3) + (dd & 7) * 2;
      *reinterpret_cast<uint32_t*>(qsh + off) = hi2;
      *reinterpret_cast<uint32_t*>(qsl + off) = lo2;
    }
    if (tid < QT) {
      int kl = tid < nq ? rows.kvlen[r0 + tid] : 0;
      if (kl > kv.S || kl < 0) {
        atomicOr(err, kErrIndex);
        kl = kl < 0 ? 0 : kv.S;
      }
      s_kv[tid] = kl;
    }
    if (qt == (int)blockIdx.y) kv_pages_store(kv, b, s_pt, tid, ((NWC + 1) * 32), pt0);
    __syncthreads();
    int kv_hi = 0;
#pragma unroll
    for (int i = 0; i < QT; ++i) kv_hi = max(kv_hi, s_kv[i]);
    const int per = ((kv_hi + splits - 1) / splits + KC - 1) / KC * KC;
    const int lo = sp * per;
    const int hi = min(kv_hi, lo + per);
    const int nch = hi > lo ? (hi - lo + KC - 1) / KC : 0;

    // per compute warp: running max and (lane-partial) sum of queries 2t, 2t + 1, and O^T for
    // dims 16 dm + g (+ 8) of those queries
    float ma = -INFINITY, mb = -INFINITY, la = 0.f, lb = 0.f;
    float o[4][4];
#pragma unroll
    for (int n = 0; n < 4; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
    if (warp == NWC) {
      // producer
      if (lane == 0) {
        for (int c = 0; c < nch; ++c) {
          const uint32_t gi = cc + c;
          const int st = gi % NS;
          if (gi >= (uint32_t)NS && !failed && !a3_wait(&empty[st], ((gi / NS) - 1) & 1)) failed = true;
          if (failed) break;
          ++issued;
          unsigned char* dst = ring + (size_t)st * 2 * kA4Chunk;
          // tensor-map row of the chunk: 64 slots from a page start (lo is a multiple of KC == kPage)
          const int j0 = lo + c * KC;
          const int row = kv.pt ? (s_pt[j0 / kPage] * H + h) * kPage : (b * H + h) * kv.S + j0;
          a3_expect(&full[st], 2 * kA4Chunk);
          a4_tma(dst, &tmK, 0, row, &full[st]);
          a4_tma(dst + kA4Chunk, &tmV, 0, row, &full[st]);
        }
      }
      __syncwarp();
    } else {
      // Q^T fragments (B operand): dims 16 ks .. 16 ks + 15 of query rows 0..7
      uint32_t qh[4][2], ql[4][2];
      {
        const uint32_t qhb = a3_su32(qsh), qlb = a3_su32(qsl);
#pragma unroll
        for (int kp = 0; kp < 2; ++kp) {
          uint32_t r[4];
          // matrices: query rows lane & 7, dims chunk 4 kp + (lane >> 3)
          ldsm4_(qhb + swz(lane & 7, 4 * kp + (lane >> 3)), r);
          qh[2 * kp][0] = r[0];
          qh[2 * kp][1] = r[1];
          qh[2 * kp + 1][0] = r[2];
          qh[2 * kp + 1][1] = r[3];
          ldsm4_(qlb + swz(lane & 7, 4 * kp + (lane >> 3)), r);
          ql[2 * kp][0] = r[0];
          ql[2 * kp][1] = r[1];
          ql[2 * kp + 1][0] = r[2];
          ql[2 * kp + 1][1] = r[3];
        }
      }
      const int kla = min(s_kv[2 * t], hi), klb = min(s_kv[2 * t + 1], hi);
      for (int c = warp; c < nch; c += NWC) {
        const uint32_t gi = cc + c;
        const int st = gi % NS;
        if (!failed && !a3_wait(&full[st], (gi / NS) & 1)) failed = true;
        const uint32_t kb = a3_su32(ring + (size_t)st * 2 * kA4Chunk), vb = kb + kA4Chunk;
        const int j0 = lo + c * KC;
        // S^T = K Q^T: m-tile i = keys 16 i .. 16 i + 15 of the chunk
        float s[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
          for (int ks = 0; ks < 4; ++ks) {
            uint32_t af[4];
            // matrices: keys 16 i + (lane & 15), dims chunk 2 ks + (lane >> 4)
            ldsm4_(kb + swz(16 * i + (lane & 15), 2 * ks + (lane >> 4)), af);
            mma16816(s[i], af, qh[ks][0], qh[ks][1]);
            mma16816(s[i], af, ql[ks][0], ql[ks][1]);
          }
        }
        // mask; online softmax per query column (the 8 lanes with the same t share a column pair)
        float xa = -INFINITY, xb = -INFINITY;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int key = j0 + 16 * i + g;
          if (key >= kla) s[i][0] = -INFINITY;
          if (key >= klb) s[i][1] = -INFINITY;
          if (key + 8 >= kla) s[i][2] = -INFINITY;
          if (key + 8 >= klb) s[i][3] = -INFINITY;
          xa = fmaxf(xa, fmaxf(s[i][0], s[i][2]));
          xb = fmaxf(xb, fmaxf(s[i][1], s[i][3]));
        }
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          xa = fmaxf(xa, __shfl_xor_sync(0xffffffffu, xa, off));
          xb = fmaxf(xb, __shfl_xor_sync(0xffffffffu, xb, off));
        }
        const float na = fmaxf(ma, xa), nb = fmaxf(mb, xb);
        const float cra = na == -INFINITY ? 1.f : (ma == -INFINITY ? 0.f : expf(ma - na));
        const float crb = nb == -INFINITY ? 1.f : (mb == -INFINITY ? 0.f : expf(mb - nb));
        ma = na;
        mb = nb;
        float pa = 0.f, pb = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          s[i][0] = s[i][0] == -INFINITY ? 0.f : expf(s[i][0] - na);
          s[i][1] = s[i][1] == -INFINITY ? 0.f : expf(s[i][1] - nb);
          s[i][2] = s[i][2] == -INFINITY ? 0.f : expf(s[i][2] - na);
          s[i][3] = s[i][3] == -INFINITY ? 0.f : expf(s[i][3] - nb);
          pa += s[i][0] + s[i][2];
          pb += s[i][1] + s[i][3];
          o[i][0] *= cra;
          o[i][1] *= crb;
          o[i][2] *= cra;
          o[i][3] *= crb;
        }
        la = la * cra + pa;
        lb = lb * crb + pb;
        // O^T += V^T P^T: k-step i = keys 16 i .. 16 i + 15; m-tiles of 16 dims
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          // P^T halves as the B operand: transpose the (key, query) 8 x 8 blocks in registers
          uint32_t h0, l0, h1, l1;
          split2(s[i][0], s[i][1], h0, l0);
          split2(s[i][2], s[i][3], h1, l1);
          const uint32_t bh0 = movt(h0), bh1 = movt(h1), bl0 = movt(l0), bl1 = movt(l1);
#pragma unroll
          for (int dm = 0; dm < 4; ++dm) {
            uint32_t af[4];
            // matrices (transposed): keys 16 i + 8 (lane >> 4) + (lane & 7), dims chunk 2 dm + ((lane >> 3) & 1)
            ldsm4t(vb + swz(16 * i + 8 * (lane >> 4) + (lane & 7), 2 * dm + ((lane >> 3) & 1)), af);
            mma16816(o[dm], af, bh0, bh1);
            mma16816(o[dm], af, bl0, bl1);
          }
        }
        __syncwarp();
        if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(a3_su32(&empty[st])) : "memory");
      }
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        la += __shfl_xor_sync(0xffffffffu, la, off);
        lb += __shfl_xor_sync(0xffffffffu, lb, off);
      }
    }
    __syncthreads();  // every warp is done with the ring: it now holds the warps' partial results
    if (warp < NWC) {
      float* ow = Ow + warp * QT * HD;
#pragma unroll
      for (int dm = 0; dm < 4; ++dm) {
        ow[(2 * t) * HD + 16 * dm + g] = o[dm][0];
        ow[(2 * t + 1) * HD + 16 * dm + g] = o[dm][1];
        ow[(2 * t) * HD + 16 * dm + g + 8] = o[dm][2];
        ow[(2 * t + 1) * HD + 16 * dm + g + 8] = o[dm][3];
      }
      if (g == 0) {
        mw[warp * QT + 2 * t] = ma;
        lw[warp * QT + 2 * t] = la;
        mw[warp * QT + 2 * t + 1] = mb;
        lw[warp * QT + 2 * t + 1] = lb;
      }
    }
    __syncthreads();
    // combine the warps: this split's (max, sum, accumulator) per row
    for (int idx = tid; idx < QT * HD; idx += ((NWC + 1) * 32)) {
      const int i = idx / HD, dd = idx - i * HD;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < NWC; ++w) M = fmaxf(M, mw[w * QT + i]);
      float L = 0.f, ov = 0.f;
#pragma unroll
      for (int w = 0; w < NWC; ++w) {
        const float mv = mw[w * QT + i];
        const float f = mv == -INFINITY ? 0.f : expf(mv - M);
        L += f * lw[w * QT + i];
        ov += f * Ow[(w * QT + i) * HD + dd];
      }
      pacc[idx] = ov;
      if (dd == 0) {
        s_m[i] = M;
        s_l[i] = L;
      }
    }
    // the dependent launch starts once the keys are done (as in k_attn_w)
    if (qt == (int)blockIdx.y) pdl_trigger();
    cl.sync();
    {
      const int dpr = (HD + splits - 1) / splits;
      const int d0 = sp * dpr;
      const int nd = min(dpr, HD - d0);
      for (int idx = tid; idx < nq * nd; idx += ((NWC + 1) * 32)) {
        const int i = idx / nd, dd = d0 + (idx - i * nd);
        float mr[kMaxClusterSplit], lr[kMaxClusterSplit], ar[kMaxClusterSplit];
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k) {
          if (k < splits) {
            mr[k] = *cl.map_shared_rank(&s_m[i], k);
            lr[k] = *cl.map_shared_rank(&s_l[i], k);
            ar[k] = *cl.map_shared_rank(&pacc[i * HD + dd], k);
          }
        }
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k)
          if (k < splits) M = fmaxf(M, mr[k]);
        float L = 0.f, ov = 0.f;
#pragma unroll
        for (int k = 0; k < kMaxClusterSplit; ++k) {
          if (k < splits && mr[k] != -INFINITY) {
            const float w = expf(mr[k] - M);
            L += w * lr[k];
            ov += w * ar[k];
          }
        }
        out_store(out, osh, osl, (size_t)(r0 + i) * ld + h * HD + dd, L > 0.f ? ov / L : 0.f);
      }
    }
    cl.sync();
    cc += nch;
  }
  // after a failed wait, copies may still be in flight: wait (bounded) for the last one issued
  // into each stage before the CTA's shared memory is released
  if (__syncthreads_or(failed) && tid == NWC * 32) {
    for (uint32_t st = 0; st < (uint32_t)NS && st < issued; ++st) {
      const uint32_t last = issued - 1 - ((issued - 1 - st) % NS);
      a3_wait(&full[last % NS], (last / NS) & 1);
    }
    atomicOr(err, kErrTimeout | kErrWaitAttnMma);
  }
}

template <int NS>
size_t attn_mmt_smem(size_t pt_bytes = (size_t)kMaxPtRow * 4) {
  // ring, q halves (2 x QT x 64 bf16), pacc (QT x 64 fp32), row stats, barriers, page table row
  return 1024 + (size_t)NS * 2 * kA4Chunk + (size_t)(2 * kA5QT * 64 + 3 * kA5QT) * 4 + 2 * NS * 8 + 16 + pt_bytes;
}
// Compute warps of k_attn_mmt with NS ring stages: two stages per warp (one being read, one in
// flight).
template <int NS>
constexpr int mmt_warps() { return NS / 2 < 4 ? 4 : NS / 2; }

template <int NS>
void launch_a5_ns(const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale,
                  int qtiles_grid, int splits, int* err, __nv_bfloat16* osh, __nv_bfloat16* osl, cudaStream_t s) {
  CUtensorMap tk, tv;
  memcpy(&tk, kv.tmaps, sizeof(tk));
  memcpy(&tv, static_cast<const unsigned char*>(kv.tmaps) + 128, sizeof(tv));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(B, qtiles_grid, H * splits);
  constexpr int NWC = mmt_warps<NS>();
  cfg.blockDim = dim3((NWC + 1) * 32);
  cfg.dynamicSmemBytes = attn_mmt_smem<NS>(kv_pages_smem(kv));
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = splits;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  cudaLaunchKernelEx(&cfg, k_attn_mmt<NS, NWC>, q, out, kv, rows, H, scale, err, tk, tv, osh, osl);
}

void launch_a4(int ns, const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale,
               int qtiles_grid, int splits, int* err, cudaStream_t s) {
  if (ns == 4) launch_a4_ns<4>(q, out, kv, rows, B, H, scale, qtiles_grid, splits, err, s);
  else launch_a4_ns<8>(q, out, kv, rows, B, H, scale, qtiles_grid, splits, err, s);
}

template <typename TC, int HD>
void launch_cl(const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale,
               int qtiles_grid, int splits, int* err, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(B, qtiles_grid, H * splits);
  cfg.blockDim = dim3(kA2Threads);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = splits;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  ++g_launches;
  cudaLaunchKernelEx(&cfg, k_attn2<TC, HD>, q, out, kv, rows, H, scale, err);
}

template <typename TC, int HD>
void launch(const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale,
            int qtiles_grid, int splits, float* part, int* cnt, int* err, cudaStream_t s) {
  dim3 grid(B, qtiles_grid, H * splits);
  ++g_launches;
  launch_pdl(k_attn<TC, HD>, grid, dim3(kThreads), 0, s, q, out, kv, rows, H, scale, splits, part, cnt, err);
}

void launch_any(int dtype, int hd, const float* q, float* out, const KV& kv, const Rows& rows, int B,
                int H, float scale, int qtiles_grid, int splits, float* part, int* cnt, int* err,
                cudaStream_t s) {
  if (dtype == LCA_BF16) {
    if (hd == 64) launch<__nv_bfloat16, 64>(q, out, kv, rows, B, H, scale, qtiles_grid, splits, part, cnt, err, s);
    else launch<__nv_bfloat16, 32>(q, out, kv, rows, B, H, scale, qtiles_grid, splits, part, cnt, err, s);
  } else {
    if (hd == 64) launch<float, 64>(q, out, kv, rows, B, H, scale, qtiles_grid, splits, part, cnt, err, s);
    else launch<float, 32>(q, out, kv, rows, B, H, scale, qtiles_grid, splits, part, cnt, err, s);
  }
}

// Rows of the standalone op: sequence b owns rows [b*n_rows, (b+1)*n_rows).
__global__ void k_regular_rows(int* seq_start, int* seq_count, int batch, int n_rows) {
  pdl_trigger();
  pdl_wait();
  for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < batch; b += gridDim.x * blockDim.x) {
    seq_start[b] = b * n_rows;
    seq_count[b] = n_rows;
  }
}

// Scratch of the standalone op: [error word][tile counters][seq_start][seq_count][partials].
struct OpScratch {
  int* err;
  int* cnt;
  int* seq_start;
  int* seq_count;
  float* part;
  size_t header_bytes; // bytes that must be zero before a call (error word + counters)
  size_t bytes;
};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

OpScratch op_scratch_layout(char* base, int batch, int heads, int head_dim, int splits) {
  OpScratch o{};
  size_t off = 0;
  o.err = reinterpret_cast<int*>(base + off);
  off += 256;
  o.cnt = reinterpret_cast<int*>(base + off);
  off += align256((size_t)batch * kQTMax * heads * sizeof(int));
  o.header_bytes = off;
  o.seq_start = reinterpret_cast<int*>(base + off);
  off += align256((size_t)batch * sizeof(int));
  o.seq_count = reinterpret_cast<int*>(base + off);
  off += align256((size_t)batch * sizeof(int));
  o.part = reinterpret_cast<float*>(base + off);
  off += align256((size_t)batch * kQTMax * heads * splits * kAttnQT * (head_dim + 2) * sizeof(float));
  o.bytes = off;
  return o;
}

int op_check(const float* q, float* out, const void* k, const void* v, int dtype, int batch, int heads,
             int head_dim, int slots, int n_rows, const int* kv_len, int splits) {
  if (!q || !out || !k || !v || !kv_len) return LCA_E_ARG;
  if (dtype != LCA_F32 && dtype != LCA_BF16) return LCA_E_ARG;
  if (head_dim != 32 && head_dim != 64) return LCA_E_ARG;
  if (batch < 1 || heads < 1 || slots < 1 || n_rows < 1) return LCA_E_ARG;
  if (splits < 1 || splits > kMaxAttnSplit) return LCA_E_ARG;
  return LCA_OK;
}

int op_run(const float* q, float* out, const void* k, const void* v, int dtype, int batch, int heads,
           int head_dim, int slots, int n_rows, const int* kv_len, float scale, int splits,
           const OpScratch& o, cudaStream_t s) {
  if (cudaMemsetAsync(o.err, 0, o.header_bytes, s) != cudaSuccess) return LCA_E_CUDA;
  launch_pdl(k_regular_rows, dim3((batch + 255) / 256), dim3(256), 0, s, o.seq_start, o.seq_count, batch, n_rows);
  Rows rows{};
  rows.kvlen = const_cast<int*>(kv_len);
  rows.seq_start = o.seq_start;
  rows.seq_count = o.seq_count;
  KV kv{const_cast<void*>(k), const_cast<void*>(v), slots};
  const int qt = (n_rows + kAttnQT - 1) / kAttnQT;
  launch_any(dtype, head_dim, q, out, kv, rows, batch, heads, scale, qt < 64 ? qt : 64, splits,
             o.part, o.cnt, o.err, s);
  return cudaGetLastError() == cudaSuccess ? LCA_OK : LCA_E_CUDA;
}

// ---------------------------------------------------------------- scratch without allocation
// Scratch of lca_decode_attention_noalloc: a fixed array in device memory, shared by all calls
// on a device and held by every GPU that loads the library until the process exits.
constexpr size_t kNoAllocScratchBytes = 8u << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device, looked up once per device.
int noalloc_scratch(char** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LCA_E_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_addr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return LCA_E_CUDA;
    g_noalloc_addr[dev] = p;
  }
  *out = reinterpret_cast<char*>(g_noalloc_addr[dev]);
  return LCA_OK;
}

} // namespace

size_t attention_scratch_floats(int B, int H, int hd) {
  return (size_t)B * kQTMax * H * kMaxAttnSplit * kAttnQT * (hd + 2);
}
size_t attention_counters(int B, int H) { return (size_t)B * kQTMax * H; }

// Tensor maps (K, V) of a bf16 cache layer viewed as [rows][64]: 64-dim x 64-key boxes, 128-byte swizzle.
int make_kv_tmaps(void* out, const void* k, const void* v, long long rows) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (!encode) {
    cudaDriverEntryPointQueryResult qr;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &qr) !=
            cudaSuccess ||
        qr != cudaDriverEntryPointSuccess || !fn)
      return LCA_E_CUDA;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  const cuuint64_t dims[2] = {64, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {128};
  const cuuint32_t box[2] = {64, (cuuint32_t)kA4Keys};
  const cuuint32_t estr[2] = {1, 1};
  for (int i = 0; i < 2; ++i) {
    const CUresult r = encode(reinterpret_cast<CUtensorMap*>(static_cast<unsigned char*>(out) + 128 * i),
                              CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(i ? v : k), dims, strides, box,
                              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return LCA_E_CUDA;
  }
  return LCA_OK;
}

void kernel_attrs_attn() {
  cudaFuncSetAttribute(k_attn_mma<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)attn_mma_smem<4>());
  cudaFuncSetAttribute(k_attn_mma<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)attn_mma_smem<8>());
  cudaFuncSetAttribute(k_attn_mmt<4, mmt_warps<4>()>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)attn_mmt_smem<4>());
  cudaFuncSetAttribute(k_attn_mmt<8, mmt_warps<8>()>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)attn_mmt_smem<8>());
  cudaFuncSetAttribute(k_attn_mmt<12, mmt_warps<12>()>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)attn_mmt_smem<12>());
  cudaFuncSetAttribute(k_attn3<__nv_bfloat16, 64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaFuncSetAttribute(k_attn_w<4>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaFuncSetAttribute(k_attn_w<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       kAwStageMax * 64 * 2 * 2 + kA4MaxSplit * 4 * (64 + 2) * 4 + kMaxPtRow * 4);
  cudaFuncSetAttribute(k_attn_w<kAttnQT>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaFuncSetAttribute(k_attn_w<kAttnQT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       kAwStageMax * 64 * 2 * 2 + kA4MaxSplit * kAttnQT * (64 + 2) * 4 + kMaxPtRow * 4);
  cudaFuncSetAttribute(k_attn3<__nv_bfloat16, 32>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaFuncSetAttribute(k_attn3<float, 64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaFuncSetAttribute(k_attn3<float, 32>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaFuncSetAttribute(k_attn3<__nv_bfloat16, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)attn3_smem<__nv_bfloat16, 64>());
  cudaFuncSetAttribute(k_attn3<__nv_bfloat16, 32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)attn3_smem<__nv_bfloat16, 32>());
  cudaFuncSetAttribute(k_attn3<float, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)attn3_smem<float, 64>());
  cudaFuncSetAttribute(k_attn3<float, 32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)attn3_smem<float, 32>());
}

// The attention kernel family a launch of these arguments uses: tensor cores (prefill or decode).
static bool attn_tensor_cores(const Dev& D, const KV& kv, int B, bool short_kv) {
  return D.attn_pipe == 2 && D.dtype == LCA_BF16 && D.hd == 64 && kv.tmaps && B * D.H >= D.attn_tc_min && !short_kv;
}

bool attention_split_out(const Dev& D, const KV& kv, int B, int qtiles_grid, bool short_kv) {
  if (attn_tensor_cores(D, kv, B, short_kv)) return qtiles_grid == 1 && D.attn_t;
  return D.attn_pipe != 0;
}

void attention(const Dev& D, const float* q, float* out, const KV& kv, const Rows& rows, int B,
               int qtiles_grid, int splits, cudaStream_t s, const int* stable, bool short_kv, int stable_add,
               int rows_seq, __nv_bfloat16* osh, __nv_bfloat16* osl) {
  ProfScope ps(PK_ATTN, 0.0, s);
  if (splits < 1) splits = 1;
  if (osh && !attention_split_out(D, kv, B, qtiles_grid, short_kv)) {
    fprintf(stderr, "lca: split attention output requested from a kernel without it\n");
    osh = osl = nullptr;
  }
  const int ss = (int)(sizeof(SeqState) / sizeof(int));
  // the tensor-core kernel holds two CTAs per SM: it pays off with many (sequence, head) pairs over
  // long caches; with few pairs, or short caches (the multi-byte window), the CUDA-core pipelined
  // kernel (three CTAs per SM) runs, spreading keys over up to 16 splits
  if (attn_tensor_cores(D, kv, B, short_kv)) {
    const int sc = std::min(splits, kMaxClusterSplit);
    // decode steps (one query tile of a few rows per sequence): the transposed kernel
    if (qtiles_grid == 1 && D.attn_t) {
      if (D.attn_ns_t == 4) launch_a5_ns<4>(q, out, kv, rows, B, D.H, D.scale, 1, sc, D.err, osh, osl, s);
      else if (D.attn_ns_t == 12)
        launch_a5_ns<12>(q, out, kv, rows, B, D.H, D.scale, 1, sc, D.err, osh, osl, s);
      else launch_a5_ns<8>(q, out, kv, rows, B, D.H, D.scale, 1, sc, D.err, osh, osl, s);
    } else {
      launch_a4(D.attn_ns, q, out, kv, rows, B, D.H, D.scale, qtiles_grid, sc, D.err, s);
    }
    return;
  }
  if (D.attn_pipe) {
    splits = std::min(splits, kA4MaxSplit);
    // decode steps (one query tile per sequence) of bf16 head-dim-64 caches: the warp-walk kernel
    if (qtiles_grid == 1 && D.attn_w && D.dtype == LCA_BF16 && D.hd == 64 && kv.pt) {
      launch_aw(q, out, kv, rows, B, D.H, D.scale, splits, D.err, stable, ss, stable_add, rows_seq, osh, osl, s);
      return;
    }
    if (D.dtype == LCA_BF16) {
      if (D.hd == 64)
        launch_a3<__nv_bfloat16, 64>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, osh, osl, s);
      else
        launch_a3<__nv_bfloat16, 32>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, osh, osl, s);
    } else {
      if (D.hd == 64) launch_a3<float, 64>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, osh, osl, s);
      else launch_a3<float, 32>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, osh, osl, s);
    }
    return;
  }
  if (splits > kMaxClusterSplit) splits = kMaxClusterSplit;
  if (D.dtype == LCA_BF16) {
    if (D.hd == 64) launch_cl<__nv_bfloat16, 64>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, s);
    else launch_cl<__nv_bfloat16, 32>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, s);
  } else {
    if (D.hd == 64) launch_cl<float, 64>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, s);
    else launch_cl<float, 32>(q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.err, s);
  }
}

} // namespace lca

using namespace lca;

extern "C" {

int lca_debug_attn_diag(int32_t* out16) {
  if (!out16) return LCA_E_ARG;
  if (cudaMemcpyFromSymbol(out16, g_a4_diag, 16 * sizeof(int)) != cudaSuccess) return LCA_E_CUDA;
  const int zero[16] = {0};
  cudaMemcpyToSymbol(g_a4_diag, zero, sizeof(zero));
  return LCA_OK;
}

int lca_decode_attention_scratch_bytes(int32_t batch, int32_t heads, int32_t head_dim,
                                       int32_t splits, size_t* out) {
  if (!out || batch < 1 || heads < 1 || (head_dim != 32 && head_dim != 64) || splits < 1 ||
      splits > kMaxAttnSplit)
    return LCA_E_ARG;
  *out = op_scratch_layout(nullptr, batch, heads, head_dim, splits).bytes;
  return LCA_OK;
}

int lca_decode_attention(const float* q, float* out, const void* k_cache, const void* v_cache,
                         int32_t dtype, int32_t batch, int32_t heads, int32_t head_dim,
                         int32_t slots, int32_t n_rows, const int32_t* kv_len, float scale,
                         int32_t splits, void* scratch, size_t scratch_bytes, void* stream) {
  int st = op_check(q, out, k_cache, v_cache, dtype, batch, heads, head_dim, slots, n_rows, kv_len, splits);
  if (st != LCA_OK) return st;
  if (!scratch || reinterpret_cast<uintptr_t>(scratch) % 256) return LCA_E_ARG;
  const OpScratch o = op_scratch_layout(reinterpret_cast<char*>(scratch), batch, heads, head_dim, splits);
  if (scratch_bytes < o.bytes) return LCA_E_CAPACITY;
  return op_run(q, out, k_cache, v_cache, dtype, batch, heads, head_dim, slots, n_rows, kv_len, scale,
                splits, o, reinterpret_cast<cudaStream_t>(stream));
}

int lca_decode_attention_noalloc(const float* q, float* out, const void* k_cache, const void* v_cache,
                                 int32_t dtype, int32_t batch, int32_t heads, int32_t head_dim,
                                 int32_t slots, int32_t n_rows, const int32_t* kv_len, float scale,
                                 int32_t splits, void* stream) {
  int st = op_check(q, out, k_cache, v_cache, dtype, batch, heads, head_dim, slots, n_rows, kv_len, splits);
  if (st != LCA_OK) return st;
  if (op_scratch_layout(nullptr, batch, heads, head_dim, splits).bytes > kNoAllocScratchBytes)
    return LCA_E_CAPACITY;
  char* base = nullptr;
  st = noalloc_scratch(&base);
  if (st != LCA_OK) return st;
  const OpScratch o = op_scratch_layout(base, batch, heads, head_dim, splits);
  return op_run(q, out, k_cache, v_cache, dtype, batch, heads, head_dim, slots, n_rows, kv_len, scale,
                splits, o, reinterpret_cast<cudaStream_t>(stream));
}

size_t lca_decode_attention_noalloc_capacity(void) { return kNoAllocScratchBytes; }

}  // extern "C"

namespace {
// The status the kernels of the last call recorded in the error word (word 0 of the scratch):
// waits for the stream, then maps the bits to a status code.
int op_status(const void* word, cudaStream_t s) {
  int e = 0;
  if (cudaMemcpyAsync(&e, word, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return LCA_E_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return LCA_E_CUDA;
  if (e & kErrTimeout) return LCA_E_TIMEOUT;
  if (e & kErrIndex) return LCA_E_DEVICE_STATE;
  return LCA_OK;
}
}  // namespace

extern "C" {

int lca_decode_attention_status(const void* scratch, void* stream) {
  if (!scratch || reinterpret_cast<uintptr_t>(scratch) % 256) return LCA_E_ARG;
  return op_status(scratch, reinterpret_cast<cudaStream_t>(stream));
}

int lca_decode_attention_noalloc_status(void* stream) {
  char* base = nullptr;
  const int st = noalloc_scratch(&base);
  if (st != LCA_OK) return st;
  return op_status(base, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"

namespace lca {

LCA_TRACE_SETTER(trace_set_attn)

} // namespace lca
