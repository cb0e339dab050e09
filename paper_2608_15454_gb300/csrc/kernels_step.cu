// Per-step glue of the MBP decode step and of prefill: window planning for the multi-byte
// head, candidate embedding, space-rule segmentation with mean pooling, upsampling into the
// next-byte decoder, the unembedding heads, and the acceptance scan with commit/rollback.
#include <cuda_runtime.h>

#include "common.cuh"

namespace lca {

namespace {

__device__ __forceinline__ float ld_w(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ld_w(const __nv_bfloat16* p, size_t i) { return __bfloat162float(p[i]); }

__device__ __forceinline__ void err_or(int* e, int bits) { atomicOr(e, bits); }

// Maps a page to every page of slots [s0, s1] of sequence b that has none, from the pool's bump
// counter. One thread per sequence row of the table. A page stays mapped until the next prefill
// (a multi-byte window that restarts reuses its pages); an exhausted pool leaves the entry
// unmapped (-1) and raises kErrPages, and the writers then skip those slots. Returns the pages of
// slots s0 and s1 in *pg0 and *pg1.
__device__ void map_pages(int* pt, int ld, int pages, int* next, int b, int s0, int s1, int* err, int* pg0,
                          int* pg1) {
  if (s0 < 0) s0 = 0;
  int first = -1, last = -1;
  for (int j = s0 / kPage; j <= s1 / kPage && j < ld; ++j) {
    int* e = pt + (size_t)b * ld + j;
    int pg = *e;
    if (pg < 0) {
      pg = atomicAdd(next, 1);
      if (pg < pages) {
        *e = pg;
      } else {
        err_or(err, kErrPages);
        pg = -1;
      }
    }
    if (j == s0 / kPage) first = pg;
    last = pg;
  }
  *pg0 = first;
  *pg1 = last;
}
// Page of slot s of sequence b (after map_pages), -1 if unmapped.
__device__ __forceinline__ int page_of(const int* pt, int ld, int b, int s) {
  const int j = s / kPage;
  return (s < 0 || j >= ld) ? -1 : pt[(size_t)b * ld + j];
}

// ---------------------------------------------------------------- multi-byte window plan
// Algorithm 1, drafting: the window of sequence b is the previous and the current latent
// group, then n-2 copies of the last row. Inside the window the LCA mask is causal, and a
// row depends only on the window start and the rows before it, so rows computed in earlier
// steps stay valid while the window start is unchanged: their keys/values are kept in the
// MB cache (slot = position - window start) and only new committed rows plus the copies are
// computed. A changed window start (a committed boundary) rebuilds the cache.
__global__ void k_mb_plan(Dev D, int fill) {
  TraceScope _trace(TT_MB_PLAN);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  // the plan stays in shared memory for the rows and the fill (no global read-back)
  __shared__ int s_cnt[1024];
  __shared__ int s_first[1024];
  __shared__ int s_start[1024];
  __shared__ int s_ms[1024];
  __shared__ int s_pg0[1024], s_pg1[1024];  // pages of the first and last window row of each sequence
  __shared__ int s_K[4], s_gsK[4];  // fill (at most 4 sequences): K and the start of group K
  __shared__ int s_M;
  const Params P = *D.params;
  const int n = P.n, batch = P.batch;
  const int tid = threadIdx.x;
  for (int b = tid; b < batch; b += blockDim.x) {
    SeqState& st = D.seq[b];
    const int t = st.t, g = st.K;
    const int s = g >= 1 ? D.gstart[(size_t)b * D.L + g - 1] : 0;
    if (fill && b < 4) {
      s_K[b] = g;
      s_gsK[b] = D.gstart[(size_t)b * D.L + g];
    }
    int len = st.mb_len;
    if (st.mb_start != s) {
      st.mb_start = s;
      len = 0;
    }
    int first = s + len;
    if (first > t - 1) first = t - 1;
    s_first[b] = first;
    s_cnt[b] = (t - first) + (n - 2);
    s_ms[b] = s;
    st.mb_len = t - s;
    int pg0 = -1, pg1 = -1;
    if (s_cnt[b] > 0)
      map_pages(D.pt_mb, D.pt_ld_mb, D.pages_mb, &D.pool_next[2], b, first - s, first - s + s_cnt[b] - 1, D.err,
                &pg0, &pg1);
    s_pg0[b] = pg0;
    s_pg1[b] = pg1;
  }
  __syncthreads();
  if (tid == 0) {
    int acc = 0;
    for (int b = 0; b < batch; ++b) {
      s_start[b] = acc;
      acc += s_cnt[b];
    }
    if (acc > D.R) {
      err_or(D.err, kErrIndex);
      for (int b = 0; b < batch; ++b) {
        s_start[b] = 0;
        s_cnt[b] = 0;
      }
      acc = 0;
    }
    for (int b = 0; b < batch; ++b) {
      D.r_mb.seq_start[b] = s_start[b];
      D.r_mb.seq_count[b] = s_cnt[b];
    }
    for (int b = batch; b < D.B; ++b) {
      D.r_mb.seq_start[b] = acc;
      D.r_mb.seq_count[b] = 0;
    }
    s_M = acc;
    *D.r_mb.M = acc;
    *D.M_head_mb = batch * (n - 1);
    D.stats->mb_rows += acc;
  }
  __syncthreads();
  const int warp = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
  for (int b = warp; b < batch; b += nw) {
    const int st0 = s_start[b], cnt = s_cnt[b];
    const int s = s_ms[b], first = s_first[b];
    for (int j = lane; j < cnt; j += 32) {
      const int p = first + j;
      const int r = st0 + j;
      D.r_mb.b[r] = b;
      D.r_mb.pos[r] = p;
      D.r_mb.slot[r] = p - s;
      const int sl = p - s, f0 = (first - s) / kPage, l0 = (first - s + cnt - 1) / kPage;
      D.r_mb.page[r] = sl / kPage == f0 ? s_pg0[b] : sl / kPage == l0 ? s_pg1[b] : page_of(D.pt_mb, D.pt_ld_mb, b, sl);
      D.r_mb.kvlen[r] = p - s + 1;
    }
    for (int j = lane; j < n - 1; j += 32)
      D.head_rows_mb[b * (n - 1) + j] = cnt > 0 ? st0 + cnt - (n - 1) + j : 0;
  }
  if (!fill) return;  // many sequences: k_mb_fill writes the rows with a full grid
  // window rows: byte p of group k gets o_k + u_k (Algorithm 1, drafting input; residual r_2 added before
  // upsampling); copies beyond t belong to the current group K
  const int M = s_M;
  const int nb = batch < 4 ? batch : 4;
  const int d4 = D.d / 4;
  for (int idx = tid; idx < M * d4; idx += blockDim.x) {
    const int r = idx / d4, c4 = idx - r * d4;
    int b = 0;
    for (int bb = 1; bb < nb; ++bb)
      if (r >= s_start[bb] && s_cnt[bb] > 0) b = bb;
    const int p = s_first[b] + (r - s_start[b]);
    const int g = s_K[b];
    const int k = (g >= 1 && p < s_gsK[b]) ? g - 1 : g;
    const float4 o = reinterpret_cast<const float4*>(D.o_tab + ((size_t)b * D.L + k) * D.d)[c4];
    const float4 u = reinterpret_cast<const float4*>(D.u_tab + ((size_t)b * D.L + k) * D.d)[c4];
    reinterpret_cast<float4*>(D.x_mb + (size_t)r * D.d)[c4] = make_float4(o.x + u.x, o.y + u.y, o.z + u.z, o.w + u.w);
  }
}

// MB input rows: byte p of group k gets o_k + u_k (Algorithm 1, drafting input; residual r_2 added
// before upsampling); copies beyond t belong to the current group K.
__global__ void k_mb_fill(Dev D) {
  TraceScope _trace(TT_MB_FILL);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const int M = *D.r_mb.M;
  const int d4 = D.d / 4;
  for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < (size_t)M * d4;
       idx += (size_t)gridDim.x * blockDim.x) {
    const int r = (int)(idx / d4), c = (int)(idx - (size_t)r * d4) * 4;
    const int b = D.r_mb.b[r], p = D.r_mb.pos[r];
    const SeqState& st = D.seq[b];
    const int g = st.K;
    const int gs = D.gstart[(size_t)b * D.L + g];
    const int k = (g >= 1 && p < gs) ? g - 1 : g;
    const float4 o = *reinterpret_cast<const float4*>(D.o_tab + ((size_t)b * D.L + k) * D.d + c);
    const float4 u = *reinterpret_cast<const float4*>(D.u_tab + ((size_t)b * D.L + k) * D.d + c);
    *reinterpret_cast<float4*>(D.x_mb + (size_t)r * D.d + c) =
        make_float4(o.x + u.x, o.y + u.y, o.z + u.z, o.w + u.w);
  }
}

// MLP-MBP heads: row j*batch + b starts from the last next-byte hidden state of b.
__global__ void k_mlp_plan(Dev D) {
  TraceScope _trace(TT_MLP_PLAN);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const Params P = *D.params;
  const int n = P.n, batch = P.batch;
  const int rows = batch * (n - 1);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    *D.r_mb.M = batch;  // rows per head (grouped linear)
    *D.M_head_mb = rows;
  }
  for (int q = blockIdx.x; q < rows; q += gridDim.x) {
    const int j = q / batch, b = q - j * batch;
    const int r = j * D.B + b;  // head j owns rows [j*B, j*B + batch)
    for (int c = threadIdx.x; c < D.d; c += blockDim.x)
      D.x_mb[(size_t)r * D.d + c] = D.y_last[(size_t)b * D.d + c];
    if (threadIdx.x == 0) D.head_rows_mb[b * (n - 1) + j] = r;
  }
}

// ---------------------------------------------------------------- unembedding heads
// Final RMSNorm of the head, shared unembedding (Section 3), then per row the argmax (lowest
// byte among equal maxima) and its softmax probability exp(l_max - logsumexp(l)).
constexpr int kHR = 8;   // rows per CTA
constexpr int kHV = 8;   // vocab entries per CTA (one per warp)

__device__ __forceinline__ uint4 ldg_nc16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}
__device__ __forceinline__ void unpack8w(const uint4* u, float* w, const __nv_bfloat16*) {
  w[0] = __uint_as_float(u[0].x << 16); w[1] = __uint_as_float(u[0].x & 0xFFFF0000u);
  w[2] = __uint_as_float(u[0].y << 16); w[3] = __uint_as_float(u[0].y & 0xFFFF0000u);
  w[4] = __uint_as_float(u[0].z << 16); w[5] = __uint_as_float(u[0].z & 0xFFFF0000u);
  w[6] = __uint_as_float(u[0].w << 16); w[7] = __uint_as_float(u[0].w & 0xFFFF0000u);
}
__device__ __forceinline__ void unpack8w(const uint4* u, float* w, const float*) {
  w[0] = __uint_as_float(u[0].x); w[1] = __uint_as_float(u[0].y);
  w[2] = __uint_as_float(u[0].z); w[3] = __uint_as_float(u[0].w);
  w[4] = __uint_as_float(u[1].x); w[5] = __uint_as_float(u[1].y);
  w[6] = __uint_as_float(u[1].z); w[7] = __uint_as_float(u[1].w);
}

// One CTA: kHR rows x kHV vocab entries; warp w owns vocab row blockIdx.y*kHV + w, whose
// weights are loaded into registers before the grid-dependency wait. The last CTA of a row
// tile reduces the 256 logits of each row to (argmax, probability).
template <typename TW, int HCH>
__global__ void __launch_bounds__(256)
k_head(Dev D, const float* __restrict__ x, const int* __restrict__ rows, const int* Mp, int M_cap,
       const float* __restrict__ norm, float* __restrict__ logits, int* __restrict__ arg,
       float* __restrict__ prob, int* __restrict__ cnt) {
  TraceScope _trace(TT_HEAD);
  constexpr int VEC = sizeof(TW) == 2 ? 1 : 2;
  extern __shared__ float xs[];  // [kHR][d]
  __shared__ int s_last;
  const int d = D.d;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int v = blockIdx.y * kHV + warp;
  const TW* Wu = reinterpret_cast<const TW*>(D.unembed) + (size_t)v * d;
  uint4 wr[HCH][VEC];
#pragma unroll
  for (int c = 0; c < HCH; ++c) {
    const int k = lane * 8 + c * 256;
    if (k < d) {
#pragma unroll
      for (int e = 0; e < VEC; ++e) wr[c][e] = ldg_nc16(reinterpret_cast<const uint4*>(Wu + k) + e);
    }
  }
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  int M = *Mp;
  M = M < M_cap ? M : M_cap;
  const int rt = blockIdx.x;
  const int r0 = rt * kHR;
  if (r0 >= M) return;
  const int mr = min(kHR, M - r0);
  // warp w stages row w (raw, loads batched), computes its inverse RMS, then scales in place
  if (warp < kHR) {
    const int i = warp;
    float ss = 0.f;
    constexpr int NQ = HCH * 2;  // float4 per lane (d <= HCH * 256)
    float4 q[NQ];
    const int src = i < mr ? (rows ? rows[r0 + i] : r0 + i) : 0;
#pragma unroll
    for (int u = 0; u < NQ; ++u) {
      const int k = (lane + u * 32) * 4;
      q[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (i < mr && k < d) q[u] = *reinterpret_cast<const float4*>(x + (size_t)src * d + k);
      ss += q[u].x * q[u].x + q[u].y * q[u].y + q[u].z * q[u].z + q[u].w * q[u].w;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    const float sc = rsqrtf(ss / (float)d + D.eps);
#pragma unroll
    for (int u = 0; u < NQ; ++u) {
      const int k = (lane + u * 32) * 4;
      if (k < d) {
        const float4 g = *reinterpret_cast<const float4*>(norm + k);
        float4 v = q[u];
        v.x *= sc * g.x; v.y *= sc * g.y; v.z *= sc * g.z; v.w *= sc * g.w;
        *reinterpret_cast<float4*>(xs + i * d + k) = v;
      }
    }
  }
  __syncthreads();
  float acc[kHR];
#pragma unroll
  for (int i = 0; i < kHR; ++i) acc[i] = 0.f;
#pragma unroll
  for (int c = 0; c < HCH; ++c) {
    const int k = lane * 8 + c * 256;
    if (k < d) {
      float w[8];
      unpack8w(wr[c], w, (const TW*)nullptr);
#pragma unroll
      for (int i = 0; i < kHR; ++i) {
        const float4 xa = *reinterpret_cast<const float4*>(xs + i * d + k);
        const float4 xb = *reinterpret_cast<const float4*>(xs + i * d + k + 4);
        float sacc = acc[i];
        sacc = fmaf(w[0], xa.x, sacc); sacc = fmaf(w[1], xa.y, sacc);
        sacc = fmaf(w[2], xa.z, sacc); sacc = fmaf(w[3], xa.w, sacc);
        sacc = fmaf(w[4], xb.x, sacc); sacc = fmaf(w[5], xb.y, sacc);
        sacc = fmaf(w[6], xb.z, sacc); sacc = fmaf(w[7], xb.w, sacc);
        acc[i] = sacc;
      }
    }
  }
#pragma unroll
  for (int i = 0; i < kHR; ++i) {
    float sacc = acc[i];
#pragma unroll
    for (int o = 16; o; o >>= 1) sacc += __shfl_xor_sync(0xffffffffu, sacc, o);
    if (lane == 0 && i < mr) logits[(size_t)(r0 + i) * kVocab + v] = sacc;
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(cnt + rt, 1) == (int)gridDim.y - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (warp < mr) {
    const int i = warp;
    const float* lg = logits + (size_t)(r0 + i) * kVocab;
    float best = -INFINITY;
    int bi = kVocab;
    bool bad = false;
    float lv[kVocab / 32];
#pragma unroll
    for (int j = 0; j < kVocab / 32; ++j) {
      const int vv = lane + 32 * j;
      const float l = __ldcg(lg + vv);
      lv[j] = l;
      if (!isfinite(l)) bad = true;
      if (l > best || (l == best && vv < bi)) {
        best = l;
        bi = vv;
      }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float ob = __shfl_xor_sync(0xffffffffu, best, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ob > best || (ob == best && oi < bi)) {
        best = ob;
        bi = oi;
      }
    }
    bad = __any_sync(0xffffffffu, bad);
    float se = 0.f;
#pragma unroll
    for (int j = 0; j < kVocab / 32; ++j) se += expf(lv[j] - best);
#pragma unroll
    for (int o = 16; o; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
    if (lane == 0) {
      if (bad) {
        err_or(D.err, kErrNumeric);
        bi = 0;
      }
      arg[r0 + i] = bi;
      prob[r0 + i] = bad ? 0.f : 1.f / se;
    }
  }
  if (tid == 0) cnt[rt] = 0;
}

// ---------------------------------------------------------------- verify rows
// Candidates c_1 (next-byte argmax) and d_2..d_n (drafts) at positions t..t+n-1; embed them.
__global__ void k_verify_plan(Dev D) {
  TraceScope _trace(TT_VERIFY_PLAN);
  __shared__ int s_c[64];
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const Params P = *D.params;
  const int n = P.n, batch = P.batch;
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  if (b >= batch) {
    if (tid == 0) {
      D.r_v.seq_start[b] = batch * n;
      D.r_v.seq_count[b] = 0;
    }
    return;
  }
  // pages of positions t..t+n-1 (one thread maps them: at most two pages for n <= 64)
  __shared__ int s_pg[2];
  if (tid == 0) {
    const int t = D.seq[b].t;
    map_pages(D.pt_byte, D.pt_ld_byte, D.pages_byte, &D.pool_next[0], b, t, min(t + n - 1, D.S - 1), D.err,
              &s_pg[0], &s_pg[1]);
  }
  __syncthreads();
  if (tid < n) {
    const int i = tid;
    const int t = D.seq[b].t;
    int c;
    if (P.force_cand) c = D.forced_cand[b * D.NMAX + i];
    else c = i == 0 ? D.seq[b].next_c1 : D.mb_arg[b * (n - 1) + i - 1];
    c &= 255;
    s_c[i] = c;
    D.cand[b * D.NMAX + i] = c;
    const int r = b * n + i;
    int p = t + i;
    if (p >= D.S) {
      err_or(D.err, kErrIndex);
      p = D.S - 1;
    }
    D.r_v.b[r] = b;
    D.r_v.pos[r] = p;
    D.r_v.slot[r] = p;
    D.r_v.page[r] = p / kPage == t / kPage ? s_pg[0] : s_pg[1];
    D.r_v.kvlen[r] = p + 1;
  }
  if (tid == 0) {
    D.r_v.seq_start[b] = b * n;
    D.r_v.seq_count[b] = n;
    if (b == 0) *D.r_v.M = batch * n;
  }
  __syncthreads();
  // embedding rows of the candidates, 16-byte vectors, loads issued before the stores
  const int ev = D.dtype == LCA_BF16 ? 8 : 4;  // elements per 16-byte vector
  const int per_row = D.d / ev;
  const int total = n * per_row;
  constexpr int UNR = 4;
  for (int base = tid; base < total; base += blockDim.x * UNR) {
    uint4 u[UNR];
#pragma unroll
    for (int k = 0; k < UNR; ++k) {
      const int idx = base + k * blockDim.x;
      if (idx < total) {
        const int i = idx / per_row, j = idx - i * per_row;
        const char* row = reinterpret_cast<const char*>(D.embed) + (size_t)s_c[i] * D.d * (ev == 8 ? 2 : 4);
        u[k] = *reinterpret_cast<const uint4*>(row + (size_t)j * 16);
      }
    }
#pragma unroll
    for (int k = 0; k < UNR; ++k) {
      const int idx = base + k * blockDim.x;
      if (idx < total) {
        const int i = idx / per_row, j = idx - i * per_row;
        float* dst = D.x_enc + (size_t)(b * n + i) * D.d + (size_t)j * ev;
        if (ev == 8) {
          float f[8];
          unpack8w(&u[k], f, (const __nv_bfloat16*)nullptr);
          reinterpret_cast<float4*>(dst)[0] = make_float4(f[0], f[1], f[2], f[3]);
          reinterpret_cast<float4*>(dst)[1] = make_float4(f[4], f[5], f[6], f[7]);
        } else {
          reinterpret_cast<float4*>(dst)[0] = make_float4(__uint_as_float(u[k].x), __uint_as_float(u[k].y),
                                                          __uint_as_float(u[k].z), __uint_as_float(u[k].w));
        }
      }
    }
  }
}

// ---------------------------------------------------------------- segments and latents
// Space rule (b_p = [x_p == 0x20], the boundary byte ends its segment). Every boundary among
// the candidates closes a segment: z = mean of the encoder output over the segment (committed
// bytes from h_store, candidate rows from x_enc), which becomes the LM input of latent K+j.
// K(p) of candidate row i counts boundaries at positions <= p. New latents of all sequences
// are compacted into LM rows; the LM module runs (graph conditional) only if there are any.
__global__ void k_segment(Dev D, cudaGraphConditionalHandle hcond, int use_handle) {
  TraceScope _trace(TT_SEGMENT);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const Params P = *D.params;
  const int n = P.n, batch = P.batch;
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  __shared__ int s_c[64];
  __shared__ int s_sp[64];
  __shared__ int s_nsp;
  __shared__ SeqState s_st;
  if (b >= batch) {
    if (tid == 0) {
      D.r_lm.seq_start[b] = 0;
      D.r_lm.seq_count[b] = 0;
    }
    return;
  }
  // boundaries among the candidates of earlier sequences (compaction offset) and of all
  int off = 0, total = 0;
  for (int base = 0; base < batch * n; base += blockDim.x) {
    const int idx = base + tid;
    const int bb = idx / n, i = idx - bb * n;
    const bool sp = idx < batch * n && D.cand[bb * D.NMAX + i] == D.boundary;
    off += __syncthreads_count(sp && bb < b);
    if (b == 0) total += __syncthreads_count(sp);
  }
  if (tid < n) s_c[tid] = D.cand[b * D.NMAX + tid];
  if (tid == 0) s_st = D.seq[b];
  __syncthreads();
  if (tid == 0) {
    int m = 0;
    for (int i = 0; i < n; ++i)
      if (s_c[i] == D.boundary) s_sp[m++] = i;
    s_nsp = m;
    D.r_lm.seq_start[b] = off;
    D.r_lm.seq_count[b] = m;
    if (b == 0) {
      *D.r_lm.M = total;
      if (use_handle) cudaGraphSetConditional(hcond, total > 0 ? 1u : 0u);
      D.step_log[D.stats->steps % kStepLog] = total > 0 ? 1 : 0;
      D.stats->steps += 1;
      D.stats->lm_steps += total > 0;
      D.stats->lm_rows += total;
    }
  }
  const int t = s_st.t, K = s_st.K;
  if (tid < n) {
    int k = K;
    for (int i = 0; i <= tid; ++i) k += s_c[i] == D.boundary;
    D.kc[b * D.NMAX + tid] = k;
  }
  __syncthreads();
  const int m = s_nsp;
  const int d4 = D.d / 4;
  for (int j = 0; j < m; ++j) {
    const int i = s_sp[j];
    const int k = K + 1 + j;
    const int seg0 = j == 0 ? s_st.open_start : t + s_sp[j - 1] + 1;
    const int seg1 = t + i;  // inclusive
    const int row = off + j;
    if (k >= D.L) {
      if (tid == 0) err_or(D.err, kErrIndex);
      continue;
    }
    const float inv_cnt = 1.f / (float)(seg1 - seg0 + 1);
    for (int c4 = tid; c4 < d4; c4 += blockDim.x) {
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      int p = seg0;
      // four positions per round, loads issued together
      for (; p + 3 <= seg1; p += 4) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int q = p + u;
          v[u] = q < t ? reinterpret_cast<const float4*>(D.h_store + ((size_t)b * D.S + q) * D.d)[c4]
                       : reinterpret_cast<const float4*>(D.x_enc + (size_t)(b * n + q - t) * D.d)[c4];
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          acc.x += v[u].x; acc.y += v[u].y; acc.z += v[u].z; acc.w += v[u].w;
        }
      }
      for (; p <= seg1; ++p) {
        const float4 v = p < t ? reinterpret_cast<const float4*>(D.h_store + ((size_t)b * D.S + p) * D.d)[c4]
                               : reinterpret_cast<const float4*>(D.x_enc + (size_t)(b * n + p - t) * D.d)[c4];
        acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
      }
      const float4 z = make_float4(acc.x * inv_cnt, acc.y * inv_cnt, acc.z * inv_cnt, acc.w * inv_cnt);
      reinterpret_cast<float4*>(D.x_lm + (size_t)row * D.d)[c4] = z;
      reinterpret_cast<float4*>(D.u_tab + ((size_t)b * D.L + k) * D.d)[c4] = z;
    }
    if (tid == 0) {
      D.gstart[(size_t)b * D.L + k] = seg1;
      int pg, pg1;
      map_pages(D.pt_lm, D.pt_ld_lm, D.pages_lm, &D.pool_next[1], b, k, k, D.err, &pg, &pg1);
      D.r_lm.b[row] = b;
      D.r_lm.pos[row] = k;
      D.r_lm.slot[row] = k;
      D.r_lm.page[row] = pg;
      D.r_lm.kvlen[row] = k + 1;
    }
  }
}

// o_k of the latents the LM module just produced.
__global__ void k_lm_scatter(Dev D) {
  TraceScope _trace(TT_LM_SCATTER);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const int M = *D.r_lm.M;
  for (int r = blockIdx.x; r < M; r += gridDim.x) {
    const int b = D.r_lm.b[r], k = D.r_lm.pos[r];
    for (int c = threadIdx.x; c < D.d; c += blockDim.x)
      D.o_tab[((size_t)b * D.L + k) * D.d + c] = D.x_lm[(size_t)r * D.d + c];
  }
}

// Next-byte decoder input: upsampled LM output plus the encoder residual r_1 (Algorithm 1,
// next-byte step): o_{K(p)} + h_e[p].
__global__ void k_nb_input(Dev D) {
  TraceScope _trace(TT_NB_INPUT);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const Params P = *D.params;
  const int n = P.n, batch = P.batch;
  const int rows = batch * n;
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    const int b = r / n, i = r - b * n;
    const int k = D.kc[b * D.NMAX + i];
    const float* o = D.o_tab + ((size_t)b * D.L + k) * D.d;
    for (int c = threadIdx.x; c < D.d; c += blockDim.x)
      D.x_nb[(size_t)r * D.d + c] = o[c] + D.x_enc[(size_t)r * D.d + c];
  }
}

// ---------------------------------------------------------------- accept and commit
// Section 3.1 "Byte Acceptance": c_1 is always kept; drafts are kept left to right while the
// drafter's probability is >= tau (THRESH) or while they equal the next-byte argmax at the
// position before them (SPEC); the first failure drops the rest. The accepted prefix of every
// cache is kept by advancing t and K; everything beyond is dropped (overwritten later).
__global__ void k_commit(Dev D) {
  TraceScope _trace(TT_COMMIT);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  const Params P = *D.params;
  const int n = P.n, batch = P.batch;
  const int b = blockIdx.x;
  if (b >= batch) return;
  const int tid = threadIdx.x;
  __shared__ int s_c[64], s_kc[64], s_nb[64];
  __shared__ SeqState s_st;
  __shared__ int s_e, s_a, s_last_sp;
  if (tid < n) {
    s_c[tid] = D.cand[b * D.NMAX + tid];
    s_kc[tid] = D.kc[b * D.NMAX + tid];
    s_nb[tid] = D.nb_arg[b * n + tid];
  }
  if (tid == 0) s_st = D.seq[b];
  __syncthreads();
  if (tid < 32) {
    // Acceptance scan, one warp per sequence (n <= 16 <= 32 lanes): lane i holds the flag of draft
    // d_{i+2}: its drafter probability >= tau (threshold acceptance, Section 3.1) or its equality with
    // the next-byte argmax of the row before it (greedy speculative acceptance, Section 6.2). The
    // accepted drafts are the leading run of set flags: the index of the first clear bit of the
    // ballot (lanes >= n-1 vote 0, so a clear bit exists).
    const int lane = tid;
    bool ok = false;
    if (lane < n - 1)
      ok = P.accept == LCA_SPEC ? s_c[lane + 1] == s_nb[lane] : D.mb_prob[b * (n - 1) + lane] >= P.tau;
    const unsigned vote = __ballot_sync(0xffffffffu, ok);
    int a = __ffs(~vote) - 1;
    int e = 0;
    if (!(P.gen && s_st.done)) {
      if (P.force_accept) {
        a = D.forced_a[b];
        a = a < 0 ? 0 : (a > n - 1 ? n - 1 : a);
      }
      e = 1 + a;
      if (P.gen) {
        const int rem = s_st.budget - s_st.generated;
        e = e < rem ? e : rem;
      }
    } else {
      a = 0;
    }
    // the last committed boundary byte (it starts the new open segment)
    const unsigned sp = __ballot_sync(0xffffffffu, lane < e && s_c[lane] == D.boundary);
    if (lane == 0) {
      s_e = e;
      s_a = a;
      s_last_sp = sp ? 31 - __clz((int)sp) : -1;
    }
  }
  __syncthreads();
  const int e = s_e, t = s_st.t;
  if (e == 0) {
    if (tid == 0) D.out_cnt[b] = 0;
    return;
  }
  // encoder outputs of the committed candidates join the pooled history; the last next-byte
  // hidden state feeds the MLP heads (float4 copies, loads before stores)
  const int d4 = D.d / 4;
  const int tot = e * d4 + d4;
  for (int base = tid; base < tot; base += blockDim.x * 4) {
    float4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx < e * d4) {
        const int i = idx / d4, c4 = idx - i * d4;
        v[u] = reinterpret_cast<const float4*>(D.x_enc + (size_t)(b * n + i) * D.d)[c4];
      } else if (idx < tot) {
        v[u] = reinterpret_cast<const float4*>(D.x_nb + (size_t)(b * n + e - 1) * D.d)[idx - e * d4];
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx < e * d4) {
        const int i = idx / d4, c4 = idx - i * d4;
        reinterpret_cast<float4*>(D.h_store + ((size_t)b * D.S + t + i) * D.d)[c4] = v[u];
      } else if (idx < tot) {
        reinterpret_cast<float4*>(D.y_last + (size_t)b * D.d)[idx - e * d4] = v[u];
      }
    }
  }
  if (tid < n) {
    const int i = tid;
    D.out_step[b * D.NMAX + i] = (uint8_t)(i < e ? s_c[i] : 0);
    if (P.gen && i < e && s_st.generated + i < D.S) D.out_gen[(size_t)b * D.S + s_st.generated + i] = (uint8_t)s_c[i];
  }
  if (tid == 0) {
    const int last_sp = s_last_sp;
    SeqState& st = D.seq[b];
    D.out_cnt[b] = e;
    st.t = t + e;
    st.K = s_kc[e - 1];
    if (last_sp >= 0) st.open_start = t + last_sp + 1;
    st.next_c1 = s_nb[e - 1];
    st.generated = s_st.generated + e;
    if (P.gen && st.generated >= s_st.budget) st.done = 1;
    atomicAdd(D.hist + s_a, 1);
    atomicAdd(&D.stats->committed, (unsigned long long)e);
  }
}

// Generate loop control: keep looping while a sequence is short of its budget (and never more
// than max_iter steps, each of which commits at least one byte per unfinished sequence).
__global__ void k_loop_ctl(Dev D, cudaGraphConditionalHandle h) {
  TraceScope _trace(TT_LOOP_CTL);
  pdl_trigger();
  pdl_wait();
  _trace.waited();
  if (threadIdx.x != 0) return;
  Params* P = D.params;
  const int it = P->iter + 1;
  P->iter = it;
  int any = 0;
  for (int b = 0; b < P->batch; ++b) any |= (D.seq[b].active && !D.seq[b].done);
  cudaGraphSetConditional(h, (any && it < P->max_iter) ? 1u : 0u);
}

__global__ void k_gen_init(Dev D, int max_new) {
  pdl_trigger();
  pdl_wait();
  const int b = threadIdx.x;
  if (b < D.B) {
    SeqState& st = D.seq[b];
    st.generated = 0;
    st.budget = max_new;
    st.done = st.active ? 0 : 1;
  }
  if (b < D.NMAX) D.hist[b] = 0;
  if (b == 0) D.params->iter = 0;
}

// cos/sin of RoPE angles pos * base^(-2i/hd), computed in double.
__global__ void k_rope_table(float2* tab, int slots, int hd, double base) {
  const int half = hd / 2;
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < slots * half;
       idx += gridDim.x * blockDim.x) {
    const int p = idx / half, i = idx - p * half;
    const double ang = (double)p * pow(base, -2.0 * i / hd);
    tab[idx] = make_float2((float)cos(ang), (float)sin(ang));
  }
}

// ---------------------------------------------------------------- prefill
__global__ void k_prefill_embed(Dev D, const uint8_t* __restrict__ bytes, int M) {
  pdl_trigger();
  pdl_wait();
  for (size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x; idx < (size_t)M * D.d;
       idx += (size_t)gridDim.x * blockDim.x) {
    const int r = (int)(idx / D.d), k = (int)(idx - (size_t)r * D.d);
    const int c = bytes[r];
    D.x_enc[idx] = D.dtype == LCA_BF16
                       ? ld_w(reinterpret_cast<const __nv_bfloat16*>(D.embed), (size_t)c * D.d + k)
                       : ld_w(reinterpret_cast<const float*>(D.embed), (size_t)c * D.d + k);
  }
}

// One CTA per sequence: K(p) for every prompt byte and the group starts.
__global__ void k_prefill_segment(Dev D, const uint8_t* __restrict__ bytes, const int* row0,
                                  const int* lens) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  __shared__ int s_scan[1024];
  __shared__ int s_carry;
  const int len = lens[b];
  const uint8_t* x = bytes + row0[b];
  if (tid == 0) {
    s_carry = 0;
    D.gstart[(size_t)b * D.L] = 0;
  }
  __syncthreads();
  for (int base = 0; base < len; base += blockDim.x) {
    const int p = base + tid;
    const int isb = (p < len && x[p] == D.boundary) ? 1 : 0;
    s_scan[tid] = isb;
    __syncthreads();
    for (int o = 1; o < (int)blockDim.x; o <<= 1) {
      const int v = tid >= o ? s_scan[tid - o] : 0;
      __syncthreads();
      s_scan[tid] += v;
      __syncthreads();
    }
    const int k = s_carry + s_scan[tid];
    if (p < len) {
      D.kpos[(size_t)b * D.S + p] = k;
      if (isb) {
        if (k < D.L) D.gstart[(size_t)b * D.L + k] = p;
        else err_or(D.err, kErrIndex);
      }
    }
    __syncthreads();
    if (tid == blockDim.x - 1) s_carry = k;
    __syncthreads();
  }
  if (tid == 0) {
    const int K = s_carry;
    D.seq[b].K = K;
    D.seq[b].open_start = K > 0 ? D.gstart[(size_t)b * D.L + K] + 1 : 0;
  }
}

// CTA (b, k): latent k of sequence b: BOS for k = 0, else the mean of segment k.
__global__ void k_prefill_pool(Dev D, const int* row0, const int* lm_row0) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int k = blockIdx.y;
  const int K = D.seq[b].K;
  if (k > K) return;
  const int row = lm_row0[b] + k;
  if (k == 0) {
    for (int c = threadIdx.x; c < D.d; c += blockDim.x) {
      D.x_lm[(size_t)row * D.d + c] = D.bos[c];
      D.u_tab[((size_t)b * D.L) * D.d + c] = D.bos[c];
    }
    return;
  }
  const int seg1 = D.gstart[(size_t)b * D.L + k];
  const int seg0 = k == 1 ? 0 : D.gstart[(size_t)b * D.L + k - 1] + 1;
  const float inv_cnt = 1.f / (float)(seg1 - seg0 + 1);
  for (int c = threadIdx.x; c < D.d; c += blockDim.x) {
    float s = 0.f;
    for (int p = seg0; p <= seg1; ++p) s += D.x_enc[(size_t)(row0[b] + p) * D.d + c];
    const float z = s * inv_cnt;
    D.x_lm[(size_t)row * D.d + c] = z;
    D.u_tab[((size_t)b * D.L + k) * D.d + c] = z;
  }
}

__global__ void k_prefill_nb_input(Dev D, int M) {
  pdl_trigger();
  pdl_wait();
  for (int r = blockIdx.x; r < M; r += gridDim.x) {
    const int b = D.r_v.b[r], p = D.r_v.pos[r];
    const int k = D.kpos[(size_t)b * D.S + p];
    const float* o = D.o_tab + ((size_t)b * D.L + k) * D.d;
    for (int c = threadIdx.x; c < D.d; c += blockDim.x) {
      const float h = D.x_enc[(size_t)r * D.d + c];
      D.h_store[((size_t)b * D.S + p) * D.d + c] = h;
      D.x_nb[(size_t)r * D.d + c] = o[c] + h;
    }
  }
}

__global__ void k_prefill_finish(Dev D, const int* row0, const int* lens) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int last = row0[b] + lens[b] - 1;
  for (int c = threadIdx.x; c < D.d; c += blockDim.x)
    D.y_last[(size_t)b * D.d + c] = D.x_nb[(size_t)last * D.d + c];
  if (threadIdx.x == 0) {
    SeqState& st = D.seq[b];
    st.t = lens[b];
    st.mb_start = -1;
    st.mb_len = 0;
    st.next_c1 = D.nb_arg[b];
    st.generated = 0;
    st.budget = 0x3fffffff;
    st.done = 0;
    st.active = 1;
  }
}

// Repack rows: dst[(dst_row0 + i*row_step)] = src[i] for i < rows (row = cols elements).
__global__ void k_pack_rows(uint8_t* dst, const uint8_t* src, int rows, size_t row_bytes,
                            int dst_row0, int row_step) {
  for (int i = blockIdx.x; i < rows; i += gridDim.x) {
    const uint8_t* s = src + (size_t)i * row_bytes;
    uint8_t* d = dst + (size_t)(dst_row0 + (size_t)i * row_step) * row_bytes;
    for (size_t c = threadIdx.x * 16; c < row_bytes; c += blockDim.x * 16)
      *reinterpret_cast<uint4*>(d + c) = *reinterpret_cast<const uint4*>(s + c);
  }
}

} // namespace

// ---------------------------------------------------------------- launch wrappers
template <typename TW>
void head_attrs() {
  cudaFuncSetAttribute(k_head<TW, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
  cudaFuncSetAttribute(k_head<TW, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
  cudaFuncSetAttribute(k_head<TW, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
  cudaFuncSetAttribute(k_head<TW, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
}

void kernel_attrs_step() {
  head_attrs<__nv_bfloat16>();
  head_attrs<float>();
}

thread_local long long g_launches = 0;
thread_local ProfHook* g_prof = nullptr;

// One CTA plans the windows; with few sequences it also writes the window rows (one launch less
// on the latency-bound path), with many the rows are written by k_mb_fill over the whole GPU.
void launch_mb_fill(const Dev& D, cudaStream_t s);
void launch_mb_plan(const Dev& D, cudaStream_t s) {
  const int fill = D.B <= 4;
  {
    ++g_launches;
    ProfScope ps(PK_GLUE, 0.0, s);
    launch_pdl(k_mb_plan, dim3(1), dim3(1024), 0, s, D, fill);
  }
  if (!fill) launch_mb_fill(D, s);
}
void launch_mb_fill(const Dev& D, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_mb_fill, dim3(D.num_sms * 2), dim3(256), 0, s, D);
}
void launch_mlp_plan(const Dev& D, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_mlp_plan, dim3(256), dim3(256), 0, s, D);
}

template <typename TW, int HCH>
void head_launch(const Dev& D, const float* x, const int* rows, const int* M, int M_cap,
                 const float* norm, float* logits, int* arg, float* prob, cudaStream_t s) {
  dim3 grid((M_cap + kHR - 1) / kHR, kVocab / kHV);
  const size_t smem = (size_t)kHR * D.d * sizeof(float);
  launch_pdl(k_head<TW, HCH>, grid, dim3(256), smem, s, D, x, rows, M, M_cap, norm, logits, arg,
             prob, D.head_cnt);
}

template <typename TW>
void head_dispatch(const Dev& D, const float* x, const int* rows, const int* M, int M_cap,
                   const float* norm, float* logits, int* arg, float* prob, cudaStream_t s) {
  if (D.d <= 256) head_launch<TW, 1>(D, x, rows, M, M_cap, norm, logits, arg, prob, s);
  else if (D.d <= 512) head_launch<TW, 2>(D, x, rows, M, M_cap, norm, logits, arg, prob, s);
  else if (D.d <= 1024) head_launch<TW, 4>(D, x, rows, M, M_cap, norm, logits, arg, prob, s);
  else head_launch<TW, 8>(D, x, rows, M, M_cap, norm, logits, arg, prob, s);
}

void launch_head(const Dev& D, const float* x, const int* rows, const int* M, int M_cap,
                 const float* norm, float* logits, int* arg, float* prob, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_HEAD, 256.0 * D.d * (D.dtype == LCA_BF16 ? 2 : 4), s);
  if (D.dtype == LCA_BF16) head_dispatch<__nv_bfloat16>(D, x, rows, M, M_cap, norm, logits, arg, prob, s);
  else head_dispatch<float>(D, x, rows, M, M_cap, norm, logits, arg, prob, s);
}

void launch_verify_plan(const Dev& D, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_verify_plan, dim3(D.B), dim3(256), 0, s, D);
}
void launch_segment(const Dev& D, cudaGraphConditionalHandle h, int use_handle, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_segment, dim3(D.B), dim3(256), 0, s, D, h, use_handle);
}
void launch_lm_scatter(const Dev& D, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_lm_scatter, dim3(256), dim3(256), 0, s, D);
}
void launch_nb_input(const Dev& D, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_nb_input, dim3(256), dim3(256), 0, s, D);
}
void launch_commit(const Dev& D, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_commit, dim3(D.B), dim3(256), 0, s, D);
}
void launch_loop_ctl(const Dev& D, cudaGraphConditionalHandle h, cudaStream_t s) {
  ++g_launches;
  ProfScope ps(PK_GLUE, 0.0, s);
  launch_pdl(k_loop_ctl, dim3(1), dim3(32), 0, s, D, h);
}
void launch_gen_init(const Dev& D, int max_new, cudaStream_t s) {
  launch_pdl(k_gen_init, dim3(1), dim3(1024), 0, s, D, max_new);
}
void launch_rope_table(const Dev& D, float base, cudaStream_t s) {
  k_rope_table<<<256, 256, 0, s>>>(D.rope, D.rope_slots, D.hd, (double)base);
}
void launch_pack_rows(void* dst, const void* src, int rows, int cols, int dst_row0, int row_step,
                      int elem_bytes, cudaStream_t s) {
  k_pack_rows<<<256, 128, 0, s>>>((uint8_t*)dst, (const uint8_t*)src, rows,
                                  (size_t)cols * elem_bytes, dst_row0, row_step);
}
void launch_prefill_embed(const Dev& D, const uint8_t* bytes, int M, cudaStream_t s) {
  launch_pdl(k_prefill_embed, dim3(1024), dim3(256), 0, s, D, bytes, M);
}
void launch_prefill_segment(const Dev& D, const uint8_t* bytes, const int* row0, const int* lens,
                            int batch, const int* lm_row0, cudaStream_t s) {
  (void)lm_row0;
  launch_pdl(k_prefill_segment, dim3(batch), dim3(1024), 0, s, D, bytes, row0, lens);
}
void launch_prefill_pool(const Dev& D, const int* row0, const int* lens, const int* lm_row0,
                         int batch, int max_lat, cudaStream_t s) {
  (void)lens;
  launch_pdl(k_prefill_pool, dim3(batch, max_lat + 1), dim3(256), 0, s, D, row0, lm_row0);
}
void launch_prefill_nb_input(const Dev& D, int M, cudaStream_t s) {
  launch_pdl(k_prefill_nb_input, dim3(1024), dim3(256), 0, s, D, M);
}
void launch_prefill_finish(const Dev& D, const int* row0, const int* lens, const int* lm_row0,
                           int batch, cudaStream_t s) {
  (void)lm_row0;
  launch_pdl(k_prefill_finish, dim3(batch), dim3(256), 0, s, D, row0, lens);
}

LCA_TRACE_SETTER(trace_set_step)

} // namespace lca
