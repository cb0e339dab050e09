// Causal softmax attention of query rows over a KV-cache layer (Section 2.2 causal masks;
// inside the multi-byte window of Algorithm 1 line 12 the LCA mask is causal as well, so
// every attention of the decode step is "query row r sees cache slots [0, kvlen[r])").
//
// One CTA serves one (sequence, query tile of up to 8 rows, head, key split). Keys and
// values stream through shared memory in tiles of 32; softmax is computed online in fp32.
// With several key splits each CTA writes (max, sum, acc) partials and the last CTA of the
// (sequence, head) combines them in split order (deterministic).
#include <mutex>

#include "common.cuh"

namespace lca {

namespace {

constexpr int kKT = 32;     // keys per tile
constexpr int kThreads = 128;
constexpr int kQTMax = 4;   // query tiles per sequence that may split their key range

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename TC, int HD>
__global__ void __launch_bounds__(kThreads)
k_attn(const float* __restrict__ q, float* __restrict__ out, KV kv, Rows rows, int H, float scale,
       int splits, float* __restrict__ part, int* __restrict__ cnt, int* err) {
  constexpr int QT = kAttnQT;
  __shared__ float qs[QT][HD];
  __shared__ float ks[kKT][HD + 1];
  __shared__ float vs[kKT][HD];
  __shared__ float ps[QT][kKT];
  __shared__ float s_m[QT], s_l[QT], s_corr[QT];
  __shared__ int s_kv[QT];
  __shared__ int s_last;

  const int b = blockIdx.x;
  const int h = blockIdx.z / splits;
  const int sp = blockIdx.z - h * splits;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nrows = rows.seq_count[b];
  const int rbeg = rows.seq_start[b];
  const int ntiles = (nrows + QT - 1) / QT;
  const TC* Kc = reinterpret_cast<const TC*>(kv.k) + ((size_t)b * H + h) * kv.S * HD;
  const TC* Vc = reinterpret_cast<const TC*>(kv.v) + ((size_t)b * H + h) * kv.S * HD;
  const int ld = H * HD;

  // accumulator ownership: row ai, dims ad..ad+DPT-1
  constexpr int DPT = QT * HD / kThreads;
  const int ai = tid / (HD / DPT);
  const int ad = (tid % (HD / DPT)) * DPT;

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
    const int chunk = ((kv_hi + nsp - 1) / nsp + kKT - 1) / kKT * kKT;
    const int lo = split_mode ? sp * chunk : 0;
    const int hi = min(kv_hi, lo + chunk);

    float acc[DPT];
#pragma unroll
    for (int j = 0; j < DPT; ++j) acc[j] = 0.f;

    for (int j0 = lo; j0 < hi; j0 += kKT) {
      const int nk = min(kKT, hi - j0);
      for (int idx = tid; idx < kKT * HD; idx += kThreads) {
        const int kk = idx / HD, dd = idx - kk * HD;
        float kvk = 0.f, kvv = 0.f;
        if (kk < nk) {
          kvk = to_f(Kc[(size_t)(j0 + kk) * HD + dd]);
          kvv = to_f(Vc[(size_t)(j0 + kk) * HD + dd]);
        }
        ks[kk][dd] = kvk;
        vs[kk][dd] = kvv;
      }
      __syncthreads();
      // scores: thread -> key lane, rows warp, warp+4
      for (int i = warp; i < QT; i += kThreads / 32) {
        float sc = -INFINITY;
        if (lane < nk && j0 + lane < s_kv[i]) {
          float s = 0.f;
#pragma unroll 16
          for (int dd = 0; dd < HD; ++dd) s = fmaf(qs[i][dd], ks[lane][dd], s);
          sc = s;
        }
        // online softmax update of row i
        float mx = sc;
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_old = s_m[i];
        const float m_new = fmaxf(m_old, mx);
        const float p = (sc == -INFINITY) ? 0.f : expf(sc - m_new);
        float ssum = p;
#pragma unroll
        for (int o = 16; o; o >>= 1) ssum += __shfl_xor_sync(0xffffffffu, ssum, o);
        ps[i][lane] = p;
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
    // split partials: [b][h][sp] -> acc[QT][HD], m[QT], l[QT]
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
    if (ai < nq) {
      const float* base = part + tile_id * splits * (QT * (HD + 2));
      float M = -INFINITY;
      for (int k = 0; k < splits; ++k) M = fmaxf(M, __ldcg(base + k * (QT * (HD + 2)) + QT * HD + ai));
      float L = 0.f, o[DPT];
#pragma unroll
      for (int j = 0; j < DPT; ++j) o[j] = 0.f;
      for (int k = 0; k < splits; ++k) {
        const float* pk = base + k * (QT * (HD + 2));
        const float mk = __ldcg(pk + QT * HD + ai);
        if (mk == -INFINITY) continue;
        const float w = expf(mk - M);
        L += w * __ldcg(pk + QT * HD + QT + ai);
#pragma unroll
        for (int j = 0; j < DPT; ++j) o[j] += w * __ldcg(pk + ai * HD + ad + j);
      }
      const float il = L > 0.f ? 1.f / L : 0.f;
      float* dst = out + (size_t)(r0 + ai) * ld + h * HD + ad;
#pragma unroll
      for (int j = 0; j < DPT; ++j) dst[j] = o[j] * il;
    }
    if (tid == 0) cnt[tile_id] = 0;
  }
}

template <typename TC, int HD>
void launch(const float* q, float* out, const KV& kv, const Rows& rows, int B, int H, float scale,
            int qtiles_grid, int splits, float* part, int* cnt, int* err, cudaStream_t s) {
  dim3 grid(B, qtiles_grid, H * splits);
  ++g_launches;
  k_attn<TC, HD><<<grid, kThreads, 0, s>>>(q, out, kv, rows, H, scale, splits, part, cnt, err);
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
  k_regular_rows<<<(batch + 255) / 256, 256, 0, s>>>(o.seq_start, o.seq_count, batch, n_rows);
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

void attention(const Dev& D, const float* q, float* out, const KV& kv, const Rows& rows, int B,
               int qtiles_grid, int splits, cudaStream_t s) {
  ProfScope ps(PK_ATTN, 0.0, s);
  if (splits > kMaxAttnSplit) splits = kMaxAttnSplit;
  if (splits < 1) splits = 1;
  launch_any(D.dtype, D.hd, q, out, kv, rows, B, D.H, D.scale, qtiles_grid, splits, D.attn_part,
             D.attn_cnt, D.err, s);
}

} // namespace lca

using namespace lca;

extern "C" {

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

namespace lca {

} // namespace lca
