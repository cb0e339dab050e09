// Persistent block stack: every block of one module (encoder, LM module, next-byte decoder or
// multi-byte window; the pre-norm Llama blocks of Section 2.2 and Section 4.2) in one launch, for
// decode steps with few rows (batch 1 to 4 with a few candidates each).
//
// At batch 1 a block is five dependent operations with little arithmetic each: RMSNorm + Q/K/V +
// RoPE + cache append, attention, Wo + residual, RMSNorm + W1/W3 + SwiGLU, W2 + residual. As five
// launches per block each pays a launch boundary, an activation load and an exit. Here one CTA per
// SM runs the five phases of every block in turn, separated by grid-wide barriers, while a copy
// warp streams the CTA's share of every weight matrix of the whole stack into a ring of shared
// memory. The weights do not depend on the data, so the copy warp runs ahead across phase and
// block boundaries and the HBM weight stream (the roofline of the step) never waits for a barrier.
//
// Work units: 16 output columns x one K-slice of at most 1024 inputs (33 KB of bf16 weights, rows
// padded by 16 bytes). Q/K/V, Wo and W1/W3 have K = d and one slice; W2 has K = F in F / KS slices
// that the same CTA accumulates (no cross-CTA reduction, deterministic). Units go round robin over
// the CTAs, each phase starting where the previous one stopped, so every CTA streams about the same
// bytes over a block.
//
// Split on write: each phase's epilogue stores the next phase's input already in the form the dot
// products take, bf16 halves v = hi + lo (about 16 significant bits): the residual epilogues store
// x * g (g: the next RMSNorm's gain) and the sums of squares of x per 16-column tile, the attention
// stores its output, W1/W3 its SwiGLU output. A phase then stages its rows with a few bulk copies
// issued by one thread (two staging buffers, the next group of rows in flight while the tensor
// cores work on the current one) and converts nothing. Dot products: mma m16n8k16 with the 16
// output columns as M and up to 8 rows as N, hi and lo against the exact bf16 weights, fp32
// accumulation; RMSNorm scales them by the row's inverse RMS from the staged tile sums.
//
// Attention: (sequence, head, key split) items over the CTAs. Each warp walks 16-key tiles: scores
// S^T = K Q^T and values O^T += V^T P^T on mma m16n8k16 (queries and probabilities as bf16 halves),
// its own online softmax per row; the warps combine in shared memory and write the item's partial
// (max, sum, unnormalised output) per row; the last split of a (sequence, head) to finish combines
// the splits in split order. The committed cache prefix (stable during a step) of each item is
// prefetched into L2 during the Q/K/V phase. Everything this kernel writes and reads again is read
// through L2 (ld.global.cg or bulk copies), never from a possibly stale L1 line.
//
// Every wait is bounded. A grid barrier or ring wait that runs out sets kErrTimeout | kErrWaitStack
// in the error word and an abort flag that all CTAs check at each barrier; the copies in flight are
// drained (bounded) before a CTA leaves. No trap. All CTAs must be resident at once: one CTA per SM
// (its shared memory allows no second), a grid of at most the SM count, launched without
// programmatic dependent launch (it starts once its predecessor has completed) and never releasing
// its dependents early (its successor cannot take SMs before every CTA of the stack has exited).
#include <algorithm>
#include <cstdio>

#include "common.cuh"
#include "epilogue.cuh"

namespace lca {

namespace {

constexpr int kSkWarps = 8;                       // compute warps
constexpr int kSkThreads = (kSkWarps + 1) * 32;   // + the copy warp
constexpr int kSkSlots = 5;                       // weight ring slots
constexpr int kSkCols = 16;                       // output columns per unit
constexpr int kSkKS = 1024;                       // largest K-slice
constexpr int kSkKP = kSkKS + 8;                  // padded slot and staging row (bf16 elements)
constexpr int kSkMC = 8;                          // rows per chunk (the MMA's N)
constexpr int kSkHD = 64;                         // head dim
constexpr int kSkQP = kSkHD + 8;                  // padded attention rows (bf16 elements)
constexpr int kSkMaxUnits = 8;                    // units of one phase per CTA
constexpr int kSkSpins = 1 << 22;                 // bounded waits
constexpr int kSkPart = kSkHD + 4;                // floats per attention partial row: O[64], max, sum
constexpr int kSkSsMax = 64;                      // 16-column tiles per row (d <= 1024)

enum : int { PH_QKV = 0, PH_WO = 1, PH_W13 = 2, PH_W2 = 3, PH_N = 4 };

// shared memory (bytes)
constexpr size_t kSlotBytes = (size_t)kSkCols * kSkKP * 2;           // one ring slot
constexpr size_t kRingBytes = kSkSlots * kSlotBytes;
constexpr size_t kStageBufBytes = 2 * (size_t)kSkMC * kSkKP * 2;     // one staging buffer: hi, lo
constexpr size_t kWarpKvBytes = 2 * 16 * kSkQP * 2;                  // a warp's K and V tile
constexpr size_t kQBytes = 2 * (size_t)kSkMC * kSkQP * 2;            // query halves
constexpr size_t kPsBytes = (size_t)kSkWarps * kSkMC * 16 * 4;       // warps' probability tiles
constexpr size_t kAttnBytes = kSkWarps * kWarpKvBytes + kQBytes + kPsBytes;
constexpr size_t kWorkBytes = kStageBufBytes > kAttnBytes ? kStageBufBytes : kAttnBytes;
constexpr size_t kRedBytes = (size_t)kSkWarps * kSkCols * kSkMC * 4;  // warp partials
constexpr size_t kSsBytes = (size_t)kSkMC * kSkSsMax * 4;             // staged tile sums
constexpr size_t kRopeBytes = (size_t)kSkMC * (kSkHD / 2) * 8;        // RoPE cos/sin of rows 0..7
constexpr size_t kSmemBytes = kRingBytes + kWorkBytes + kRedBytes + kSsBytes + kRopeBytes + 1024;
static_assert(kSmemBytes <= 227 * 1024, "shared memory of the stack kernel");
static_assert(kWarpKvBytes >= (size_t)(kSkMC * kSkHD + 2 * kSkMC) * 4, "warp combine area");

struct StackArgs {
  StackRun r;
  float* q;       // [rows][d] queries (after RoPE), fp32
  float* apart;   // attention partials [B][H][splits][rows_cap][kSkPart]
  size_t apart_rows;
  int* cnt;       // [B * H] last-arriver counters
  unsigned* bar;  // [0] barrier arrivals, [1] exits, [2] abort
  __nv_bfloat16 *ahi, *alo;  // normalised-input rows x * g, [rows][d]
  __nv_bfloat16 *thi, *tlo;  // attention output [rows][d]
  __nv_bfloat16 *mhi, *mlo;  // SwiGLU output [rows][F]
  float* ss;                 // sums of squares of x per 16-column tile [rows][d / 16]
  float* w2part;             // W2 partial sums [nsl][w2rows][d]
  int* w2cnt;                // [d / 16] last-arriver counters of W2's column tiles
  int w2rows;
  const float2* rope;
  int* err;
  int d, H, F, B, splits;
  float eps, scale;
};

static __device__ TraceRec* g_trace_s = nullptr;

// The cache layer of a stack layer as the paging helpers see it.
__device__ __forceinline__ KV cache_view(const StackArgs& a, const StackLayer& Ly) {
  KV kv;
  kv.k = Ly.k;
  kv.v = Ly.v;
  kv.S = a.r.S;
  kv.tmaps = nullptr;
  kv.pt = a.r.pt;
  kv.pt_ld = a.r.pt_ld;
  kv.pages = a.r.pages;
  return kv;
}

// ---------------------------------------------------------------- primitives
__device__ __forceinline__ uint32_t su32(const void* p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }
__device__ __forceinline__ void mb_init(uint64_t* b, uint32_t n) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(b)), "r"(n) : "memory");
}
__device__ __forceinline__ void mb_expect(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mb_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(b)) : "memory");
}
__device__ __forceinline__ bool mb_try(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(su32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mb_wait(uint64_t* b, uint32_t parity, int spins = kSkSpins) {
  for (int i = 0; i < spins; ++i)
    if (mb_try(b, parity)) return true;
  return false;
}

// Spin budget of the first ring wait of a phase (a test hook, lca_debug_set_wait_spins, can shorten
// it so that the wait reports late at once; the wait that follows keeps the full budget).
static __device__ int g_stack_first_wait = kSkSpins;

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   su32(dst)),
               "l"(src), "r"(bytes), "r"(su32(bar))
               : "memory");
}
// order this thread's generic-proxy view before its later bulk copies (async proxy)
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.global;" ::: "memory"); }
// barrier of the compute warps (named barrier 1; the copy warp does not take part)
__device__ __forceinline__ void cbar() { asm volatile("bar.sync 1, %0;" ::"n"(kSkWarps * 32) : "memory"); }
__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(su32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(su32(p)));
}
// bf16 halves of a pair: (a, b) = hi + lo
__device__ __forceinline__ void split2(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  const float2 f = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(a - f.x, b - f.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}
__device__ __forceinline__ void split1(float a, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(a);
  lo = __float2bfloat16_rn(a - __bfloat162float(hi));
}

// ---------------------------------------------------------------- units
struct Shape {
  int d, F, KS, nsl;  // K-slice of every unit, W2 slices
};
// units of a phase; W2's unit u is column tile u / nsl, K-slice u % nsl (slice-minor, so that with
// nsl dividing the grid the units one CTA owns share a slice)
__device__ __forceinline__ int units_of(const Shape& z, int p) {
  return p == PH_QKV ? 3 * z.d / kSkCols : p == PH_W13 ? 2 * z.F / kSkCols : p == PH_WO ? z.d / kSkCols
                                                                                  : z.d / kSkCols * z.nsl;
}
// unit i of phase p of block l that CTA c owns (-1: none): round robin over the G CTAs, each phase
// starting after the last CTA of the phase before it
__device__ __forceinline__ int my_unit(const Shape& z, int l, int p, int c, int G, int i) {
  const int per_layer = units_of(z, PH_QKV) + units_of(z, PH_WO) + units_of(z, PH_W13) + units_of(z, PH_W2);
  long long off = (long long)l * per_layer;
  for (int q = 0; q < p; ++q) off += units_of(z, q);
  const int first = (int)(((long long)c - off) % G + G) % G;
  const int u = first + i * G;
  return u < units_of(z, p) ? u : -1;
}
// weight rows of a unit: the first row of its 16 and the row length K
__device__ __forceinline__ const __nv_bfloat16* unit_src(const StackLayer& L, const Shape& z, int p, int u, int& K) {
  switch (p) {
    case PH_QKV: K = z.d; return L.wqkv + (size_t)u * kSkCols * z.d;
    case PH_WO: K = z.d; return L.wo + (size_t)u * kSkCols * z.d;
    case PH_W13: K = z.d; return L.w13 + (size_t)u * kSkCols * z.d;
    default: K = z.F; return L.w2 + (size_t)(u / z.nsl) * kSkCols * z.F + (size_t)(u % z.nsl) * z.KS;
  }
}

// [lo, hi) of split sp when n keys from base are shared in 16-key tiles
__device__ __forceinline__ void key_share(int base, int n, int splits, int sp, int& lo, int& hi) {
  const int per = ((n + splits - 1) / splits + 15) / 16 * 16;
  lo = base + min(n, sp * per);
  hi = base + min(n, sp * per + per);
}

struct Smem {
  __nv_bfloat16* ring;  // [slots][16][KP]
  unsigned char* work;  // two staging buffers ([8][KP] hi, [8][KP] lo each), or the attention tiles
  float* red;           // [warps][16][8] warp partials
  float* ss;            // [2][8][64] staged tile sums of squares
  float2* rope;         // [8][32] RoPE cos/sin of rows 0..7
  uint64_t* full;       // [slots]
  uint64_t* empty;      // [slots]
  uint64_t* sbar;       // [2] staging buffers
  float* inv;           // [2][8] inverse RMS of the staged rows
  int* misc;  // [0] abort, [1] issued, [2] copy warp done, [3] last arriver, [8..15] kl, [16..23] b, [24..31] slot,
              // [32..] W2 last arrivers, [40..47] page of the slot
};
__device__ __forceinline__ __nv_bfloat16* stage_hi(Smem& S, int b) {
  return reinterpret_cast<__nv_bfloat16*>(S.work + (size_t)b * kStageBufBytes);
}

// Phase timeline for the launch tracer: thread 0 of every CTA records, per phase of every block,
// when the phase began (its barrier returned) and when its own work ended (it entered the next
// barrier); tag 100 + phase, mark[0] = block.
__device__ __forceinline__ void trace_phase(int phase, int layer, unsigned long long t0) {
  if (!g_trace_s || threadIdx.x != 0) return;
  const unsigned i = atomicAdd(g_trace_n, 1u);
  if (i >= g_trace_cap) return;
  TraceRec r{};
  r.t0 = t0;
  r.tw = t0;
  r.t1 = gtimer();
  r.tag = 100 + phase;
  r.cta = blockIdx.x;
  r.sm = (int)smid();
  r.mark[0] = layer;
  g_trace_s[i] = r;
}

// Grid-wide barrier of the compute warps; false when it ran out or another CTA gave up.
__device__ bool grid_sync(const StackArgs& a, unsigned& target, int G, Smem& S) {
  cbar();
  if (threadIdx.x == 0) {
    // a CTA that gave up a ring wait tells the others at once
    if (*(volatile int*)&S.misc[0]) atomicExch(a.bar + 2, 1u);
    target += (unsigned)G;
    __threadfence();
    atomicAdd(a.bar, 1u);
    int n = 0;
    bool ok = true;
    while (ld_acquire(a.bar) < target) {
      if (++n >= kSkSpins || ((n & 255) == 0 && *(volatile unsigned*)(a.bar + 2))) {
        ok = false;
        break;
      }
    }
    __threadfence();
    if (!ok || *(volatile unsigned*)(a.bar + 2)) {
      if (n >= kSkSpins) atomicOr(a.err, kErrTimeout | kErrWaitStack);
      atomicExch(a.bar + 2, 1u);
      *(volatile int*)&S.misc[0] = 1;
    }
  }
  cbar();
  return *(volatile int*)&S.misc[0] == 0;
}

// ---------------------------------------------------------------- staging by bulk copies
// A phase's input: pre-split rows (hi, lo) of row stride ld, and, for the RMSNorm phases, the
// per-tile sums of squares (ss_ld tiles per row). Its rows in blocks (chunk of up to 8 rows, K-slice)
// in chunk-major order; consecutive blocks are packed into groups of at most 8 staged rows.
struct PhaseIn {
  const __nv_bfloat16* hi;
  const __nv_bfloat16* lo;
  int ld;
  const float* ss;  // nullptr: no RMSNorm
  int ss_ld;
};
__device__ __forceinline__ int chunk_rows(int M, int chunk) { return min(kSkMC, M - chunk * kSkMC); }

// Thread 0: bulk copies of the blocks [k0, k1) into staging buffer b (rows packed from slot 0).
__device__ void issue_group(const PhaseIn& in, int KS, int M, int nsl, int k0, int k1, int b, Smem& S,
                            int sl_fixed = -1) {
  uint32_t bytes = 0;
  for (int k = k0; k < k1; ++k) {
    const int mc = chunk_rows(M, k / nsl);
    bytes += (uint32_t)mc * (uint32_t)(KS * 2 * 2 + (in.ss ? in.ss_ld * 4 : 0));
  }
  fence_proxy_async();
  mb_expect(&S.sbar[b], bytes);
  __nv_bfloat16* hi = stage_hi(S, b);
  __nv_bfloat16* lo = hi + (size_t)kSkMC * kSkKP;
  float* ss = S.ss + (size_t)b * kSkMC * kSkSsMax;
  int slot = 0;
  for (int k = k0; k < k1; ++k) {
    const int chunk = k / nsl, mc = chunk_rows(M, chunk);
    const int sl = sl_fixed >= 0 ? sl_fixed : k - chunk * nsl;
    for (int i = 0; i < mc; ++i, ++slot) {
      const size_t row = (size_t)(chunk * kSkMC + i);
      bulk_g2s(hi + (size_t)slot * kSkKP, in.hi + row * in.ld + (size_t)sl * KS, (uint32_t)(KS * 2), &S.sbar[b]);
      bulk_g2s(lo + (size_t)slot * kSkKP, in.lo + row * in.ld + (size_t)sl * KS, (uint32_t)(KS * 2), &S.sbar[b]);
      if (in.ss) bulk_g2s(ss + (size_t)slot * kSkSsMax, in.ss + row * in.ss_ld, (uint32_t)(in.ss_ld * 4), &S.sbar[b]);
    }
  }
}

// Sum over the 8 lanes of a row (its 16 columns in the epilogue layout); every lane gets it.
__device__ __forceinline__ float row8_sum(float v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  v += __shfl_xor_sync(0xffffffffu, v, 2);
  v += __shfl_xor_sync(0xffffffffu, v, 4);
  return v;
}

// Residual epilogue (Wo, W2): x += v for the pair (r, col); then the next RMSNorm's input, split,
// and the tile's sum of squares (gain == nullptr: x only). Called by all 64 epilogue threads.
__device__ __forceinline__ void resid_out(const StackArgs& a, int r, int col, bool ok, float2 res, float v0, float v1,
                                          const float2* gain, int tile) {
  const float2 xn = make_float2(res.x + v0, res.y + v1);
  if (ok) *reinterpret_cast<float2*>(a.r.x + (size_t)r * a.d + col) = xn;
  if (gain) {
    const float sq = row8_sum(ok ? xn.x * xn.x + xn.y * xn.y : 0.f);
    if (ok) {
      const float2 g = *gain;
      uint32_t hi, lo;
      split2(xn.x * g.x, xn.y * g.y, hi, lo);
      *reinterpret_cast<uint32_t*>(a.ahi + (size_t)r * a.d + col) = hi;
      *reinterpret_cast<uint32_t*>(a.alo + (size_t)r * a.d + col) = lo;
      if ((threadIdx.x & 7) == 0) a.ss[(size_t)r * (a.d / kSkCols) + tile] = sq;
    }
  }
}

// Partial dot products of weight slot wt against the 8 staged rows (hi, lo at xh) over the K-steps
// kw, kw + step, ... of this warp: ldmatrix fragments (weights: 16 columns x 16 K; rows: hi and lo
// of 8 rows x 16 K in one x4 load), four independent accumulation chains. Staged rows past the
// chunk's rows hold stale values; they only reach output columns that are not stored.
__device__ __forceinline__ void wave_mma(const __nv_bfloat16* wt, int KS, const __nv_bfloat16* xh, int kw, int step,
                                         float (&acc)[4]) {
  const int lane = threadIdx.x & 31;
  const int jm = lane >> 3, rm = lane & 7;
  // weights: matrix jm = (columns 8 (jm & 1).., K 8 (jm >> 1)..); rows: matrix jm = (hi | lo for
  // jm >> 1, K 8 (jm & 1)..)
  const __nv_bfloat16* pa = wt + (size_t)(rm + 8 * (jm & 1)) * kSkKP + 8 * (jm >> 1);
  const __nv_bfloat16* pb = xh + (size_t)(jm >> 1) * kSkMC * kSkKP + (size_t)rm * kSkKP + 8 * (jm & 1);
  float c[4][4];
#pragma unroll
  for (int u = 0; u < 4; ++u) c[u][0] = c[u][1] = c[u][2] = c[u][3] = 0.f;
  const int nk = (KS / 16 - kw + step - 1) / step;  // K-steps of this warp
  int i = 0;
  for (; i + 4 <= nk; i += 4) {
    uint32_t af[4][4], bf[4][4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int kb = (kw + (i + u) * step) * 16;
      ldsm_x4(af[u], pa + kb);
      ldsm_x4(bf[u], pb + kb);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      mma16816(c[u], af[u], bf[u][0], bf[u][1]);
      mma16816(c[u], af[u], bf[u][2], bf[u][3]);
    }
  }
  for (; i < nk; ++i) {
    const int kb = (kw + i * step) * 16;
    uint32_t af[4], bf[4];
    ldsm_x4(af, pa + kb);
    ldsm_x4(bf, pb + kb);
    mma16816(c[0], af, bf[0], bf[1]);
    mma16816(c[0], af, bf[2], bf[3]);
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) acc[j] = (c[0][j] + c[1][j]) + (c[2][j] + c[3][j]);
}

// Thread 0: stage chunk k (rows 8k..8k+7) of K-slice sl of the phase input.
__device__ __forceinline__ void stage_chunk(const PhaseIn& in, int KS, int M, int sl, int k, Smem& S) {
  issue_group(in, KS, M, 1, k, k + 1, 0, S, sl);
}

// One linear phase (p) of block l. This CTA's units go in waves of up to kSkSlots units that share a
// K-slice (their weights resident together): the wave's warps split over its units (8, 4 or 2 warps
// a unit, each over every 8th, 4th or 2nd K-step), one reduction and one epilogue pass per chunk of
// 8 rows serve every unit of the wave. W2 units write K-slice partials; the last of a column tile's
// nsl units to finish adds them (in slice order) and runs the residual epilogue.
// Lnext: the next block (its attention RMSNorm gain for W2's split output), or nullptr.
__device__ void linear_phase(const StackArgs& a, const StackLayer& Ly, const StackLayer* Lnext, const Shape& z,
                             int l, int p, int c, int G, int M, int& seq, int (&uses)[2], Smem& S) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, q4 = lane & 3;
  PhaseIn in{};
  switch (p) {
    case PH_QKV: in = PhaseIn{a.ahi, a.alo, a.d, a.ss, a.d / kSkCols}; break;
    case PH_WO: in = PhaseIn{a.thi, a.tlo, a.d, nullptr, 0}; break;
    case PH_W13: in = PhaseIn{a.ahi, a.alo, a.d, a.ss, a.d / kSkCols}; break;
    default: in = PhaseIn{a.mhi, a.mlo, a.F, nullptr, 0}; break;
  }
  const bool w2 = p == PH_W2;
  const bool w2split = w2 && z.nsl > 1;
  int us[kSkMaxUnits];
  int nu = 0;
  for (int i = 0; i < kSkMaxUnits; ++i) {
    const int u = my_unit(z, l, p, c, G, i);
    if (u < 0) break;
    us[nu++] = u;
  }
  const int chunks = (M + kSkMC - 1) / kSkMC;
  const float* gain_next = p == PH_WO ? Ly.mlp_norm : (w2 && Lnext ? Lnext->attn_norm : nullptr);
  // epilogue layout: unit j of the wave, row er of the chunk, column pair ep of the unit's 16
  const int ej = tid >> 6, er = (tid & 63) >> 3, ep = tid & 7;
  int staged_sl = -1;  // K-slice whose chunks 0 and 1 sit in the staging buffers
  const bool tr = g_trace_s && tid == 0;
  for (int i0 = 0; i0 < nu;) {
    const int sl = w2 ? us[i0] % z.nsl : 0;
    int i1 = i0 + 1;
    while (i1 < nu && i1 - i0 < kSkSlots && (w2 ? us[i1] % z.nsl : 0) == sl) ++i1;
    const int nw = i1 - i0;
    const unsigned long long tu0 = tr ? gtimer() : 0;
    unsigned long long tw = 0, tst = 0, tmm = 0;
    // stage this slice's first chunk (kept for the next wave when it is the only chunk)
    if (chunks > 0 && !(staged_sl == sl && chunks == 1)) {
      if (staged_sl != -1) cbar();  // every warp is done with the staging buffer
      if (tid == 0) stage_chunk(in, z.KS, M, sl, 0, S);
      ++uses[0];
      staged_sl = sl;
    }
    // epilogue operands that do not depend on the dot products: residual (chunk 0) and gain
    const int u_e = ej < nw ? us[i0 + ej] : 0;
    const int tile_e = w2 ? u_e / z.nsl : u_e;
    const int col = tile_e * kSkCols + 2 * ep;
    float2 res0 = make_float2(0.f, 0.f), gn = make_float2(1.f, 1.f);
    if (ej < nw && (p == PH_WO || (w2 && !w2split))) {
      if (M > 0 && er < chunk_rows(M, 0)) res0 = __ldcg(reinterpret_cast<const float2*>(a.r.x + (size_t)er * a.d + col));
      if (gain_next) gn = __ldg(reinterpret_cast<const float2*>(gain_next + col));
    }
    // the wave's weight slots have landed (bounded; on a timeout the data is garbage and the kernel
    // gives up at the next barrier)
    for (int j = 0; j < nw; ++j) {
      const int s = (seq + j) % kSkSlots;
      const uint32_t par = (uint32_t)(((seq + j) / kSkSlots) & 1);
      if (!mb_wait(&S.full[s], par, i0 == 0 && j == 0 ? g_stack_first_wait : kSkSpins)) {
        // late: record it, then wait once more (bounded) so that no copy is in flight into a slot
        // that goes back to the copy warp; the kernel gives up at the next barrier
        if (tid == 0) atomicOr(a.err, kErrTimeout | kErrWaitStack);
        *(volatile int*)&S.misc[0] = 1;
        mb_wait(&S.full[s], par);
      }
    }
    if (tr) tw = gtimer();
    const int wpu = nw == 1 ? kSkWarps : (nw == 2 ? kSkWarps / 2 : kSkWarps / 4);
    const int wj = warp / wpu, kw = warp - wj * wpu;
    for (int k = 0; k < chunks; ++k) {
      const int mc = chunk_rows(M, k);
      if (k >= 1) {
        // chunk k replaces chunk k - 1 (every warp left it at the barrier that ended its epilogue)
        if (tid == 0) stage_chunk(in, z.KS, M, sl, k, S);
        ++uses[0];
      }
      if (!mb_wait(&S.sbar[0], (uint32_t)((uses[0] - 1) & 1))) {
        if (tid == 0) atomicOr(a.err, kErrTimeout | kErrWaitStack);
        *(volatile int*)&S.misc[0] = 1;
        mb_wait(&S.sbar[0], (uint32_t)((uses[0] - 1) & 1));
      }
      if (in.ss) {
        // inverse RMS of each staged row from its tile sums (warp w: row w)
        const float* ssb = S.ss + (size_t)warp * kSkSsMax;
        float t = 0.f;
        for (int j = lane; j < in.ss_ld; j += 32) t += ssb[j];
#pragma unroll
        for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) S.inv[warp] = rsqrtf(t / (float)a.d + a.eps);
      }
      if (tr && k == 0) tst = gtimer();
      float c0[4] = {0.f, 0.f, 0.f, 0.f};
      if (wj < nw) {
        const __nv_bfloat16* wt = S.ring + (size_t)((seq + wj) % kSkSlots) * kSkCols * kSkKP;
        wave_mma(wt, z.KS, stage_hi(S, 0), kw, wpu, c0);
      }
      *reinterpret_cast<float2*>(S.red + ((size_t)(warp * kSkCols + g) * kSkMC + 2 * q4)) = make_float2(c0[0], c0[1]);
      *reinterpret_cast<float2*>(S.red + ((size_t)(warp * kSkCols + g + 8) * kSkMC + 2 * q4)) =
          make_float2(c0[2], c0[3]);
      cbar();
      if (tr && k == 0) tmm = gtimer();
      if (ej < nw) {
        const int r = k * kSkMC + er;
        const bool ok = er < mc;
        const int c0i = 2 * ep;
        float v0 = 0.f, v1 = 0.f;
        for (int w = ej * wpu; w < (ej + 1) * wpu; ++w) {
          v0 += S.red[(w * kSkCols + c0i) * kSkMC + er];
          v1 += S.red[(w * kSkCols + c0i + 1) * kSkMC + er];
        }
        if (in.ss && ok) {
          const float iv = S.inv[er];
          v0 *= iv;
          v1 *= iv;
        }
        if (p == PH_QKV) {
          if (ok) {
            const int part = col / a.d, cc = col - part * a.d, h = cc / kSkHD, dd = cc - h * kSkHD;
            int rb, rslot, rpg;
            float2 cs;
            if (r < kSkMC) {
              rb = S.misc[16 + r];
              rslot = S.misc[24 + r];
              rpg = S.misc[40 + r];
              cs = S.rope[r * (kSkHD / 2) + (dd >> 1)];
            } else {
              rb = a.r.rows.b[r];
              rslot = a.r.rows.slot[r];
              rpg = a.r.pt ? a.r.rows.page[r] : 0;
              cs = a.rope[(size_t)a.r.rows.pos[r] * (kSkHD / 2) + (dd >> 1)];
            }
            if (part < 2) {
              const float x0 = v0 * cs.x - v1 * cs.y, x1 = v0 * cs.y + v1 * cs.x;
              v0 = x0;
              v1 = x1;
            }
            if (part == 0) {
              *reinterpret_cast<float2*>(a.q + (size_t)r * a.d + cc) = make_float2(v0, v1);
            } else if (!kv_write_ok(cache_view(a, Ly), rslot, rpg)) {
              atomicOr(a.err, kErrIndex);
            } else {
              __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(part == 1 ? Ly.k : Ly.v) +
                                   kv_addr(cache_view(a, Ly), a.H, kSkHD, rb, h, rslot, rpg) + dd;
              *reinterpret_cast<__nv_bfloat162*>(dst) = __floats2bfloat162_rn(v0, v1);
            }
          }
        } else if (p == PH_W13) {
          if (ok) {
            // packed rows (2j, 2j + 1) = (W1_j, W3_j): SwiGLU output column j, split
            const float m = silu_f(v0) * v1;
            __nv_bfloat16 hi, lo;
            split1(m, hi, lo);
            const size_t o = (size_t)r * a.F + (col >> 1);
            a.mhi[o] = hi;
            a.mlo[o] = lo;
          }
        } else if (w2split) {
          if (ok)
            *reinterpret_cast<float2*>(a.w2part + ((size_t)sl * a.w2rows + r) * a.d + col) = make_float2(v0, v1);
        } else {
          const float2 res =
              k == 0 ? res0
                     : (ok ? __ldcg(reinterpret_cast<const float2*>(a.r.x + (size_t)r * a.d + col)) : make_float2(0.f, 0.f));
          resid_out(a, r, col, ok, res, v0, v1, gain_next ? &gn : nullptr, tile_e);
        }
      }
      cbar();  // S.red and this chunk's staging are free again
    }
    if (chunks > 1) staged_sl = -2;  // the buffer holds the last chunk: stage again for the next wave
    // the wave's slots go back to the copy warp
    if (tid == 0)
      for (int j = 0; j < nw; ++j) mb_arrive(&S.empty[(seq + j) % kSkSlots]);
    seq += nw;
    if (tr) {
      const unsigned k = atomicAdd(g_trace_n, 1u);
      if (k < g_trace_cap) {
        TraceRec rr{};
        rr.t0 = tu0;
        rr.tw = tu0;
        rr.t1 = gtimer();
        rr.tag = 120 + p;
        rr.cta = c;
        rr.sm = l;
        rr.mark[0] = (int)(tw - tu0);
        rr.mark[1] = tst ? (int)(tst - tu0) : 0;
        rr.mark[2] = tmm ? (int)(tmm - tu0) : 0;
        g_trace_s[k] = rr;
      }
    }
    i0 = i1;
  }
  if (!w2split) return;
  // W2: the last of a column tile's slice units adds the slices in order, then the residual epilogue.
  // Residual and gain of the first chunk are loaded before the arrival (x does not change in this
  // phase before the finalisation, which only the last arriver of a tile runs).
  constexpr int kPre = 2;  // units whose operands are loaded early (a CTA owns at most two W2 units)
  float2 fres[kPre], fgain[kPre];
  for (int i = 0; i < kPre; ++i) {
    fres[i] = make_float2(0.f, 0.f);
    fgain[i] = make_float2(1.f, 1.f);
    if (i < nu && tid < 64) {
      const int col = (us[i] / z.nsl) * kSkCols + 2 * ep;
      if (M > 0 && er < chunk_rows(M, 0)) fres[i] = __ldcg(reinterpret_cast<const float2*>(a.r.x + (size_t)er * a.d + col));
      if (gain_next) fgain[i] = __ldg(reinterpret_cast<const float2*>(gain_next + col));
    }
  }
  __threadfence();
  cbar();
  for (int i = 0; i < nu; ++i)
    if (tid == 32 * i) S.misc[32 + i] = atomicAdd(a.w2cnt + us[i] / z.nsl, 1) == z.nsl - 1;
  cbar();
  __threadfence();
  for (int i = 0; i < nu; ++i) {
    if (!S.misc[32 + i]) continue;
    const int tile = us[i] / z.nsl;
    if (tid < 64) {
      const int col = tile * kSkCols + 2 * ep;
      const float2 gn = i < kPre ? fgain[i]
                                 : (gain_next ? __ldg(reinterpret_cast<const float2*>(gain_next + col))
                                              : make_float2(1.f, 1.f));
      for (int k = 0; k < chunks; ++k) {
        const int r = k * kSkMC + er;
        const bool ok = er < chunk_rows(M, k);
        float v0 = 0.f, v1 = 0.f;
        float2 res = make_float2(0.f, 0.f);
        if (ok) {
          res = (k == 0 && i < kPre) ? fres[i] : __ldcg(reinterpret_cast<const float2*>(a.r.x + (size_t)r * a.d + col));
          for (int s2 = 0; s2 < z.nsl; ++s2) {
            const float2 pv = __ldcg(reinterpret_cast<const float2*>(a.w2part + ((size_t)s2 * a.w2rows + r) * a.d + col));
            v0 += pv.x;
            v1 += pv.y;
          }
        }
        resid_out(a, r, col, ok, res, v0, v1, gain_next ? &gn : nullptr, tile);
      }
    }
    if (tid == 0) a.w2cnt[tile] = 0;
  }
}

// Before the first block: x (written by the kernels before this one) into the split input of the
// first Q/K/V phase (x * g_attn of block 0) with its tile sums of squares; 16-column tiles over the
// CTAs.
__device__ void prologue(const StackArgs& a, const StackLayer& L0, int c, int G, int M) {
  const int tid = threadIdx.x;
  if (tid >= 64) return;
  const int er = tid >> 3, ep = tid & 7;
  const int tiles = a.d / kSkCols;
  for (int t = c; t < tiles; t += G) {
    const int col = t * kSkCols + 2 * ep;
    const float2 g = __ldg(reinterpret_cast<const float2*>(L0.attn_norm + col));
    for (int r0 = 0; r0 < M; r0 += kSkMC) {
      const int r = r0 + er;
      const bool ok = r < M;
      const float2 xv =
          ok ? __ldcg(reinterpret_cast<const float2*>(a.r.x + (size_t)r * a.d + col)) : make_float2(0.f, 0.f);
      const float sq = row8_sum(xv.x * xv.x + xv.y * xv.y);
      if (ok) {
        uint32_t hi, lo;
        split2(xv.x * g.x, xv.y * g.y, hi, lo);
        *reinterpret_cast<uint32_t*>(a.ahi + (size_t)r * a.d + col) = hi;
        *reinterpret_cast<uint32_t*>(a.alo + (size_t)r * a.d + col) = lo;
        if (ep == 0) a.ss[(size_t)r * tiles + t] = sq;
      }
    }
  }
}

// The attention of block l: (sequence, head, key split) items of this CTA, then the last split of
// each (sequence, head) combines; the output rows are stored split (hi, lo) for Wo.
__device__ void attention_phase(const StackArgs& a, const StackLayer& Ly, int c, int G, Smem& S) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, q4 = lane & 3;
  const int H = a.H, splits = a.splits;
  const int items = a.B * H * splits;
  unsigned char* wk = S.work + (size_t)warp * kWarpKvBytes;
  __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(wk);  // [16][QP]
  __nv_bfloat16* Vs = Ks + 16 * kSkQP;                        // [16][QP]
  __nv_bfloat16* Qh = reinterpret_cast<__nv_bfloat16*>(S.work + kSkWarps * kWarpKvBytes);  // [8][QP]
  __nv_bfloat16* Ql = Qh + kSkMC * kSkQP;
  float* Ps = reinterpret_cast<float*>(S.work + kSkWarps * kWarpKvBytes + kQBytes) + warp * kSkMC * 16;  // [8][16]
  float* cw = reinterpret_cast<float*>(wk);  // after the key loop: [8][64] O, [8] max, [8] sum
  int* s_kl = S.misc + 8;                    // [8] cache lengths of the tile's rows
  const size_t ld = (size_t)H * kSkHD;
  const bool tr = g_trace_s && tid == 0;
  for (int item = c; item < items; item += G) {
    const unsigned long long ti0 = tr ? gtimer() : 0;
    unsigned long long tq = 0, tk = 0, tpw = 0;
    const int b = item / (H * splits), h = (item / splits) % H, sp = item % splits;
    const int nrows = a.r.rows.seq_count[b], rbeg = a.r.rows.seq_start[b];
    int Sb = 0;
    if (a.r.stable) {
      Sb = a.r.stable[(size_t)b * a.r.stable_stride] + a.r.stable_add;
      Sb = Sb < 0 ? 0 : (Sb > a.r.S ? a.r.S : Sb);
    }
    const KV kvv = cache_view(a, Ly);
    const __nv_bfloat16* Kc = reinterpret_cast<const __nv_bfloat16*>(Ly.k);
    const __nv_bfloat16* Vc = reinterpret_cast<const __nv_bfloat16*>(Ly.v);
    float* part = a.apart + (((size_t)b * H + h) * splits + sp) * a.apart_rows * kSkPart;
    const int tiles = (nrows + kSkMC - 1) / kSkMC;
    for (int qt = 0; qt < tiles; ++qt) {
      const int r0 = rbeg + qt * kSkMC, nq = min(kSkMC, nrows - qt * kSkMC);
      if (qt * kSkMC >= (int)a.apart_rows) {
        if (tid == 0) atomicOr(a.err, kErrIndex);
        break;
      }
      // queries (pre-scaled) as bf16 halves; cache lengths
      for (int idx = tid; idx < kSkMC * kSkHD / 2; idx += kSkWarps * 32) {
        const int i = idx / (kSkHD / 2), c2 = idx - i * (kSkHD / 2);
        float2 v = make_float2(0.f, 0.f);
        if (i < nq) v = __ldcg(reinterpret_cast<const float2*>(a.q + (size_t)(r0 + i) * ld + h * kSkHD + 2 * c2));
        uint32_t hi, lo;
        split2(v.x * a.scale, v.y * a.scale, hi, lo);
        *reinterpret_cast<uint32_t*>(Qh + i * kSkQP + 2 * c2) = hi;
        *reinterpret_cast<uint32_t*>(Ql + i * kSkQP + 2 * c2) = lo;
      }
      if (tid < kSkMC) {
        int k = 0;
        if (tid < nq) {
          k = a.r.rows.kvlen[r0 + tid];
          if (k < 0 || k > a.r.S) {
            atomicOr(a.err, kErrIndex);
            k = k < 0 ? 0 : a.r.S;
          }
        }
        s_kl[tid] = k;
      }
      cbar();
      if (tr && qt == 0) tq = gtimer();
      int kl[kSkMC];
      int kv_hi = 0;
#pragma unroll
      for (int i = 0; i < kSkMC; ++i) {
        kl[i] = s_kl[i];
        kv_hi = max(kv_hi, kl[i]);
      }
      // this split's keys: stable slots [lo1, hi1), then slots [lo2, hi2) appended in this step
      int lo1, hi1, lo2, hi2;
      key_share(0, min(Sb, kv_hi), splits, sp, lo1, hi1);
      key_share(Sb, max(kv_hi - Sb, 0), splits, sp, lo2, hi2);
      const int n1 = hi1 - lo1, nv = n1 + (hi2 - lo2);
      const int rr0 = 2 * q4, rr1 = 2 * q4 + 1;  // this lane's rows in the score tile
      float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
      float o[4][4];
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
      for (int t0 = warp * 16; t0 < nv; t0 += kSkWarps * 16) {
        // K and V rows of the tile's 16 keys through L2 (keys of this step were written by this
        // kernel); rows past the range are zero
        uint4 kv[8];
#pragma unroll
        for (int m = 0; m < 8; ++m) {
          const int idx = lane + 32 * (m & 3);
          const int j = idx >> 3, e8 = idx & 7;
          const int v = t0 + j;
          kv[m] = make_uint4(0u, 0u, 0u, 0u);
          if (v < nv) {
            const int slot = v < n1 ? lo1 + v : lo2 + (v - n1);
            const __nv_bfloat16* base = (m < 4 ? Kc : Vc) + kv_off(kvv, H, kSkHD, b, h, slot) + e8 * 8;
            kv[m] = __ldcg(reinterpret_cast<const uint4*>(base));
          }
        }
#pragma unroll
        for (int m = 0; m < 8; ++m) {
          const int idx = lane + 32 * (m & 3);
          const int j = idx >> 3, e8 = idx & 7;
          *reinterpret_cast<uint4*>((m < 4 ? Ks : Vs) + j * kSkQP + e8 * 8) = kv[m];
        }
        __syncwarp();
        // S^T[16 keys][8 rows] = K Q^T
        float sacc[4] = {0.f, 0.f, 0.f, 0.f};
        const int jm = lane >> 3, rm = lane & 7;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          uint32_t af[4];
          ldsm_x4(af, Ks + (rm + 8 * (jm & 1)) * kSkQP + ks * 16 + 8 * (jm >> 1));
          const uint32_t* ph = reinterpret_cast<const uint32_t*>(Qh + g * kSkQP + ks * 16 + 2 * q4);
          const uint32_t* pl = reinterpret_cast<const uint32_t*>(Ql + g * kSkQP + ks * 16 + 2 * q4);
          mma16816(sacc, af, ph[0], ph[4]);
          mma16816(sacc, af, pl[0], pl[4]);
        }
        // mask: key t0 + g (c0, c1) and t0 + g + 8 (c2, c3); rows rr0 (c0, c2) and rr1 (c1, c3)
        const int va = t0 + g, vb = t0 + g + 8;
        const int sa = va < n1 ? lo1 + va : lo2 + (va - n1);
        const int sb = vb < n1 ? lo1 + vb : lo2 + (vb - n1);
        int klr0 = 0, klr1 = 0;
#pragma unroll
        for (int i = 0; i < kSkMC; ++i) {
          if (i == rr0) klr0 = kl[i];
          if (i == rr1) klr1 = kl[i];
        }
        const float s0 = (va < nv && sa < klr0) ? sacc[0] : -INFINITY;
        const float s1 = (va < nv && sa < klr1) ? sacc[1] : -INFINITY;
        const float s2 = (vb < nv && sb < klr0) ? sacc[2] : -INFINITY;
        const float s3 = (vb < nv && sb < klr1) ? sacc[3] : -INFINITY;
        float t0m = fmaxf(s0, s2), t1m = fmaxf(s1, s3);
#pragma unroll
        for (int o2 = 4; o2 <= 16; o2 <<= 1) {
          t0m = fmaxf(t0m, __shfl_xor_sync(0xffffffffu, t0m, o2));
          t1m = fmaxf(t1m, __shfl_xor_sync(0xffffffffu, t1m, o2));
        }
        const float n0 = fmaxf(m0, t0m), n1m = fmaxf(m1, t1m);
        const float c0s = n0 == -INFINITY ? 1.f : __expf(m0 - n0);
        const float c1s = n1m == -INFINITY ? 1.f : __expf(m1 - n1m);
        const float p0 = s0 == -INFINITY ? 0.f : __expf(s0 - n0);
        const float p1 = s1 == -INFINITY ? 0.f : __expf(s1 - n1m);
        const float p2 = s2 == -INFINITY ? 0.f : __expf(s2 - n0);
        const float p3 = s3 == -INFINITY ? 0.f : __expf(s3 - n1m);
        m0 = n0;
        m1 = n1m;
        l0 = l0 * c0s + p0 + p2;
        l1 = l1 * c1s + p1 + p3;
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) {
          o[mt][0] *= c0s;
          o[mt][1] *= c1s;
          o[mt][2] *= c0s;
          o[mt][3] *= c1s;
        }
        // P^T as the B operand: through shared memory (row-major [row][key])
        Ps[rr0 * 16 + g] = p0;
        Ps[rr1 * 16 + g] = p1;
        Ps[rr0 * 16 + g + 8] = p2;
        Ps[rr1 * 16 + g + 8] = p3;
        __syncwarp();
        uint32_t bh0, bl0, bh1, bl1;
        split2(Ps[g * 16 + 2 * q4], Ps[g * 16 + 2 * q4 + 1], bh0, bl0);
        split2(Ps[g * 16 + 2 * q4 + 8], Ps[g * 16 + 2 * q4 + 9], bh1, bl1);
        // O^T[64 dims][8 rows] += V^T P^T
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) {
          uint32_t af[4];
          ldsm_x4_t(af, Vs + (rm + 8 * (jm >> 1)) * kSkQP + mt * 16 + 8 * (jm & 1));
          mma16816(o[mt], af, bh0, bh1);
          mma16816(o[mt], af, bl0, bl1);
        }
        __syncwarp();  // Ks, Vs and Ps are rewritten by the next tile
      }
      if (tr && qt == 0) tk = gtimer();
      // the warp's sums over its lanes' keys
#pragma unroll
      for (int o2 = 4; o2 <= 16; o2 <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, o2);
        l1 += __shfl_xor_sync(0xffffffffu, l1, o2);
      }
      // warp partials into the warp's own area (its K/V tile is no longer needed)
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        cw[rr0 * kSkHD + mt * 16 + g] = o[mt][0];
        cw[rr1 * kSkHD + mt * 16 + g] = o[mt][1];
        cw[rr0 * kSkHD + mt * 16 + g + 8] = o[mt][2];
        cw[rr1 * kSkHD + mt * 16 + g + 8] = o[mt][3];
      }
      if (g == 0) {
        cw[kSkMC * kSkHD + rr0] = m0;
        cw[kSkMC * kSkHD + rr1] = m1;
        cw[kSkMC * kSkHD + kSkMC + rr0] = l0;
        cw[kSkMC * kSkHD + kSkMC + rr1] = l1;
      }
      cbar();
      // the CTA's partial per row: max, sum and unnormalised output over the warps
      {
        const int i = tid >> 5, d2 = (tid & 31) * 2;
        if (i < nq && qt * kSkMC + i < (int)a.apart_rows) {
          float M = -INFINITY;
#pragma unroll
          for (int w = 0; w < kSkWarps; ++w)
            M = fmaxf(M, reinterpret_cast<const float*>(S.work + (size_t)w * kWarpKvBytes)[kSkMC * kSkHD + i]);
          float L = 0.f, oa = 0.f, ob = 0.f;
#pragma unroll
          for (int w = 0; w < kSkWarps; ++w) {
            const float* cww = reinterpret_cast<const float*>(S.work + (size_t)w * kWarpKvBytes);
            const float mw = cww[kSkMC * kSkHD + i];
            const float f = mw == -INFINITY ? 0.f : __expf(mw - M);
            L += cww[kSkMC * kSkHD + kSkMC + i] * f;
            oa += cww[i * kSkHD + d2] * f;
            ob += cww[i * kSkHD + d2 + 1] * f;
          }
          float* pr = part + (size_t)(qt * kSkMC + i) * kSkPart;
          *reinterpret_cast<float2*>(pr + d2) = make_float2(oa, ob);
          if (d2 == 0) *reinterpret_cast<float2*>(pr + kSkHD) = make_float2(M, L);
        }
      }
      cbar();
    }
    if (tr) tpw = gtimer();
    // the last split of this (sequence, head) combines the splits in split order
    __threadfence();
    cbar();
    if (tid == 0) S.misc[3] = atomicAdd(a.cnt + b * H + h, 1) == splits - 1;
    cbar();
    if (S.misc[3]) {
      __threadfence();
      const int rows_ok = min(nrows, (int)a.apart_rows);
      const float* p0 = a.apart + ((size_t)b * H + h) * splits * a.apart_rows * kSkPart;
      for (int idx = tid; idx < rows_ok * (kSkHD / 2); idx += kSkWarps * 32) {
        const int i = idx / (kSkHD / 2), d2 = (idx - i * (kSkHD / 2)) * 2;
        // every split's (max, sum, output pair) in one batch of loads, then added in split order
        // with a running maximum (four splits per batch)
        float M = -INFINITY, L = 0.f, oa = 0.f, ob = 0.f;
        for (int s0 = 0; s0 < splits; s0 += 4) {
          float2 ml[4], ov[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            ml[j] = make_float2(-INFINITY, 0.f);
            ov[j] = make_float2(0.f, 0.f);
            if (s0 + j < splits) {
              const float* pr = p0 + ((size_t)(s0 + j) * a.apart_rows + i) * kSkPart;
              ml[j] = __ldcg(reinterpret_cast<const float2*>(pr + kSkHD));
              ov[j] = __ldcg(reinterpret_cast<const float2*>(pr + d2));
            }
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            if (ml[j].x == -INFINITY) continue;
            const float nm = fmaxf(M, ml[j].x);
            const float fo = M == -INFINITY ? 0.f : __expf(M - nm), fn = __expf(ml[j].x - nm);
            L = L * fo + ml[j].y * fn;
            oa = oa * fo + ov[j].x * fn;
            ob = ob * fo + ov[j].y * fn;
            M = nm;
          }
        }
        const float inv = L > 0.f ? 1.f / L : 0.f;
        uint32_t hi, lo;
        split2(oa * inv, ob * inv, hi, lo);
        const size_t o = (size_t)(rbeg + i) * ld + h * kSkHD + d2;
        *reinterpret_cast<uint32_t*>(a.thi + o) = hi;
        *reinterpret_cast<uint32_t*>(a.tlo + o) = lo;
      }
      if (tid == 0) a.cnt[b * H + h] = 0;
    }
    cbar();
    if (tr) {
      const unsigned k = atomicAdd(g_trace_n, 1u);
      if (k < g_trace_cap) {
        TraceRec rr{};
        rr.t0 = ti0;
        rr.tw = ti0;
        rr.t1 = gtimer();
        rr.tag = 130 + (S.misc[3] ? 1 : 0);
        rr.cta = c;
        rr.sm = 0;
        rr.mark[0] = tq ? (int)(tq - ti0) : 0;
        rr.mark[1] = tk ? (int)(tk - ti0) : 0;
        rr.mark[2] = (int)(tpw - ti0);
        g_trace_s[k] = rr;
      }
    }
  }
}

__global__ void __launch_bounds__(kSkThreads, 1) k_stack(StackArgs a) {
  extern __shared__ __align__(128) unsigned char sm[];
  Smem S;
  S.ring = reinterpret_cast<__nv_bfloat16*>(sm);
  S.work = sm + kRingBytes;
  S.red = reinterpret_cast<float*>(S.work + kWorkBytes);
  S.ss = S.red + kRedBytes / 4;
  S.rope = reinterpret_cast<float2*>(S.ss + kSsBytes / 4);
  unsigned char* tail = reinterpret_cast<unsigned char*>(S.rope) + kRopeBytes;
  S.full = reinterpret_cast<uint64_t*>(tail);
  S.empty = S.full + kSkSlots;
  S.sbar = S.empty + kSkSlots;
  S.inv = reinterpret_cast<float*>(S.sbar + 2);
  S.misc = reinterpret_cast<int*>(S.inv + 2 * kSkMC);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x, G = gridDim.x;
  const int KS = a.d < kSkKS ? a.d : kSkKS;
  const Shape z{a.d, a.F, KS, a.F / KS};
  unsigned long long t_start = 0;
  int M = *a.r.rows.M;
  M = M < 0 ? 0 : (M > a.r.M_cap ? a.r.M_cap : M);
  if (tid == 0) {
    for (int s = 0; s < kSkSlots; ++s) {
      mb_init(&S.full[s], 1);
      mb_init(&S.empty[s], 1);
    }
    mb_init(&S.sbar[0], 1);
    mb_init(&S.sbar[1], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    for (int i = 0; i < 8; ++i) S.misc[i] = 0;
    if (g_trace_s) t_start = gtimer();
  }
  // rows 0..7: sequence, cache slot and RoPE angles, for the Q/K/V epilogues (fixed for the launch)
  if (tid < kSkMC) {
    const bool ok = tid < M;
    S.misc[16 + tid] = ok ? a.r.rows.b[tid] : 0;
    S.misc[24 + tid] = ok ? a.r.rows.slot[tid] : 0;
    S.misc[40 + tid] = ok && a.r.pt ? a.r.rows.page[tid] : 0;
  }
  if (tid < kSkMC * (kSkHD / 2)) {
    const int r = tid / (kSkHD / 2), j = tid - r * (kSkHD / 2);
    S.rope[tid] = r < M ? a.rope[(size_t)a.r.rows.pos[r] * (kSkHD / 2) + j] : make_float2(1.f, 0.f);
  }
  __syncthreads();
  const int L = a.r.L;

  if (warp == kSkWarps) {
    // ---------------- copy warp: every unit of this CTA, block after block, phase after phase
    if (lane == 0) {
      int seq = 0;
      bool stop = false;
      for (int l = 0; l < L && !stop; ++l) {
        const StackLayer Ly = a.r.layers[l];
        for (int p = 0; p < PH_N && !stop; ++p) {
          for (int i = 0; i < kSkMaxUnits && !stop; ++i) {
            const int u = my_unit(z, l, p, c, G, i);
            if (u < 0) break;
            {
              const int s = seq % kSkSlots, use = seq / kSkSlots;
              if (use > 0) {
                bool ok = false;
                for (int n = 0; n < kSkSpins && !ok; ++n) {
                  ok = mb_try(&S.empty[s], (uint32_t)((use - 1) & 1));
                  if (!ok && (n & 1023) == 1023 && *(volatile int*)&S.misc[0]) break;
                }
                if (!ok) {
                  stop = true;
                  continue;
                }
              }
              int K;
              const __nv_bfloat16* W = unit_src(Ly, z, p, u, K);
              __nv_bfloat16* dst = S.ring + (size_t)s * kSkCols * kSkKP;
              mb_expect(&S.full[s], (uint32_t)(kSkCols * z.KS * 2));
              for (int col = 0; col < kSkCols; ++col)
                bulk_g2s(dst + (size_t)col * kSkKP, W + (size_t)col * K, (uint32_t)(z.KS * 2), &S.full[s]);
              ++seq;
              *(volatile int*)&S.misc[1] = seq;
            }
          }
        }
      }
      __threadfence_block();
      *(volatile int*)&S.misc[2] = 1;
    }
    return;
  }

  // ---------------- compute warps
  unsigned target = 0;
  int seq = 0;
  int uses[2] = {0, 0};
  unsigned long long tp = g_trace_s && tid == 0 ? gtimer() : 0;
  auto phase_end = [&](int ph, int l) { trace_phase(ph, l, tp); };
  auto phase_begin = [&]() {
    if (g_trace_s && tid == 0) tp = gtimer();
  };
  bool ok = true;
  if (L > 0) {
    const StackLayer L0 = a.r.layers[0];
    prologue(a, L0, c, G, M);
    phase_end(5, 0);
    ok = grid_sync(a, target, G, S);
    phase_begin();
  }
  for (int l = 0; l < L && ok; ++l) {
    const StackLayer Ly = a.r.layers[l];
    StackLayer Ln{};
    if (l + 1 < L) Ln = a.r.layers[l + 1];
    const StackLayer* Lnext = l + 1 < L ? &Ln : nullptr;
    if (l > 0) {
      if (!grid_sync(a, target, G, S)) break;
      phase_begin();
    }
    // the committed cache prefix of this CTA's attention items into L2 (it does not change in a step)
    if (tid < 32) {
      const int items = a.B * a.H * a.splits;
      for (int item = c; item < items; item += G) {
        const int b = item / (a.H * a.splits), h = (item / a.splits) % a.H, sp = item % a.splits;
        if (!a.r.stable || lane > 1) continue;
        int Sb = a.r.stable[(size_t)b * a.r.stable_stride] + a.r.stable_add;
        Sb = Sb < 0 ? 0 : (Sb > a.r.S ? a.r.S : Sb);
        int lo, hi;
        key_share(0, Sb, a.splits, sp, lo, hi);
        kv_prefetch_l2(cache_view(a, Ly), lane == 0 ? Ly.k : Ly.v, 2, a.H, kSkHD, b, h, lo, hi);
      }
    }
    linear_phase(a, Ly, Lnext, z, l, PH_QKV, c, G, M, seq, uses, S);
    phase_end(0, l);
    if (!grid_sync(a, target, G, S)) break;
    phase_begin();
    attention_phase(a, Ly, c, G, S);
    phase_end(1, l);
    if (!grid_sync(a, target, G, S)) break;
    phase_begin();
    linear_phase(a, Ly, Lnext, z, l, PH_WO, c, G, M, seq, uses, S);
    phase_end(2, l);
    if (!grid_sync(a, target, G, S)) break;
    phase_begin();
    linear_phase(a, Ly, Lnext, z, l, PH_W13, c, G, M, seq, uses, S);
    phase_end(3, l);
    if (!grid_sync(a, target, G, S)) break;
    phase_begin();
    linear_phase(a, Ly, Lnext, z, l, PH_W2, c, G, M, seq, uses, S);
    phase_end(4, l);
  }
  cbar();
  if (tid == 0) {
    // after a failure: wait (bounded) for the copy warp to stop, then for its copies in flight;
    // and the staging copies of the last fill of each buffer
    if (*(volatile int*)&S.misc[0]) {
      for (int n = 0; n < kSkSpins && !*(volatile int*)&S.misc[2]; ++n) {
      }
      const int issued = *(volatile int*)&S.misc[1];
      for (int q = seq; q < issued; ++q) mb_wait(&S.full[q % kSkSlots], (uint32_t)((q / kSkSlots) & 1));
    }
    for (int b = 0; b < 2; ++b)
      if (uses[b] > 0) mb_wait(&S.sbar[b], (uint32_t)((uses[b] - 1) & 1));
    // the last CTA to leave resets the barrier words for the next launch
    __threadfence();
    if (atomicAdd(a.bar + 1, 1u) == (unsigned)G - 1) {
      a.bar[0] = 0;
      a.bar[2] = 0;
      __threadfence();
      a.bar[1] = 0;
    }
    if (g_trace_s) {
      TraceRec r{};
      r.t0 = t_start;
      r.tw = t_start;
      r.t1 = gtimer();
      r.tag = TT_STACK;
      r.cta = c;
      r.sm = (int)smid();
      const unsigned i = atomicAdd(g_trace_n, 1u);
      if (i < g_trace_cap) g_trace_s[i] = r;
    }
  }
}

}  // namespace

void trace_set_stack(TraceRec* buf, unsigned* counter, unsigned cap) {
  cudaMemcpyToSymbol(g_trace_s, &buf, sizeof(buf));
  cudaMemcpyToSymbol(g_trace_n, &counter, sizeof(counter));
  cudaMemcpyToSymbol(g_trace_cap, &cap, sizeof(cap));
}

void stack_set_first_wait(int spins) {
  const int v = spins < 0 ? kSkSpins : spins;
  cudaMemcpyToSymbol(g_stack_first_wait, &v, sizeof(v));
}

void kernel_attrs_stack(Dev* D) {
  if (cudaFuncSetAttribute(k_stack, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes) != cudaSuccess) {
    D->persist = 0;
    return;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_stack, kSkThreads, kSmemBytes) != cudaSuccess ||
      per_sm < 1)
    D->persist = 0;
}

bool stack_ready(const Dev& D) { return D.persist && D.stk_enc != nullptr; }

bool launch_stack(const Dev& D, const StackRun& r, cudaStream_t s) {
  if (!stack_ready(D) || r.L <= 0 || !r.layers) return false;
  const int KS = D.d < kSkKS ? D.d : kSkKS;
  if (D.hd != kSkHD || D.d % kSkCols || D.d % KS || D.F % KS || D.d > kSkKS || KS % 16 ||
      D.d / kSkCols > kSkSsMax)
    return false;
  // every unit of a phase of one CTA fits the unit list, every W2 unit (F / KS slots) the ring
  const int G = D.stk_grid;
  const int most = std::max(std::max(3 * D.d, 2 * D.F) / kSkCols, D.d / kSkCols * (D.F / KS));
  if (G < 1 || (most + G - 1) / G > kSkMaxUnits || r.M_cap > D.R) return false;
  StackArgs a{};
  a.r = r;
  a.q = D.qbuf;
  a.apart = D.stk_apart;
  a.apart_rows = D.stk_apart_rows;
  a.cnt = D.stk_cnt;
  a.bar = D.stk_bar;
  a.ahi = D.stk_ahi;
  a.alo = D.stk_alo;
  a.thi = D.stk_thi;
  a.tlo = D.stk_tlo;
  a.mhi = D.stk_mhi;
  a.mlo = D.stk_mlo;
  a.ss = D.stk_ss;
  a.w2part = D.stk_w2part;
  a.w2cnt = D.stk_w2cnt;
  a.w2rows = D.R;
  a.rope = D.rope;
  a.err = D.err;
  a.d = D.d;
  a.H = D.H;
  a.F = D.F;
  a.B = D.B;
  a.splits = D.stk_splits;
  a.eps = D.eps;
  a.scale = D.scale;
  const double tb = 2.0;
  ProfScope ps(PK_LINEAR, (double)r.L * (4.0 * D.d * D.d + 3.0 * D.d * D.F) * tb, s);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(D.stk_grid);
  cfg.blockDim = dim3(kSkThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = s;
  cfg.attrs = nullptr;
  cfg.numAttrs = 0;
  ++g_launches;
  return cudaLaunchKernelEx(&cfg, k_stack, a) == cudaSuccess;
}

}  // namespace lca
