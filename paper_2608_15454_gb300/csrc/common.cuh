// Shared device-side types of the MBP decode step: model shape, workspace layout,
// per-sequence state and the launch wrappers each kernel file exports.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "lca.h"

namespace lca {

// ---------------------------------------------------------------- programmatic dependent launch
// Every kernel of the step is launched with programmatic stream serialization: it lets its
// successor launch at once (pdl_trigger), does only work that reads no upstream result (weight
// loads), and waits for its predecessor's completion (pdl_wait) before touching anything else.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// ---------------------------------------------------------------- optional launch trace
// When enabled, thread 0 of every CTA records (kernel tag, globaltimer at entry and exit) in a
// device buffer, so the timeline of the kernels inside a graph can be rebuilt on the host.
// The pointers are per translation unit (no relocatable device code); trace_set() fills them.
struct TraceRec {
  unsigned long long t0, t1, tw;  // entry, exit, grid-dependency wait returned
  int tag, cta, sm;
  int mark[3];  // optional mid-kernel times, ns after entry (0: none)
};
static_assert(sizeof(TraceRec) == 48, "trace record layout");
enum TraceTag : int {
  TT_GEMV = 1, TT_GEMV_F32, TT_GEMM, TT_ROWSTATS, TT_ATTN, TT_HEAD, TT_MB_PLAN, TT_MB_FILL,
  TT_MLP_PLAN, TT_VERIFY_PLAN, TT_SEGMENT, TT_LM_SCATTER, TT_NB_INPUT, TT_COMMIT, TT_LOOP_CTL,
  TT_OTHER, TT_UMMA, TT_SPLIT, TT_SGEMM, TT_STACK
};
static __device__ TraceRec* g_trace = nullptr;
static __device__ unsigned int* g_trace_n = nullptr;
static __device__ unsigned int g_trace_cap = 0;
__device__ __forceinline__ unsigned long long gtimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ unsigned smid() {
  unsigned r;
  asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
  return r;
}
struct TraceScope {
  unsigned long long t0, tw;
  int tag;
  unsigned mk[3];  // optional mid-kernel marks: nanoseconds after entry (0: none)
  bool on;
  __device__ __forceinline__ explicit TraceScope(int t) : t0(0), tw(0), tag(t), mk{0, 0, 0}, on(false) {
    if (threadIdx.x == 0 && threadIdx.y == 0 && g_trace) {
      on = true;
      t0 = gtimer();
      tw = t0;
    }
  }
  __device__ __forceinline__ void waited() {
    if (on) tw = gtimer();
  }
  __device__ __forceinline__ void mark(int i = 0) {
    if (on) mk[i] = (unsigned)(gtimer() - t0);
  }
  // a plain value (a row count, a chunk count) in a mark slot instead of a time
  __device__ __forceinline__ void value(int i, unsigned v) {
    if (on) mk[i] = v;
  }
  // a mark taken by another thread of the CTA (globaltimer value), handed over through shared memory
  __device__ __forceinline__ void mark_at(int i, unsigned long long t) {
    if (on && t > t0) mk[i] = (unsigned)(t - t0);
  }
  __device__ __forceinline__ ~TraceScope() {
    if (on) {
      const unsigned i = atomicAdd(g_trace_n, 1u);
      if (i < g_trace_cap) {
        TraceRec r;
        r.t0 = t0;
        r.t1 = gtimer();
        r.tw = tw;
        r.tag = tag;
        r.cta = (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
        r.sm = (int)smid();
        r.mark[0] = (int)mk[0];
        r.mark[1] = (int)mk[1];
        r.mark[2] = (int)mk[2];
        g_trace[i] = r;
      }
    }
  }
};
#define LCA_TRACE_SETTER(name)                                                         \
  void name(TraceRec* buf, unsigned* counter, unsigned cap) {                          \
    cudaMemcpyToSymbol(g_trace, &buf, sizeof(buf));                                    \
    cudaMemcpyToSymbol(g_trace_n, &counter, sizeof(counter));                          \
    cudaMemcpyToSymbol(g_trace_cap, &cap, sizeof(cap));                                \
  }
void trace_set_linear(TraceRec* buf, unsigned* counter, unsigned cap);
void trace_set_attn(TraceRec* buf, unsigned* counter, unsigned cap);
void trace_set_step(TraceRec* buf, unsigned* counter, unsigned cap);

constexpr int kVocab = 256;
constexpr int kMaxKSplit = 8;     // split-K ways of the skinny linear kernel
constexpr int kMaxAttnSplit = 16; // key-range splits of decode attention
constexpr int kAttnQT = 8;        // query rows per attention tile (decode)
constexpr int kStepLog = 1 << 16; // steps remembered by the per-step log

// device error word bits
constexpr int kErrIndex = 1;   // an index was out of range; the access was skipped
constexpr int kErrNumeric = 2; // non-finite logits
constexpr int kErrTimeout = 4; // a bounded wait ran out
constexpr int kErrPages = 8;   // a cache pool had no free page; the slots stayed unmapped
// which kernel family's wait ran out (set together with kErrTimeout; reported on stderr)
constexpr int kErrWaitAttn3 = 1 << 8, kErrWaitAttnMma = 1 << 9, kErrWaitGemv = 1 << 10, kErrWaitGemm = 1 << 11,
              kErrWaitAttnW = 1 << 13,
              kErrWaitGemvReduce = 1 << 12, kErrWaitStack = 1 << 14;

// Linear epilogues.
enum Epi : int {
  EPI_STORE = 0,      // y = acc
  EPI_RESID = 1,      // y = res + acc (res may alias y)
  EPI_SWIGLU = 2,     // packed rows (2j, 2j+1) = (W1_j, W3_j): y_j = silu(acc_2j) * acc_2j+1
  EPI_QKV = 3,        // packed rows [q | k | v]: RoPE on q and k, q -> y, k/v -> KV cache
  EPI_RESID_SILU = 4, // y = res + silu(acc) (MLP-MBP head layer)
};

// Per-row descriptors of one stack run. Row r belongs to sequence b[r], sits at RoPE
// position pos[r], writes its key/value to cache slot slot[r] and sees slots [0, kvlen[r]).
struct Rows {
  int* b;
  int* pos;
  int* slot;
  int* page;      // physical page of the row's cache slot (paged caches), written with slot
  int* kvlen;
  int* seq_start; // [B] first row of each sequence (rows of a sequence are contiguous)
  int* seq_count; // [B]
  int* M;         // total rows (device scalar)
};

// One KV-cache layer of the storage type. Paged (pt != nullptr): the layer is a pool of pages of
// kPage slots, [pages][H][kPage][hd]; slot s of sequence b lives in page pt[b * pt_ld + s / kPage]
// (-1: not mapped). Contiguous (pt == nullptr, the standalone attention op): [B][H][S][hd].
constexpr int kPage = 64;
struct KV {
  void* k;
  void* v;
  int S; // logical slots per (b, h)
  // host copies of the TMA tensor maps of K and V (bf16, head_dim 64: 64-key x 64-dim boxes with
  // the 128-byte swizzle, over [pages * H * kPage][64] rows when paged), or nullptr; used by the
  // tensor-core decode attention
  const void* tmaps;
  const int* pt;  // page table [B][pt_ld], or nullptr
  int pt_ld;
  int pages;      // pages of the pool (paged)
};
// Element offset of (sequence b, head h, slot s) when slot s lies in physical page pg (paged; the
// caller checked pg) or in the contiguous layout (pg ignored).
__device__ __forceinline__ size_t kv_addr(const KV& kv, int H, int hd, int b, int h, int s, int pg) {
  if (!kv.pt) return (((size_t)b * H + h) * kv.S + s) * hd;
  return (((size_t)pg * H + h) * kPage + (s & (kPage - 1))) * hd;
}
// A cache write of slot s in page pg is in range (the writers take pg from the row's page).
__device__ __forceinline__ bool kv_write_ok(const KV& kv, int s, int pg) {
  return s >= 0 && s < kv.S && (!kv.pt || (pg >= 0 && pg < kv.pages));
}
// Page of slot s of sequence b from the table, read through L2 (the decode steps' plan kernels
// map pages while the readers of an earlier launch may still run); an unmapped or out-of-range
// entry (or a slot past the table) reads page 0, whose keys the callers mask. 0 for the contiguous
// layout.
__device__ __forceinline__ int kv_page_cg(const KV& kv, int b, int s) {
  if (!kv.pt || s < 0 || s / kPage >= kv.pt_ld) return 0;
  const int pg = __ldcg(kv.pt + (size_t)b * kv.pt_ld + s / kPage);
  return (pg < 0 || pg >= kv.pages) ? 0 : pg;
}
// Element offset of (b, h, s), looking the page up.
__device__ __forceinline__ size_t kv_off(const KV& kv, int H, int hd, int b, int h, int s) {
  return kv_addr(kv, H, hd, b, h, s, kv_page_cg(kv, b, s));
}
// The page table row of sequence b into shared memory, in two halves so that the loads overlap the
// caller's other loads: kv_pages_load issues this thread's first entry (tid < pt_ld), the caller
// issues its own loads, then kv_pages_store writes that entry and loads and writes the rest of the
// row (pt_ld entries, checked as kv_page_cg does). Nothing for the contiguous layout. The caller
// synchronises before the first use.
__device__ __forceinline__ int kv_pages_load(const KV& kv, int b, int tid) {
  return (kv.pt && tid < kv.pt_ld) ? __ldcg(kv.pt + (size_t)b * kv.pt_ld + tid) : 0;
}
__device__ __forceinline__ void kv_pages_store(const KV& kv, int b, int* s_pt, int tid, int nthreads, int first) {
  if (!kv.pt) return;
  if (tid < kv.pt_ld) s_pt[tid] = (first < 0 || first >= kv.pages) ? 0 : first;
  for (int i = tid + nthreads; i < kv.pt_ld; i += nthreads) {
    const int pg = __ldcg(kv.pt + (size_t)b * kv.pt_ld + i);
    s_pt[i] = (pg < 0 || pg >= kv.pages) ? 0 : pg;
  }
}
// Shared-memory bytes of a staged page table row (16-byte multiple).
inline size_t kv_pages_smem(const KV& kv) { return kv.pt ? ((size_t)kv.pt_ld * 4 + 15) / 16 * 16 : 0; }
// The most page-table entries a reader stages (slots per sequence and cache: kMaxPtRow * kPage).
constexpr int kMaxPtRow = 2048;
// L2 prefetch (a hint) of slots [lo, hi) of (b, h) of one cache tensor (base: kv.k or kv.v, elements
// of es bytes): one bulk prefetch per page, the table entries of up to eight pages loaded before
// their prefetches are issued.
__device__ __forceinline__ void kv_prefetch_l2(const KV& kv, const void* base, int es, int H, int hd, int b, int h,
                                               int lo, int hi) {
  const char* p = static_cast<const char*>(base);
  if (!kv.pt) {
    if (hi > lo) {
      const uint32_t bytes = (uint32_t)((size_t)(hi - lo) * hd * es) & ~15u;
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p + kv_addr(kv, H, hd, b, h, lo, 0) * es),
                   "r"(bytes)
                   : "memory");
    }
    return;
  }
  for (int s0 = lo & ~(kPage - 1); s0 < hi; s0 += 8 * kPage) {
    int pg[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) pg[i] = s0 + i * kPage < hi ? kv_page_cg(kv, b, s0 + i * kPage) : 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int a = max(lo, s0 + i * kPage), e = min(hi, s0 + (i + 1) * kPage);
      if (a < e) {
        const uint32_t bytes = (uint32_t)((e - a) * hd * es) & ~15u;
        if (bytes)
          asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p + kv_addr(kv, H, hd, b, h, a, pg[i]) * es),
                       "r"(bytes)
                       : "memory");
      }
    }
  }
}

struct EpiArgs {
  int mode;
  float* y;
  int ldy;
  const float* res;
  int ldres;
  // EPI_QKV
  KV kv;
  Rows rows;
  const float2* rope; // [slots][hd/2] (cos, sin)
  int H, hd, d;
  int* err;
  // Split on write, for a tensor-core consumer of this output (sp_hi == nullptr: none). Each output
  // value v (after the residual add or the SwiGLU) is stored once more as bf16 halves of v * sg[c]
  // (sg: the consumer's RMSNorm gain, nullptr: 1) at sp_hi / sp_lo[row * ldsp + c], and, when ss is
  // set, the sum of v^2 over each 32-column block c / 32 at ss[row * ss_ld + c / 32] (the consumer's
  // RMS; a weight-streaming GEMV producer writes per 16-column block instead, for a GEMV
  // consumer). sp_only: the fp32 output is not written (the consumer is its only reader).
  __nv_bfloat16* sp_hi;
  __nv_bfloat16* sp_lo;
  int ldsp;
  const float* sg;
  float* ss;
  int ss_ld;
  int sp_only;
};

// Per-sequence committed state.
struct SeqState {
  int t;          // committed bytes
  int K;          // committed latents
  int open_start; // first byte of the open segment
  int mb_start;   // first byte of the window the MB cache holds (-1: empty)
  int mb_len;     // cached MB rows from mb_start
  int next_c1;    // next-byte argmax at t-1
  int generated;  // bytes generated in the current lca_generate
  int budget;     // generation budget (lca_generate); INT_MAX for single steps
  int done;       // budget reached
  int active;     // sequence exists (b < batch of the last prefill)
  int pad[6];
};

// Per-call parameters, copied to the device before each launch.
struct Params {
  int n;
  float tau;
  int accept;       // LCA_THRESH | LCA_SPEC
  int gen;          // 1 inside lca_generate: budgets apply
  int force_accept; // 1: this step uses forced_a
  int force_cand;   // 1: this step uses forced_cand
  int batch;
  int iter;         // generate: steps run
  int max_iter;     // generate: hard cap on steps
  int pad[7];
};

// Counters of work done, for algorithmic-byte accounting.
struct Stats {
  unsigned long long steps;     // decode steps run
  unsigned long long lm_steps;  // steps in which the LM module ran
  unsigned long long lm_rows;   // LM rows (new latents, committed or not)
  unsigned long long mb_rows;   // multi-byte window rows computed
  unsigned long long committed; // bytes committed
  unsigned long long pad[3];
};

// Kernels launched by this thread's wrappers (counted at capture time).
extern thread_local long long g_launches;

// Optional per-launch timing hook (eager steps only): the wrappers bracket each launch with
// begin/end so the runtime can record CUDA events on the launching stream.
enum ProfKind { PK_LINEAR = 0, PK_ATTN = 1, PK_HEAD = 2, PK_GLUE = 3, PK_COUNT = 4 };
struct ProfHook {
  virtual void begin(int kind, double bytes, cudaStream_t s) = 0;
  virtual void end(cudaStream_t s) = 0;
};
extern thread_local ProfHook* g_prof;
struct ProfScope {
  cudaStream_t s;
  bool on;
  ProfScope(int kind, double bytes, cudaStream_t s_) : s(s_), on(g_prof != nullptr) {
    if (on) g_prof->begin(kind, bytes, s);
  }
  ~ProfScope() {
    if (on) g_prof->end(s);
  }
};

struct StackLayer;

// Workspace layout (device pointers into the caller's workspace).
struct Dev {
  // shape
  int d, H, hd, F, n_enc, n_lm, n_nb, n_mb, mb_kind, n_mlp_heads, dtype;
  int B, S, L, NMAX, R; // batch cap, byte slots, latent slots, max n, row cap
  int boundary;
  float eps, scale;
  int num_sms;  // streaming multiprocessors of the device
  int use_tma;  // bf16 linear layers use the bulk-copy weight pipeline
  int attn_split_cap;  // largest cluster (key split) of decode attention
  int tiled_min_rows;  // layers with more typical rows than this run on the tensor cores
  int attn_pipe;       // decode attention: 2 = tensor cores (bf16, head_dim 64), 1 = bulk-copy pipelined
                       // CUDA-core kernel, 0 = register-tiled kernel
  int attn_ns;         // ring stages of the tensor-core prefill attention (4 or 8)
  int attn_ns_t;       // ring stages of the tensor-core decode attention (4, 8 or 12; half as many compute warps)
  int attn_tc_min;     // fewest (sequence, head) pairs for the tensor-core attention kernels
  int gemv_ks_big, gemv_ks_small;  // K-split of the weight-streaming GEMV (K >= 2048, K < 2048)
  int attn_min_keys;   // fewest cache keys per key split of a decode attention launch
  int attn_t;          // decode steps use the transposed tensor-core attention (8-row query tiles)
  int attn_w;          // small-batch decode steps use the warp-walk attention
  int split_write;     // tensor-core layers split their successor's input in their epilogue
  int sgemm_max_rows;  // tensor-core layers with at most this many typical rows use the skinny
                       // (weights-as-M) GEMM; 0: never
  int sgemm_max_ks;    // largest K split (cluster size) of the skinny GEMM (8, or 16 where the
                       // GPU schedules 16-CTA clusters of it)
  int use_umma;        // many-row bf16 layers run on the tensor cores (tcgen05)

  // paged KV caches: page tables [B][pt_ld_*] of the byte modules (encoder and next-byte decoder
  // share positions), the LM module and the multi-byte window; pool sizes in pages; bump
  // allocators ([0] bytes, [1] LM, [2] window)
  int* pt_byte;
  int* pt_lm;
  int* pt_mb;
  int pt_ld_byte, pt_ld_lm, pt_ld_mb;
  int pages_byte, pages_lm, pages_mb;
  int* pool_next;

  // weights (storage type; norms and bos fp32)
  void* embed;   // [256][d]
  void* unembed; // [256][d]
  const float* bos;
  const float* nb_norm;
  const float* mb_norm;
  void* mlp_w; // [heads][n_mb][d][d]

  // per-sequence state
  SeqState* seq;
  int* gstart;     // [B][L]  gstart[b][g] = first byte of latent group g
  float* h_store;  // [B][S][d] encoder output of committed (and candidate) bytes
  float* u_tab;    // [B][L][d] LM inputs u_0 = BOS, u_k = z_k
  float* o_tab;    // [B][L][d] LM outputs
  float* y_last;   // [B][d] next-byte hidden at t-1 (MLP head input)
  int* kpos;       // [B][S] K(p) of committed positions (prefill scratch)
  // activations of a tensor-core layer split into two bf16 halves (x * g = hi + lo), in two
  // buffers that consecutive layers alternate between (a layer reads one while its epilogue
  // writes the next layer's input into the other): [2][as_rows][up to F]; written by
  // k_split_rows or by the producing layer's epilogue and read by TMA in k_tgemm. as_ss: sums of
  // squares of the rows for the RMSNorm, [as_rows][as_ss_ld] (per 32-column block, or the whole
  // row in slot 0)
  __nv_bfloat16* as_hi[2];
  __nv_bfloat16* as_lo[2];
  float* as_ss;
  int as_ss_ld;
  // sums of squares per 16-column block of split rows written by GEMV epilogues, [as_rows][d / 16]
  float* gv_ss;
  int gv_ss_ld;
  int gemv_split;  // GEMV layers take pre-split inputs from GEMV producers (1) or stage fp32 rows (0)
  int as_rows;

  // rows
  float* x_mb;
  float* x_enc;
  float* x_lm;
  float* x_nb;
  float* qbuf; // [R][d]
  float* att;  // [R][d]
  float* mid;  // [R][F]
  float* xnorm; // [R][max(d,F)] normalised rows for the tiled GEMM
  Rows r_mb, r_v, r_lm;

  // heads
  int* head_rows_mb; // [B*NMAX] row (into x_mb or x_mlp) of each draft, order b*(n-1)+j
  int* head_rows_v;  // [B*NMAX]
  int* M_head_mb;
  int* M_head_v;
  float* mb_logits; // [B*NMAX][256]
  float* nb_logits; // [B*NMAX][256]
  int* mb_arg;
  float* mb_prob;
  int* nb_arg;
  float* nb_prob;

  // candidates and outputs
  int* cand;      // [B][NMAX]
  int* kc;        // [B][NMAX] K(p) of candidate rows
  uint8_t* out_step; // [B][NMAX]
  int* out_cnt;      // [B]
  uint8_t* out_gen;  // [B][S]
  int* hist;         // [NMAX]
  int* forced_a;     // [B]
  int* forced_cand;  // [B][NMAX]
  Params* params;
  int* err;
  Stats* stats;
  uint8_t* step_log; // [kStepLog] whether step s ran the LM module, at s % kStepLog

  // scratch
  float* lin_part; // split-K partials
  size_t lin_part_floats;
  int* lin_cnt;    // split-K tile counters
  int* head_cnt;   // head row-tile counters
  float* attn_part; // attention split partials
  int* attn_cnt;
  float* inv_rms;  // [R]
  float2* rope;    // [max(S,L)][hd/2]
  int rope_slots;

  // persistent stack kernel (bf16, head_dim 64, d <= 1024): layer tables, attention partials and
  // counters, grid-barrier words; persist = 0 turns it off
  int persist;
  int stk_grid;        // CTAs of a launch (one per SM)
  int stk_splits;      // attention key splits per (sequence, head)
  StackLayer* stk_enc;
  StackLayer* stk_lm;
  StackLayer* stk_nb;
  StackLayer* stk_mb;
  float* stk_apart;    // [B][H][splits][rows of a sequence][68]
  size_t stk_apart_rows;  // rows per (sequence, head, split) the partial buffer holds
  int* stk_cnt;        // [B * H] last-arriver counters of the attention combine
  unsigned* stk_bar;   // [4]: grid-barrier arrivals, exits, abort
  // inputs of the stack kernel's linear phases, written already split by the producing phase:
  // bf16 halves (v = hi + lo) of the normalised-input rows x * g [R][d], of the attention output
  // [R][d] and of the SwiGLU output [R][F]; per-row sums of squares of x per 16-column tile [R][d/16]
  __nv_bfloat16 *stk_ahi, *stk_alo, *stk_thi, *stk_tlo, *stk_mhi, *stk_mlo;
  float* stk_ss;
  float* stk_w2part;   // [F / KS][R][d] W2 partial sums per K-slice
  int* stk_w2cnt;      // [d / 16] last-arriver counters of W2's column tiles
};

// One block of a stack as the persistent stack kernel reads it (device array, filled at create).
struct StackLayer {
  const __nv_bfloat16* wqkv; // [3d][d]
  const __nv_bfloat16* wo;   // [d][d]
  const __nv_bfloat16* w13;  // [2F][d], rows interleaved (W1_j, W3_j)
  const __nv_bfloat16* w2;   // [d][F]
  const float* attn_norm;
  const float* mlp_norm;
  void* k;                   // KV cache layer: a pool of pages [pages][H][kPage][64] bf16
  void* v;
};

// A stack run by the persistent kernel (kernels_stack.cu).
struct StackRun {
  const StackLayer* layers; // device [L]
  int L;
  float* x;                 // residual stream rows (in place)
  Rows rows;
  int M_cap;
  int S;                    // cache slots per (sequence, head)
  const int* pt;            // the layers' page table [B][pt_ld] (pools of pages [pages][H][kPage][64])
  int pt_ld, pages;
  const int* stable;        // per-sequence committed cache length (stride in ints), or nullptr
  int stable_stride;
  int stable_add;
};
bool stack_ready(const Dev& D);
// Runs the whole stack as one launch; false if the persistent kernel cannot run this stack.
bool launch_stack(const Dev& D, const StackRun& r, cudaStream_t s);
void kernel_attrs_stack(Dev* D);
void stack_set_first_wait(int spins);  // test hook (see lca_debug_set_wait_spins)
void trace_set_stack(TraceRec* buf, unsigned* counter, unsigned cap);

struct Block {
  const float* attn_norm;
  const float* mlp_norm;
  void* wqkv; // [3d][d]
  void* wo;   // [d][d]
  void* w13;  // [2F][d], rows interleaved (W1_j, W3_j)
  void* w2;   // [d][F]
  KV kv;
};

// ---------------------------------------------------------------- launch wrappers
// Linear y = epi(norm?(x) . W^T) over the rows [0, *M) of x, groups along W (grouped GEMM).
struct LinearArgs {
  const float* x;
  int ldx;
  const void* W; // [groups][N][Kd]
  int N, Kd;
  int groups;    // row groups share nothing; group g uses W + g*N*Kd and rows g*Mg..
  int Mg_stride; // rows per group (groups > 1)
  const float* norm; // RMSNorm gain or nullptr
  float eps;
  const int* M;  // device row count (per group when groups > 1)
  int M_cap;     // host upper bound of *M
  EpiArgs epi;
  // weights of the next linear layer(s), prefetched into L2 by this launch's CTAs before the
  // grid-dependency wait (nullptr: none)
  const void* pf[2];
  size_t pf_bytes[2];
  int rows_typ;  // typical row count (sizes the activation staging); 0: M_cap
  const void* tmap;  // host copy of the weight's TMA tensor map (tensor-core path), or nullptr
  // host copies of the TMA tensor maps of the split activations (hi, lo) of buffer abuf for this
  // Kd, or nullptr (then the layer runs on the CUDA cores)
  const void* amap;
  int abuf;      // split buffer (0 or 1) the tensor-core path reads
  int presplit;  // the producing layer's epilogue already wrote the split input and its sums of
                 // squares per 32-column block; otherwise k_split_rows runs first
  // Weight-streaming GEMV only: the producing layer's epilogue wrote this layer's input as bf16
  // halves of x * g (g: this layer's RMSNorm gain, or 1) into split buffer abuf, [rows][Kd], and,
  // with a norm, the sums of x^2 per 16-column block into Dev::gv_ss; the rows are then staged by
  // bulk copies. The launcher fills ghi, glo, gss, gss_ld from the workspace.
  int gsplit;
  const __nv_bfloat16* ghi;
  const __nv_bfloat16* glo;
  const float* gss;
  int gss_ld;
};
// Whether a bf16 layer without tiling runs on the bulk-copy GEMV (k_gemv_bulk), and its K-split.
bool gemv_bulk_ok(const Dev& D, const LinearArgs& a);
int gemv_bulk_ksplit(const Dev& D, const LinearArgs& a);
void linear(const Dev& D, const LinearArgs& a, bool tiled, cudaStream_t s);
bool linear_umma(const Dev& D, const LinearArgs& a, cudaStream_t s);
// whether linear() runs this layer on the tensor cores when called with tiled = true
bool umma_ready(const Dev& D, const LinearArgs& a);
int make_weight_tmap(void* out, const void* W, long long rows, long long K);
// TMA tensor maps of split activations [rows][K] bf16, 128 bytes each, K boxes of 64: (hi, lo) with
// 128-row boxes, then (hi, lo) with 32-row boxes, then (hi, lo) with 64-row boxes
constexpr int kSplitMapBytes = 768;
int make_split_tmaps(void* out, const void* hi, const void* lo, long long rows, long long K);
// TMA tensor maps (K then V, 128 bytes each) of one bf16 KV-cache layer [rows][64], 64 x 64 boxes
int make_kv_tmaps(void* out, const void* k, const void* v, long long rows);
void kernel_attrs_umma(Dev* D);
void trace_set_umma(TraceRec* buf, unsigned* counter, unsigned cap);

size_t attention_scratch_floats(int B, int H, int hd);
size_t attention_counters(int B, int H);
void kernel_attrs_linear();
void kernel_attrs_step();
void kernel_attrs_attn();
// Attention of query rows over a KV-cache layer (keys [0, kvlen[r]) of sequence b[r]).
// stable: optional per-sequence committed length (stride in ints) whose cache prefix (the first
// stable + stable_add slots) does not change during a step: the warp-walk decode kernel stages it
// in shared memory before the dependency wait; rows_seq: the most query rows a sequence has (a
// tile-size hint).
// osh/osl: also store the output as bf16 halves there (same [rows][H * hd] layout), the pre-split
// input of a weight-streaming GEMV; only where attention_split_out holds for these arguments.
void attention(const Dev& D, const float* q, float* out, const KV& kv, const Rows& rows, int B,
               int qtiles_grid, int splits, cudaStream_t s, const int* stable = nullptr,
               bool short_kv = false, int stable_add = 0, int rows_seq = kAttnQT, __nv_bfloat16* osh = nullptr,
               __nv_bfloat16* osl = nullptr);
bool attention_split_out(const Dev& D, const KV& kv, int B, int qtiles_grid, bool short_kv);

// Step / prefill glue kernels (kernels_step.cu).
void launch_mb_plan(const Dev& D, cudaStream_t s);
void launch_mb_fill(const Dev& D, cudaStream_t s);
void launch_mlp_plan(const Dev& D, cudaStream_t s);
void launch_head(const Dev& D, const float* x, const int* rows, const int* M, int M_cap,
                 const float* norm, float* logits, int* arg, float* prob, cudaStream_t s);
void launch_verify_plan(const Dev& D, cudaStream_t s);
void launch_segment(const Dev& D, cudaGraphConditionalHandle h, int use_handle, cudaStream_t s);
void launch_lm_scatter(const Dev& D, cudaStream_t s);
void launch_nb_input(const Dev& D, cudaStream_t s);
void launch_commit(const Dev& D, cudaStream_t s);
void launch_loop_ctl(const Dev& D, cudaGraphConditionalHandle h, cudaStream_t s);
void launch_gen_init(const Dev& D, int max_new, cudaStream_t s);
void launch_rope_table(const Dev& D, float base, cudaStream_t s);
void launch_pack_rows(void* dst, const void* src, int rows, int cols, int dst_row0, int row_step,
                      int elem_bytes, cudaStream_t s);

// prefill
void launch_prefill_embed(const Dev& D, const uint8_t* bytes, int M, cudaStream_t s);
void launch_prefill_segment(const Dev& D, const uint8_t* bytes, const int* row0, const int* lens,
                            int batch, const int* lm_row0, cudaStream_t s);
void launch_prefill_pool(const Dev& D, const int* row0, const int* lens, const int* lm_row0,
                         int batch, int max_lat, cudaStream_t s);
void launch_prefill_nb_input(const Dev& D, int M, cudaStream_t s);
void launch_prefill_finish(const Dev& D, const int* row0, const int* lens, const int* lm_row0,
                           int batch, cudaStream_t s);

} // namespace lca
