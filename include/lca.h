/*
 * lca.h - C ABI of the GB300 multi-byte-prediction (MBP) decode step of a byte-level
 * hierarchical language model with a Latent-Causal-Attention (LCA) multi-byte head
 * ("Dynamic Multi-Byte Prediction With Hierarchical Language Models").
 *
 * One decode step (Algorithm 1, one iteration of its loop) does, per sequence:
 *   (1) draft n-1 bytes with the multi-byte head over the previous and current latent
 *       group (Algorithm 1, drafting step; Section 3), or with independent MLP heads
 *       (MLP-MBP, Section 4.1);
 *   (2) embed the n candidates (next-byte byte c_1 plus the drafts) and run the encoder
 *       module (Section 2.2 "Encoder Module") with its byte KV cache;
 *   (3) split at space boundaries, mean-pool closed segments and run the LM module over
 *       the new latents with its KV cache, only when a segment closes (Algorithm 1
 *       LM-module branch; Eff-FxT rule, Section 4.1);
 *   (4) run the next-byte decoder over all n candidates (Algorithm 1, next-byte step);
 *   (5) accept: c_1 always, drafts left to right while their probability is >= tau
 *       (Section 3.1 "Byte Acceptance"; LCA_THRESH), or while they equal the next-byte
 *       argmax (speculative acceptance, Section 6.2 (ii); LCA_SPEC); then keep the
 *       accepted prefix of every cache and drop the rest.
 * The meaning of n used here: one next-byte byte plus n-1 drafts, so 1..n bytes are
 * committed per step (the algorithm's "n-2 copies" and "h_2[-(n-1):]").
 *
 * Conventions
 *   Status: every call returns LCA_OK (0) or a negative LCA_E_* code; lca_status_str
 *     names it. After an error the context stays valid for lca_destroy and lca_prefill.
 *   Ownership: the caller owns the weights, the workspace, the stream and all host
 *     buffers; the library keeps the workspace and stream pointers until lca_destroy
 *     and never frees them. Weights are copied (repacked) into the workspace by
 *     lca_create and need not outlive it.
 *   Memory: all device memory the library uses lies in the caller's workspace.
 *   Sync: lca_prefill, lca_mbp_step, lca_generate and the debug calls return after the
 *     stream has finished their work. lca_generate_async only enqueues.
 *   Threads: no global state; one context is used by one host thread at a time.
 */
#ifndef LCA_H
#define LCA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* status codes */
#define LCA_OK 0
#define LCA_E_ARG (-1)          /* bad pointer, size or enum value */
#define LCA_E_CAPACITY (-2)     /* batch > max_batch, n outside 1..max_n, or bytes > max_bytes */
#define LCA_E_WEIGHTS (-3)      /* a weight tensor is missing or has the wrong size or dtype */
#define LCA_E_CUDA (-4)         /* a CUDA runtime call failed */
#define LCA_E_DEVICE_STATE (-5) /* a kernel found an index out of range and skipped it */
#define LCA_E_NUMERIC (-6)      /* non-finite logits were produced */
#define LCA_E_TIMEOUT (-7)      /* a bounded device wait ran out */
#define LCA_E_STATE (-8)        /* call order: e.g. a step before any prefill */

/* storage types (weights, KV caches); activations are always fp32 */
#define LCA_F32 0
#define LCA_BF16 1

/* multi-byte head kind */
#define LCA_MB_LCA 0 /* transformer blocks with the LCA mask (Section 3) */
#define LCA_MB_MLP 1 /* independent residual-SiLU MLP heads on the last next-byte state */

/* acceptance rule */
#define LCA_THRESH 0 /* draft kept while its drafter probability >= tau (Section 3.1) */
#define LCA_SPEC 1   /* draft kept while it equals the next-byte argmax (Section 6.2) */

typedef struct lca_ctx lca_ctx; /* opaque, owned by the library */

/* Model shape and capacity. All fields are read; none is inferred. */
typedef struct {
  int32_t d_model, n_heads, head_dim, d_ff, vocab; /* vocab must be 256 */
  int32_t n_enc, n_lm, n_nb, n_mb; /* blocks per module; MLP head: residual layers per head */
  int32_t mb_kind;                 /* LCA_MB_LCA | LCA_MB_MLP */
  int32_t n_mlp_heads;             /* MLP head only: heads (>= max_n - 1) */
  int32_t boundary_byte;           /* byte that ends a segment (0x20) */
  float rope_base, rms_eps, attn_scale; /* 1e5, 1e-6, 1/sqrt(head_dim) (Section 4.2) */
  int32_t dtype;                   /* LCA_F32 | LCA_BF16 */
  int32_t max_batch, max_bytes, max_n; /* max_bytes bounds prompt + generated + max_n */
  /* Paged KV caches: every cache layer is a pool of pages of 64 slots, [pages][n_heads][64]
   * [head_dim], and each sequence maps its slots to pages through a page table (one per module
   * kind, shared by that module's layers). kv_pages: pages of each encoder and next-byte layer's
   * pool (byte positions); lm_pages: of each LM-module layer's pool (latents); mb_pages: of each
   * multi-byte layer's pool (window rows). 0: enough for every sequence at max_bytes positions
   * (max_bytes + 1 latents). The prefill maps the prompts' pages (LCA_E_CAPACITY if they do not
   * fit); a decode step maps a page when a sequence's positions, latents or window first reach it,
   * from a bump counter, and a page stays mapped until the next prefill. A step that finds a pool
   * exhausted leaves those slots unwritten and returns LCA_E_CAPACITY; its results are then
   * undefined until the next prefill. max_bytes must stay below 131,072. */
  int32_t kv_pages, lm_pages, mb_pages;
} lca_config;

/* One named weight tensor: device pointer, element count, LCA_F32|LCA_BF16.
 * Names (l = layer index, j = MLP head): "embed" [256,d]; "{enc,lm,nb,mb}.{l}.attn_norm"
 * [d], ".wq" ".wk" ".wv" ".wo" [d,d], ".mlp_norm" [d], ".w1" ".w3" [d_ff,d], ".w2" [d,d_ff];
 * "lm.bos" [d]; "nb.norm" [d]; "mb.norm" [d]; "mlp.{j}.{l}.w" [d,d]; "unembed" [256,d].
 * Linear weights are [out, in] row-major. Norm gains and lm.bos are LCA_F32; every
 * other tensor has the config dtype. */
typedef struct {
  const char* name;
  const void* ptr;
  int64_t numel;
  int32_t dtype;
} lca_tensor;

/* Committed state of one sequence. */
typedef struct {
  int32_t t;                /* committed bytes */
  int32_t K;                /* committed latents (closed segments) */
  int32_t open_start;       /* first byte of the open segment */
  int32_t prev_group_start; /* first byte of latent group K-1, or -1 when K == 0 */
  int32_t group_start;      /* first byte of latent group K */
  int32_t next_byte;        /* next-byte argmax at position t-1 (the next c_1) */
  int32_t generated;        /* bytes generated by the last lca_generate */
  int32_t pad;
} lca_seq_state;

/* Counters since lca_create (for throughput and algorithmic-byte accounting). */
typedef struct {
  int64_t steps;              /* decode steps run */
  int64_t lm_steps;           /* steps in which the LM module ran (a candidate closed a segment) */
  int64_t lm_rows;            /* latents the LM module processed (accepted or rolled back) */
  int64_t mb_rows;            /* multi-byte window rows computed */
  int64_t committed;          /* bytes committed */
  int64_t kernels_per_step;   /* kernels one step graph of the last n launches, LM aside */
  int64_t kernels_per_lm_run; /* kernels of the LM module when it runs */
  int64_t workspace_bytes;
} lca_stats;

/* Bytes of device workspace a context with this config needs (out). */
int lca_workspace_bytes(const lca_config* cfg, size_t* out);

/* Create a context. workspace: device memory of >= lca_workspace_bytes, 256-byte aligned,
 * caller-owned. stream: cudaStream_t the library enqueues on (caller-owned; 0 = legacy).
 * Copies and repacks the n_weights tensors into the workspace. */
int lca_create(const lca_config* cfg, const lca_tensor* weights, int n_weights, void* workspace,
               size_t workspace_bytes, void* stream, lca_ctx** out);

/* Start `batch` sequences from host prompts (prompts[b]: lens[b] >= 1 bytes). Runs the whole
 * forward over the prompts (filling every cache) and the next-byte head at the last byte. */
int lca_prefill(lca_ctx* ctx, int32_t batch, const uint8_t* const* prompts, const int32_t* lens);

/* One MBP decode step (Algorithm 1, one loop iteration) for every sequence.
 * out_bytes: host [batch * n], row b holds the committed bytes of sequence b;
 * out_counts: host [batch], committed bytes 1..n. Either may be NULL. */
int lca_mbp_step(lca_ctx* ctx, int32_t n, float tau, int32_t accept_mode, uint8_t* out_bytes,
                 int32_t* out_counts);

/* lca_mbp_step without outputs: enqueue one step on the stream and return at once. The
 * committed state is readable afterwards through lca_debug_state. */
int lca_mbp_step_async(lca_ctx* ctx, int32_t n, float tau, int32_t accept_mode);

/* Decode until every sequence has max_new more bytes (the last step is cut to the budget),
 * as one device-side loop without host round trips. out: host [batch * max_new];
 * out_len: host [batch] (= max_new); accepted_hist: host [n], steps by accepted drafts,
 * summed over sequences. Any output pointer may be NULL. */
int lca_generate(lca_ctx* ctx, int32_t n, float tau, int32_t accept_mode, int32_t max_new,
                 uint8_t* out, int32_t* out_len, int32_t* accepted_hist);

/* lca_generate split in two: enqueue the loop on the stream and return at once; then wait
 * and copy the results. Between the two the caller may record events on the stream. */
int lca_generate_async(lca_ctx* ctx, int32_t n, float tau, int32_t accept_mode, int32_t max_new);
int lca_generate_fetch(lca_ctx* ctx, uint8_t* out, int32_t* out_len, int32_t* accepted_hist);

/* Debug and test hooks. */
int lca_debug_state(lca_ctx* ctx, int32_t b, lca_seq_state* out);
int lca_debug_stats(lca_ctx* ctx, lca_stats* out);

/* Per-step log: out[i] = 1 if decode step first + i (counted from lca_create, as lca_stats.steps)
 * ran the LM module, else 0. The last 65,536 steps are kept; older or future steps: LCA_E_ARG. */
int lca_debug_step_log(lca_ctx* ctx, int64_t first, int32_t count, uint8_t* out);
/* Accepted-draft histogram of the steps since the last reset: out host [max_n], out[a] = steps
 * (summed over sequences) that accepted a drafts; reset != 0 zeroes it afterwards. lca_generate
 * also zeroes it when it starts. */
int lca_debug_accept_hist(lca_ctx* ctx, int32_t* out, int32_t reset);
/* Page table of one cache kind (cache: 0 byte positions of the encoder and next-byte layers, 1 LM
 * latents, 2 multi-byte windows): out host [max_batch][*row_len], out[b * row_len + j] = the pool
 * page of slots [64 j, 64 j + 64) of sequence b, or -1 (unmapped); *used = pages mapped from the
 * pool so far; *pages = the pool's size. cap (entries of out) below max_batch * row_len:
 * LCA_E_CAPACITY (and *row_len is still set). Synchronises the context's stream. */
int lca_debug_page_table(lca_ctx* ctx, int32_t cache, int32_t* out, int64_t cap, int32_t* row_len, int32_t* used,
                         int32_t* pages);

/* Run later steps as direct kernel launches instead of one graph (on != 0), so that
 * per-kernel profilers can see them; the LM decision is then read back on the host.
 * Results are identical. */
int lca_debug_set_eager(lca_ctx* ctx, int32_t on);

/* Per-kind timing of `steps` eager steps: CUDA events around every launch on the context
 * stream. Kinds: 0 linear layers, 1 attention, 2 unembedding heads, 3 glue. bytes: the
 * weight bytes each launch must read (linear layers and heads), summed. */
typedef struct {
  int64_t launches[4];
  double ms[4];
  double bytes[4];
} lca_profile;
int lca_debug_profile(lca_ctx* ctx, int32_t n, float tau, int32_t accept_mode, int32_t steps,
                      lca_profile* out);

/* Run `steps` step graphs with launch tracing on: thread 0 of every CTA of every kernel records
 * {u64 start_ns, u64 end_ns, u64 wait_done_ns, i32 kernel tag, i32 cta, i32 sm, i32 mark_ns[3]}
 * (48 bytes; a mark is a mid-kernel time after entry, 0 if the kernel sets none) into `out`
 * (host, room for `cap` records); count = records written. Needs a bf16 context (the trace
 * buffer borrows scratch that the bf16 step does not use). */
int lca_debug_trace(lca_ctx* ctx, int32_t n, float tau, int32_t accept_mode, int32_t steps,
                    void* out, int32_t cap, int32_t* count);

/* The tensor-core linear layer alone: y[0:*M_dev] = x . W^T on tcgen05 (two launches: rows split
 * into bf16 halves x = hi + lo, so that about 16 bits of each activation enter the product, then
 * a GEMM fed entirely by TMA; fp32 accumulation). Up to 64 typical rows (and N a multiple of 128)
 * the GEMM takes the weights as the MMA's M operand and splits K across a cluster (environment
 * LCA_SGEMM_MAX_ROWS sets that limit, 0 turns it off); otherwise the activations are the M
 * operand. x: device fp32 [M][K]; W: device bf16 [N][K];
 * y: device fp32 [M][N]; M_dev: device int32 rows to compute (<= M); rows_typ: the row count the
 * launch shape is chosen for (0 = M; a smaller value makes CTAs walk several row tiles); err_dev:
 * device int32 error word (bit 4: a bounded wait ran out); scratch: device,
 * lca_debug_gemm_scratch_bytes(M, K) bytes (the split rows). N and K must be multiples of 64.
 * Asynchronous on `stream`. */
int lca_debug_gemm(const float* x, const void* W, float* y, int32_t M, int32_t N, int32_t K,
                   const int32_t* M_dev, int32_t rows_typ, int32_t* err_dev, void* scratch, void* stream);
/* Where the tensor-core decode attention last gave up a bounded wait (16 int32 to host `out16`;
 * out16[0] == 0: none since the last call): {set, block x, y, z, warp, which (0: waiting for a
 * ring slot, 1: waiting for a chunk), chunk, stage, chunks, key lo, key hi, chunks before the
 * tile, copies issued}. Clears the record. */
int lca_debug_attn_diag(int32_t* out16);
/* Test hook for the bounded waits: the first wait of the weight-streaming GEMV for its weight tile,
 * and the first wait of each phase of the persistent stack kernel for its weight ring, spin at most
 * `spins` times (< 0: the default, 2^22) on the current device. With 0 the wait reports late at
 * once: the kernel records the timeout bit in the device error word, waits once more with the full
 * budget for its copies in flight, then completes (the stack kernel skips its remaining blocks),
 * and the call returns LCA_E_TIMEOUT. Outside a test, a call that returns LCA_E_TIMEOUT has undefined results, and if
 * the second wait ran out as well a copy may have been left in flight: destroy the context. */
int lca_debug_set_wait_spins(int32_t spins);
/* Bytes of device scratch lca_debug_gemm needs. */
size_t lca_debug_gemm_scratch_bytes(int32_t M, int32_t K);

/* Micro-benchmark: one graph of `iters` back-to-back launches of one kernel kind over `rows`
 * rows (0 RMSNorm+QKV, 1 Wo, 2 RMSNorm+W1/W3+SwiGLU, 3 W2, 4 decode attention over the
 * encoder cache, 5 unembedding head, 6 a glue kernel), cycling through all blocks' weights so
 * that every launch streams its weights from HBM. us: average time per launch (CUDA events);
 * bytes: the weight (or KV) bytes one launch reads. Overwrites step state: call lca_prefill
 * before the next step. */
int lca_debug_bench_kernel(lca_ctx* ctx, int32_t kind, int32_t rows, int32_t iters, double* us,
                           double* bytes);
/* Logits of the last step: nb host [batch * n * 256] (next-byte rows of the n candidates),
 * mb host [batch * (n-1) * 256] (drafter rows). Either may be NULL. */
int lca_debug_logits(lca_ctx* ctx, float* nb, float* mb);
/* Force the accepted-draft count of the NEXT step only: a host [batch], each in 0..n-1, or
 * NULL to clear. */
int lca_debug_force_accept(lca_ctx* ctx, const int32_t* a);
/* Replace the n candidates (c_1, d_2..d_n) of the NEXT step only: cand host [batch * n], or
 * NULL to clear. The drafter still runs and its logits stay readable. */
int lca_debug_force_candidates(lca_ctx* ctx, const uint8_t* cand, int32_t n);

/* Decode attention as a standalone call: the attention every module of the decode step
 * runs (causal softmax attention, Section 2.2; inside the multi-byte window of Algorithm 1
 * (drafting step) the LCA mask reduces to the same causal form). Query row r of sequence b sees the
 * cache slots [0, kv_len[r]) of its sequence; softmax scale `scale`; fp32 arithmetic.
 *   q, out:   device fp32 [batch * n_rows][heads * head_dim] (RoPE already applied to q).
 *   k_cache, v_cache: device [batch][heads][slots][head_dim] of `dtype` (LCA_F32|LCA_BF16).
 *   kv_len:   device int32 [batch * n_rows], each 1..slots. A larger value is an error: that row
 *             reads only the slots [0, slots), and the call records LCA_E_DEVICE_STATE in the error
 *             word, which lca_decode_attention_status returns.
 *   splits:   1..16; the key range of each (sequence, head) is split over `splits` CTAs whose
 *             partial results are combined in a fixed order (deterministic).
 *   scratch:  device memory of >= lca_decode_attention_scratch_bytes(...), 256-byte aligned,
 *             caller-owned; overwritten by the call. Its first 4 bytes are the call's error word
 *             (0: no error), cleared at the start of each call and read by
 *             lca_decode_attention_status.
 * head_dim must be 32 or 64. Asynchronous on `stream` (a cudaStream_t). Returns LCA_E_ARG for
 * bad arguments and LCA_E_CAPACITY for too small a scratch; what the kernels find while running
 * (an out-of-range kv_len, a bounded wait that ran out) is read afterwards with
 * lca_decode_attention_status. */
int lca_decode_attention_scratch_bytes(int32_t batch, int32_t heads, int32_t head_dim,
                                       int32_t splits, size_t* out);
int lca_decode_attention(const float* q, float* out, const void* k_cache, const void* v_cache,
                         int32_t dtype, int32_t batch, int32_t heads, int32_t head_dim,
                         int32_t slots, int32_t n_rows, const int32_t* kv_len, float scale,
                         int32_t splits, void* scratch, size_t scratch_bytes, void* stream);

/* lca_decode_attention for callers that cannot allocate device memory: plugin or custom-op
 * hosts that hand a kernel only its input and output buffers, and code paths where an
 * allocation call is not allowed because it may synchronize the device or break a fixed
 * memory budget. (The paper has no counterpart; this is a library convenience.)
 * Same arguments and results as lca_decode_attention without the scratch pair. The scratch is
 * a fixed device array inside the library, lca_decode_attention_noalloc_capacity() bytes
 * (8 MiB), which every GPU that loads the library holds until the process exits. Sizes whose
 * scratch (lca_decode_attention_scratch_bytes) exceeds it return LCA_E_CAPACITY. The call
 * allocates nothing: no cudaMalloc, no cudaFree, no allocating library routine.
 * The first call on a device looks up the array's device address (once per device, with that
 * device current); make that first call before any stream capture. All calls share the one
 * array and it keeps the last call's contents; each call clears the parts that must start at
 * zero. Calls that may overlap on the GPU (other streams, other host threads) race on it:
 * order them on one stream. */
int lca_decode_attention_noalloc(const float* q, float* out, const void* k_cache, const void* v_cache,
                                 int32_t dtype, int32_t batch, int32_t heads, int32_t head_dim,
                                 int32_t slots, int32_t n_rows, const int32_t* kv_len, float scale,
                                 int32_t splits, void* stream);
size_t lca_decode_attention_noalloc_capacity(void);

/* Status of the last lca_decode_attention call that used `scratch` (or, for the _noalloc form, of
 * the last lca_decode_attention_noalloc call on the current device): waits for `stream`, then
 * returns LCA_OK, LCA_E_DEVICE_STATE (a kv_len beyond slots: that row read only [0, slots)) or
 * LCA_E_TIMEOUT (a bounded wait ran out). Enqueue nothing between the call and its status read
 * that reuses the same scratch. The _noalloc form allocates nothing either. The device address of
 * the library's fixed array is looked up once per device and kept for the life of the process;
 * after cudaDeviceReset on a device, neither _noalloc call may be used on it again. */
int lca_decode_attention_status(const void* scratch, void* stream);
int lca_decode_attention_noalloc_status(void* stream);

int lca_destroy(lca_ctx* ctx);
const char* lca_status_str(int status);

#ifdef __cplusplus
}
#endif
#endif /* LCA_H */
