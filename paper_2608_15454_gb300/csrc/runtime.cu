// Host runtime behind include/lca.h: workspace layout, weight repacking, prefill, and the
// decode step as a CUDA graph. One step is one graph replay with no host round trip; the
// LM module sits in an IF conditional node that the segmentation kernel switches on only
// when a segment closes (Algorithm 1, LM-module branch). lca_generate wraps the step in a WHILE
// conditional node whose control kernel stops once every sequence has its bytes.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstdlib>
#include <thread>
#include <cstdio>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include "common.cuh"

using namespace lca;

namespace {

constexpr int kParamSlots = 8;
constexpr int kMaxN = 16;

struct Carver {
  char* base;
  size_t off = 0;
  template <typename T>
  T* take(size_t count) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

struct Layout {
  Dev D{};
  std::vector<Block> enc, lm, nb, mb;
  size_t bytes = 0;
};

size_t tw_bytes(int dtype) { return dtype == LCA_BF16 ? 2 : 4; }

// Carve the whole workspace; base == nullptr only measures it.
void carve(const lca_config& c, char* base, Layout& L) {
  Carver cv{base};
  Dev& D = L.D;
  D.d = c.d_model;
  D.H = c.n_heads;
  D.hd = c.head_dim;
  D.F = c.d_ff;
  D.n_enc = c.n_enc;
  D.n_lm = c.n_lm;
  D.n_nb = c.n_nb;
  D.n_mb = c.n_mb;
  D.mb_kind = c.mb_kind;
  D.n_mlp_heads = c.n_mlp_heads;
  D.dtype = c.dtype;
  D.B = c.max_batch;
  D.S = c.max_bytes;
  D.L = c.max_bytes + 1;
  D.NMAX = c.max_n;
  D.R = c.max_batch * (c.max_bytes + c.max_n);
  D.boundary = c.boundary_byte;
  D.eps = c.rms_eps;
  D.scale = c.attn_scale;
  const size_t d = D.d, F = D.F, tb = tw_bytes(c.dtype);
  const size_t B = D.B, S = D.S, Lt = D.L, R = D.R, NM = D.NMAX;

  // paged caches: page tables and pool sizes (pages of kPage positions)
  D.pt_ld_byte = (int)((S + kPage - 1) / kPage);
  D.pt_ld_lm = (int)((Lt + kPage - 1) / kPage);
  D.pt_ld_mb = D.pt_ld_byte;
  D.pages_byte = c.kv_pages > 0 ? c.kv_pages : (int)B * D.pt_ld_byte;
  D.pages_lm = c.lm_pages > 0 ? c.lm_pages : (int)B * D.pt_ld_lm;
  D.pages_mb = c.mb_pages > 0 ? c.mb_pages : (int)B * D.pt_ld_mb;
  D.pt_byte = cv.take<int>(B * D.pt_ld_byte);
  D.pt_lm = cv.take<int>(B * D.pt_ld_lm);
  D.pt_mb = cv.take<int>(B * D.pt_ld_mb);
  D.pool_next = cv.take<int>(4);

  D.embed = cv.take<char>(256 * d * tb);
  D.unembed = cv.take<char>(256 * d * tb);
  D.bos = cv.take<float>(d);
  D.nb_norm = cv.take<float>(d);
  D.mb_norm = cv.take<float>(d);
  // every cache layer: a pool of pages [pages][H][kPage][hd] behind its module's page table
  auto blocks = [&](std::vector<Block>& v, int n, size_t slots, const int* pt, int pt_ld, int pages) {
    v.resize(n);
    for (auto& b : v) {
      b.attn_norm = cv.take<float>(d);
      b.mlp_norm = cv.take<float>(d);
      b.wqkv = cv.take<char>(3 * d * d * tb);
      b.wo = cv.take<char>(d * d * tb);
      b.w13 = cv.take<char>(2 * F * d * tb);
      b.w2 = cv.take<char>(d * F * tb);
      b.kv.S = (int)slots;
      b.kv.pt = pt;
      b.kv.pt_ld = pt_ld;
      b.kv.pages = pages;
      b.kv.k = cv.take<char>((size_t)pages * D.H * kPage * D.hd * tb);
      b.kv.v = cv.take<char>((size_t)pages * D.H * kPage * D.hd * tb);
    }
  };
  blocks(L.enc, c.n_enc, S, D.pt_byte, D.pt_ld_byte, D.pages_byte);
  blocks(L.lm, c.n_lm, Lt, D.pt_lm, D.pt_ld_lm, D.pages_lm);
  blocks(L.nb, c.n_nb, S, D.pt_byte, D.pt_ld_byte, D.pages_byte);
  if (c.mb_kind == LCA_MB_LCA) {
    blocks(L.mb, c.n_mb, S, D.pt_mb, D.pt_ld_mb, D.pages_mb);
    D.mlp_w = nullptr;
  } else {
    L.mb.clear();
    D.mlp_w = cv.take<char>((size_t)c.n_mb * c.n_mlp_heads * d * d * tb);
  }

  D.seq = cv.take<SeqState>(B);
  D.gstart = cv.take<int>(B * Lt);
  D.h_store = cv.take<float>(B * S * d);
  D.u_tab = cv.take<float>(B * Lt * d);
  D.o_tab = cv.take<float>(B * Lt * d);
  D.y_last = cv.take<float>(B * d);
  D.kpos = cv.take<int>(B * S);
  // split activations of the tensor-core layers (two alternating buffers) and the rows' sums of
  // squares: any row set of the step or of prefill (bf16)
  D.as_rows = c.dtype == LCA_BF16 ? (int)R : 0;
  for (int i = 0; i < 2; ++i) {
    D.as_hi[i] = cv.take<__nv_bfloat16>((size_t)D.as_rows * std::max(d, F));
    D.as_lo[i] = cv.take<__nv_bfloat16>((size_t)D.as_rows * std::max(d, F));
  }
  D.as_ss_ld = (int)d / 32;
  D.as_ss = cv.take<float>((size_t)D.as_rows * D.as_ss_ld);
  D.gv_ss_ld = (int)d / 16;
  D.gv_ss = cv.take<float>((size_t)D.as_rows * D.gv_ss_ld);

  D.x_mb = cv.take<float>(R * d);
  D.x_enc = cv.take<float>(R * d);
  D.x_lm = cv.take<float>(R * d);
  D.x_nb = cv.take<float>(R * d);
  D.qbuf = cv.take<float>(R * d);
  D.att = cv.take<float>(R * d);
  D.mid = cv.take<float>(R * F);
  D.xnorm = nullptr;
  auto rows = [&](Rows& r) {
    r.b = cv.take<int>(R);
    r.pos = cv.take<int>(R);
    r.slot = cv.take<int>(R);
    r.page = cv.take<int>(R);
    r.kvlen = cv.take<int>(R);
    r.seq_start = cv.take<int>(B);
    r.seq_count = cv.take<int>(B);
    r.M = cv.take<int>(1);
  };
  rows(D.r_mb);
  rows(D.r_v);
  rows(D.r_lm);

  const size_t HR = std::max<size_t>(B * NM, B);
  D.head_rows_mb = cv.take<int>(HR);
  D.head_rows_v = cv.take<int>(HR);
  D.M_head_mb = cv.take<int>(1);
  D.M_head_v = cv.take<int>(1);
  D.mb_logits = cv.take<float>(HR * 256);
  D.nb_logits = cv.take<float>(HR * 256);
  D.mb_arg = cv.take<int>(HR);
  D.mb_prob = cv.take<float>(HR);
  D.nb_arg = cv.take<int>(HR);
  D.nb_prob = cv.take<float>(HR);

  D.cand = cv.take<int>(B * NM);
  D.kc = cv.take<int>(B * NM);
  D.out_step = cv.take<uint8_t>(B * NM);
  D.out_cnt = cv.take<int>(B);
  D.out_gen = cv.take<uint8_t>(B * S);
  D.hist = cv.take<int>(NM);
  D.forced_a = cv.take<int>(B);
  D.forced_cand = cv.take<int>(B * NM);
  D.params = cv.take<Params>(kParamSlots);
  D.err = cv.take<int>(1);
  D.stats = cv.take<Stats>(1);
  D.step_log = cv.take<uint8_t>(kStepLog);

  const size_t gemv_rows = B <= 4 ? R : 64;
  D.lin_part_floats = (size_t)kMaxKSplit * gemv_rows * d;
  D.lin_part = cv.take<float>(D.lin_part_floats);
  D.lin_cnt = cv.take<int>(8192);
  D.head_cnt = cv.take<int>(std::max<size_t>(R / 8 + 1, 1024));
  D.attn_part = cv.take<float>(attention_scratch_floats(D.B, D.H, D.hd));
  D.attn_cnt = cv.take<int>(attention_counters(D.B, D.H));
  D.inv_rms = cv.take<float>(R);
  D.rope_slots = (int)std::max(S, Lt);
  D.rope = cv.take<float2>((size_t)D.rope_slots * (D.hd / 2));
  // persistent stack kernel: bf16, head_dim 64, d <= 1024 (one K-slice), up to four sequences
  const size_t KS = std::min<size_t>(d, 1024);
  const bool stk = c.dtype == LCA_BF16 && D.hd == 64 && d % 16 == 0 && d <= 1024 && KS % 16 == 0 &&
                   F % KS == 0 && F / KS <= 4 && B <= 4;
  if (stk) {
    D.stk_enc = cv.take<StackLayer>(std::max(c.n_enc, 1));
    D.stk_lm = cv.take<StackLayer>(std::max(c.n_lm, 1));
    D.stk_nb = cv.take<StackLayer>(std::max(c.n_nb, 1));
    D.stk_mb = cv.take<StackLayer>(std::max(c.n_mb, 1));
    D.stk_apart_rows = (size_t)std::max(S, Lt) + NM;
    D.stk_apart = cv.take<float>(B * D.H * kMaxAttnSplit * D.stk_apart_rows * 68);
    D.stk_cnt = cv.take<int>(B * D.H);
    D.stk_bar = cv.take<unsigned>(64);
    D.stk_ahi = cv.take<__nv_bfloat16>(R * d);
    D.stk_alo = cv.take<__nv_bfloat16>(R * d);
    D.stk_thi = cv.take<__nv_bfloat16>(R * d);
    D.stk_tlo = cv.take<__nv_bfloat16>(R * d);
    D.stk_mhi = cv.take<__nv_bfloat16>(R * F);
    D.stk_mlo = cv.take<__nv_bfloat16>(R * F);
    D.stk_ss = cv.take<float>(R * (d / 16));
    D.stk_w2part = cv.take<float>((F / KS) * R * d);
    D.stk_w2cnt = cv.take<int>(d / 16);
  } else {
    D.stk_enc = D.stk_lm = D.stk_nb = D.stk_mb = nullptr;
    D.stk_apart = nullptr;
    D.stk_cnt = nullptr;
    D.stk_bar = nullptr;
    D.stk_apart_rows = 0;
    D.stk_ahi = D.stk_alo = D.stk_thi = D.stk_tlo = D.stk_mhi = D.stk_mlo = nullptr;
    D.stk_ss = nullptr;
    D.stk_w2part = nullptr;
    D.stk_w2cnt = nullptr;
  }
  L.bytes = cv.off + 256;
}

// Prefill staging lives after the layout: bytes and per-sequence offsets.
struct Staging {
  uint8_t* bytes;
  int* row0;
  int* lens;
  int* lm_row0;
};

}  // namespace

struct alignas(64) TMapBlob {
  unsigned char b[128];
};
struct alignas(64) SplitMapBlob {
  unsigned char b[kSplitMapBytes];  // (hi, lo) maps of split activations, or (K, V) of a cache layer
};

struct lca_ctx {
  std::map<const void*, TMapBlob> tmaps;  // TMA tensor maps of the bf16 weights
  std::map<int, SplitMapBlob> amaps;      // TMA tensor maps of the split activations, by 2 K + buffer
  std::map<const void*, SplitMapBlob> kvmaps;  // TMA tensor maps (K, V) of the bf16 cache layers
  lca_config cfg{};
  Layout L;
  Staging stg{};
  char* ws = nullptr;
  size_t ws_bytes = 0;
  cudaStream_t stream = nullptr;
  cudaStream_t cap = nullptr, cap2 = nullptr;
  Params* h_params = nullptr;  // pinned ring
  int param_slot = 0;
  Params host_params{};
  int batch = 0;
  bool prefilled = false;
  std::vector<long long> t_host;
  std::map<int, cudaGraphExec_t> step_exec, gen_exec;
  std::vector<cudaGraph_t> graphs;
  int last_n = 0;
  int pending_force_accept = 0;
  int pending_force_cand = 0;
  int pending_force_cand_n = 0;
  int gen_max_new = 0;
  int gen_n = 0;
  bool t_unsynced = false;
  // typical cache lengths (bytes; latents) that the step graphs' attention key splits are chosen
  // for: the longest sequence after the last prefill
  int kv_bytes_typ = 0, kv_lat_typ = 0;
  bool eager = false;
  // kernels per step graph part, by n: [pre-LM + post-LM, LM body]
  std::map<int, std::pair<long long, long long>> launches;
};

namespace {

int check(cudaError_t e, const char* what) {
  if (e != cudaSuccess) {
    fprintf(stderr, "lca: %s: %s\n", what, cudaGetErrorString(e));
    return LCA_E_CUDA;
  }
  return LCA_OK;
}
#define CK(x)                                   \
  do {                                          \
    int _s = check((x), #x);                    \
    if (_s != LCA_OK) return _s;                \
  } while (0)

int validate(const lca_config* c) {
  if (!c) return LCA_E_ARG;
  if (c->vocab != 256 || c->d_model <= 0 || c->n_heads <= 0 || c->head_dim <= 0) return LCA_E_ARG;
  if (c->n_heads * c->head_dim != c->d_model) return LCA_E_ARG;
  if (c->head_dim != 32 && c->head_dim != 64) return LCA_E_ARG;
  if (c->d_model % 16 || c->d_ff % 16) return LCA_E_ARG;
  if (c->dtype != LCA_F32 && c->dtype != LCA_BF16) return LCA_E_ARG;
  if (c->mb_kind != LCA_MB_LCA && c->mb_kind != LCA_MB_MLP) return LCA_E_ARG;
  if (c->max_batch < 1 || c->max_batch > 1024 || c->max_bytes < 2 || c->max_n < 1 || c->max_n > kMaxN)
    return LCA_E_ARG;
  if (c->mb_kind == LCA_MB_MLP && c->n_mlp_heads < c->max_n - 1) return LCA_E_ARG;
  if (c->n_enc < 0 || c->n_lm < 0 || c->n_nb < 0 || c->n_mb < 0) return LCA_E_ARG;
  if (c->boundary_byte < 0 || c->boundary_byte > 255) return LCA_E_ARG;
  if (c->kv_pages < 0 || c->lm_pages < 0 || c->mb_pages < 0) return LCA_E_ARG;
  // the attention kernels stage a sequence's page table row in shared memory
  if ((c->max_bytes + kPage) / kPage > kMaxPtRow) return LCA_E_ARG;
  return LCA_OK;
}

Params* next_params(lca_ctx* c) {
  c->param_slot = (c->param_slot + 1) % kParamSlots;
  Params* hp = c->h_params + c->param_slot;
  *hp = c->host_params;
  return hp;
}

int upload_params(lca_ctx* c) {
  Params* hp = next_params(c);
  CK(cudaMemcpyAsync(c->L.D.params, hp, sizeof(Params), cudaMemcpyHostToDevice, c->stream));
  return LCA_OK;
}

bool tiled_for(const Dev& D, int rows) { return rows > D.tiled_min_rows; }

// Split-activation maps of buffer `buf` for a layer of inner size K whose rows fit the buffers.
const void* amap_of(lca_ctx* c, int buf, int K, int rows_cap) {
  if (rows_cap > c->L.D.as_rows) return nullptr;
  auto it = c->amaps.find(2 * K + buf);
  return it == c->amaps.end() ? nullptr : it->second.b;
}

const void* tmap_of(lca_ctx* c, const void* W) {
  auto it = c->tmaps.find(W);
  return it == c->tmaps.end() ? nullptr : it->second.b;
}

constexpr int kMbWindowKeys = 32;  // the multi-byte window's cache: about two words

// Key splits of a decode attention launch: enough CTAs for about two per SM; with
// D.attn_min_keys > 0, also at least that many keys per split of a cache of about kv_typ keys
// (measured: more, shorter splits are faster even for caches of a few hundred keys, so the
// limit is off unless set).
int attn_splits(const Dev& D, int batch_cap, int qtiles, int kv_typ) {
  int s = (2 * D.num_sms) / std::max(1, batch_cap * D.H * qtiles);
  if (kv_typ > 0 && D.attn_min_keys > 0)
    s = std::min(s, std::max(1, (kv_typ + D.attn_min_keys - 1) / D.attn_min_keys));
  return std::max(1, std::min(std::min(s, kMaxAttnSplit), D.attn_split_cap));
}

// Split on write: the epilogue of `prod` also stores its output as the bf16 halves (times `gain`, the
// consumer's RMSNorm gain, or 1) that the tensor-core layer `cons` reads from split buffer `buf`,
// plus per-32-column sums of squares when the consumer normalises. Only when both layers run on
// the tensor cores; returns whether the link was made.
bool link_split(const Dev& D, bool tiled, LinearArgs& prod, LinearArgs& cons, int buf, const float* gain,
                bool drop_fp32) {
  cons.abuf = buf;
  cons.presplit = 1;
  const bool ok = D.split_write && tiled && umma_ready(D, prod) && umma_ready(D, cons) && cons.groups == prod.groups &&
                  cons.Mg_stride == prod.Mg_stride && prod.abuf != buf && (!gain || cons.Kd == prod.N);
  if (!ok) {
    cons.presplit = 0;
    return false;
  }
  prod.epi.sp_hi = D.as_hi[buf];
  prod.epi.sp_lo = D.as_lo[buf];
  prod.epi.ldsp = cons.Kd;
  prod.epi.sg = gain;
  prod.epi.ss = gain ? D.as_ss : nullptr;
  prod.epi.ss_ld = D.as_ss_ld;
  prod.epi.sp_only = drop_fp32 ? 1 : 0;
  return true;
}

// Split on write between two weight-streaming GEMV layers (few rows): the producer's epilogue also
// stores its output as bf16 halves of v * gain (gain: the consumer's RMSNorm gain, or 1) into
// split buffer `buf`, with the sums of v^2 per 16-column block when the consumer normalises, and
// the consumer stages its rows by bulk copies instead of loading and splitting fp32 rows. Only
// when both layers run on the bulk-copy GEMV; returns whether the link was made.
bool link_split_gemv(const Dev& D, bool tiled, LinearArgs& prod, LinearArgs& cons, int buf, const float* gain,
                     bool drop_fp32) {
  const bool resid = prod.epi.mode == EPI_RESID, swiglu = prod.epi.mode == EPI_SWIGLU;
  const bool ok = D.gemv_split && !tiled && D.as_rows > 0 && cons.M_cap <= D.as_rows && prod.groups == 1 &&
                  cons.groups == 1 && !prod.epi.sp_hi && gemv_bulk_ok(D, prod) && gemv_bulk_ok(D, cons) &&
                  ((resid && cons.Kd == prod.N) || (swiglu && !gain && cons.Kd == prod.N / 2)) &&
                  // a normalising consumer stages the rows' partial squares (8 rows x Kd / 16) in the
                  // gain's area of Kd / ksplit floats
                  (!gain || gemv_bulk_ksplit(D, cons) <= 2);
  if (!ok) return false;
  cons.gsplit = 1;
  cons.abuf = buf;
  prod.epi.sp_hi = D.as_hi[buf];
  prod.epi.sp_lo = D.as_lo[buf];
  prod.epi.ldsp = cons.Kd;
  prod.epi.sg = gain;
  prod.epi.ss = gain ? D.gv_ss : nullptr;
  prod.epi.ss_ld = D.gv_ss_ld;
  prod.epi.sp_only = drop_fp32 ? 1 : 0;
  return true;
}

// Run the pre-norm blocks of one module over rows [0, *rows.M) of x (in place). On the tensor
// cores, each layer's input is split into bf16 halves by the layer before it (its epilogue writes
// them into the other of the two split buffers); only a stack's first layer and the attention
// output go through k_split_rows.
void run_stack(lca_ctx* c, std::vector<Block>& blocks, float* x, const Rows& rows, int M_cap,
               int M_typ, int qt_grid, int splits, cudaStream_t s, const void* next_w = nullptr,
               size_t next_bytes = 0, const int* stable = nullptr, bool short_kv = false, int stable_add = 0,
               const StackLayer* stk = nullptr) {
  Dev& D = c->L.D;
  const bool tiled = tiled_for(D, M_typ);
  // decode steps with few rows: the whole stack as one persistent launch
  if (stk && !tiled && !blocks.empty() && stack_ready(D)) {
    StackRun r{};
    r.layers = stk;
    r.L = (int)blocks.size();
    r.x = x;
    r.rows = rows;
    r.M_cap = M_cap;
    r.S = blocks[0].kv.S;
    r.pt = blocks[0].kv.pt;
    r.pt_ld = blocks[0].kv.pt_ld;
    r.pages = blocks[0].kv.pages;
    r.stable = stable;
    r.stable_stride = (int)(sizeof(SeqState) / sizeof(int));
    r.stable_add = stable_add;
    if (launch_stack(D, r, s)) return;
  }
  const size_t tb = tw_bytes(D.dtype);
  const size_t b_qkv = 3ull * D.d * D.d * tb, b_o = (size_t)D.d * D.d * tb;
  const size_t b_13 = 2ull * D.F * D.d * tb, b_2 = (size_t)D.d * D.F * tb;
  LinearArgs base{};
  base.groups = 1;
  base.Mg_stride = 0;
  base.eps = D.eps;
  base.M = rows.M;
  base.M_cap = M_cap;
  base.rows_typ = M_typ;
  base.epi.err = D.err;
  // the QKV layer of block l; split buffer 0
  auto qkv_args = [&](const Block& bk) {
    LinearArgs a = base;
    a.x = x;
    a.ldx = D.d;
    a.W = bk.wqkv;
    a.N = 3 * D.d;
    a.Kd = D.d;
    a.norm = bk.attn_norm;
    a.epi.mode = EPI_QKV;
    a.epi.y = D.qbuf;
    a.epi.ldy = D.d;
    a.epi.kv = bk.kv;
    a.epi.rows = rows;
    a.epi.rope = D.rope;
    a.epi.H = D.H;
    a.epi.hd = D.hd;
    a.epi.d = D.d;
    a.pf[0] = bk.wo;
    a.pf_bytes[0] = b_o;
    a.pf[1] = bk.w13;
    a.pf_bytes[1] = b_13;
    a.tmap = tmap_of(c, a.W);
    a.abuf = 0;
    a.amap = amap_of(c, 0, a.Kd, a.M_cap * a.groups);
    return a;
  };
  LinearArgs aq = blocks.empty() ? base : qkv_args(blocks[0]);
  for (size_t l = 0; l < blocks.size(); ++l) {
    Block& bk = blocks[l];
    const Block* nx = l + 1 < blocks.size() ? &blocks[l + 1] : nullptr;
    const void* nqkv = nx ? nx->wqkv : next_w;
    const size_t nqkv_b = nx ? b_qkv : next_bytes;
    // x += Wo . attn (input split by k_split_rows into buffer 1)
    LinearArgs ao = base;
    ao.x = D.att;
    ao.ldx = D.d;
    ao.W = bk.wo;
    ao.N = D.d;
    ao.Kd = D.d;
    ao.epi.mode = EPI_RESID;
    ao.epi.y = x;
    ao.epi.res = x;
    ao.epi.ldy = ao.epi.ldres = D.d;
    ao.pf[0] = bk.w2;
    ao.pf_bytes[0] = b_2;
    ao.tmap = tmap_of(c, ao.W);
    ao.abuf = 1;
    ao.amap = amap_of(c, 1, ao.Kd, ao.M_cap * ao.groups);
    // mid = silu(W1 . n(x)) * (W3 . n(x)) (input in buffer 0)
    LinearArgs a13 = base;
    a13.x = x;
    a13.ldx = D.d;
    a13.W = bk.w13;
    a13.N = 2 * D.F;
    a13.Kd = D.d;
    a13.norm = bk.mlp_norm;
    a13.epi.mode = EPI_SWIGLU;
    a13.epi.y = D.mid;
    a13.epi.ldy = D.F;
    a13.pf[0] = nqkv;
    a13.pf_bytes[0] = nqkv_b;
    a13.tmap = tmap_of(c, a13.W);
    a13.amap = amap_of(c, 0, a13.Kd, a13.M_cap * a13.groups);
    // x += W2 . mid (input in buffer 1)
    LinearArgs a2 = base;
    a2.x = D.mid;
    a2.ldx = D.F;
    a2.W = bk.w2;
    a2.N = D.d;
    a2.Kd = D.F;
    a2.epi.mode = EPI_RESID;
    a2.epi.y = x;
    a2.epi.res = x;
    a2.epi.ldy = a2.epi.ldres = D.d;
    a2.pf[0] = nx ? nx->wo : nullptr;
    a2.pf_bytes[0] = nx ? b_o : 0;
    a2.tmap = tmap_of(c, a2.W);
    a2.amap = amap_of(c, 1, a2.Kd, a2.M_cap * a2.groups);
    LinearArgs aq_next = nx ? qkv_args(*nx) : base;
    link_split(D, tiled, ao, a13, 0, bk.mlp_norm, false);
    link_split(D, tiled, a13, a2, 1, nullptr, true);
    if (nx) link_split(D, tiled, a2, aq_next, 0, nx->attn_norm, false);
    link_split_gemv(D, tiled, ao, a13, 0, bk.mlp_norm, false);
    link_split_gemv(D, tiled, a13, a2, 1, nullptr, true);
    if (nx) link_split_gemv(D, tiled, a2, aq_next, 0, nx->attn_norm, false);
    // the attention output as Wo's pre-split input (split buffer 1: a2 of the block before has read it)
    const bool att_split = D.gemv_split && !tiled && D.as_rows > 0 && M_cap <= D.as_rows && gemv_bulk_ok(D, ao) &&
                           attention_split_out(D, bk.kv, D.B, qt_grid, short_kv);
    if (att_split) {
      ao.gsplit = 1;
      ao.abuf = 1;
    }

    // RMSNorm -> Q,K,V -> RoPE -> K,V appended to the cache
    linear(D, aq, tiled, s);
    attention(D, D.qbuf, D.att, bk.kv, rows, D.B, qt_grid, splits, s, stable, short_kv, stable_add,
              std::max(1, M_cap / std::max(1, D.B)), att_split ? D.as_hi[1] : nullptr,
              att_split ? D.as_lo[1] : nullptr);
    linear(D, ao, tiled, s);
    linear(D, a13, tiled, s);
    linear(D, a2, tiled, s);
    aq = aq_next;
  }
}

// MLP-MBP drafter layers: v <- v + silu(W_{j,l} v) for every head j (grouped over heads).
void run_mlp_heads(lca_ctx* c, int n, cudaStream_t s) {
  Dev& D = c->L.D;
  const size_t tb = tw_bytes(D.dtype);
  const bool tiled = tiled_for(D, D.B);
  auto layer = [&](int l) {
    LinearArgs a{};
    a.x = D.x_mb;
    a.ldx = D.d;
    a.W = reinterpret_cast<char*>(D.mlp_w) + (size_t)l * D.n_mlp_heads * D.d * D.d * tb;
    a.N = D.d;
    a.Kd = D.d;
    a.groups = n - 1;
    a.Mg_stride = D.B;
    a.norm = nullptr;
    a.eps = D.eps;
    a.M = D.r_mb.M;
    a.M_cap = D.B;
    a.rows_typ = D.B;
    a.epi.mode = EPI_RESID_SILU;
    a.epi.y = D.x_mb;
    a.epi.res = D.x_mb;
    a.epi.ldy = a.epi.ldres = D.d;
    a.epi.err = D.err;
    a.tmap = tmap_of(c, a.W);
    a.abuf = l & 1;
    a.amap = amap_of(c, a.abuf, a.Kd, a.M_cap * a.groups);
    return a;
  };
  // layer l reads split buffer l % 2; its epilogue writes layer l + 1's input into the other one
  LinearArgs a = layer(0);
  for (int l = 0; l < D.n_mb; ++l) {
    LinearArgs an = l + 1 < D.n_mb ? layer(l + 1) : LinearArgs{};
    if (l + 1 < D.n_mb) link_split(D, tiled, a, an, (l + 1) & 1, nullptr, false);
    linear(D, a, tiled, s);
    a = an;
  }
}

// The three parts of one decode step, shared by graph capture and eager execution.
void enqueue_draft_encode(lca_ctx* c, int n, cudaStream_t s) {
  Dev& D = c->L.D;
  const int B = D.B;
  // (3) draft
  if (n >= 2) {
    if (D.mb_kind == LCA_MB_LCA) {
      launch_mb_plan(D, s);
      // typical window rows. A single sequence rebuilds its window after most committed boundaries:
      // about a word of bytes, the n new bytes and the n - 2 copies. In a batch the sequences that
      // only append their n new bytes and n - 2 copies set the count.
      const int typ = B == 1 ? 2 * n + 6 : B * (2 * n - 2);
      // the window holds about two words of keys: a short cache
      run_stack(c, c->L.mb, D.x_mb, D.r_mb, D.R, typ, 2, attn_splits(D, B, 2, kMbWindowKeys), s,
                c->L.enc.empty() ? nullptr : c->L.enc[0].wqkv, 3ull * D.d * D.d * tw_bytes(D.dtype), nullptr,
                true, 0, D.stk_mb);
    } else {
      launch_mlp_plan(D, s);
      run_mlp_heads(c, n, s);
    }
    launch_head(D, D.x_mb, D.head_rows_mb, D.M_head_mb, B * (n - 1), D.mb_norm, D.mb_logits,
                D.mb_arg, D.mb_prob, s);
  }
  // (1) embed + encoder over the n candidates
  launch_verify_plan(D, s);
  run_stack(c, c->L.enc, D.x_enc, D.r_v, B * n, B * n, 1, attn_splits(D, B, 1, c->kv_bytes_typ + n), s,
            c->L.nb.empty() ? nullptr : c->L.nb[0].wqkv, 3ull * D.d * D.d * tw_bytes(D.dtype),
            &D.seq[0].t, false, 0, D.stk_enc);
}

void enqueue_lm(lca_ctx* c, int n, cudaStream_t s) {
  Dev& D = c->L.D;
  // about one new latent per sequence every few bytes
  // latent slots [0, K] (BOS and the committed latents) do not change during the step
  run_stack(c, c->L.lm, D.x_lm, D.r_lm, D.B * n, D.B, 1, attn_splits(D, D.B, 1, c->kv_lat_typ + 1), s,
            nullptr, 0, &D.seq[0].K, false, 1, D.stk_lm);
  launch_lm_scatter(D, s);
}

void enqueue_verify_commit(lca_ctx* c, int n, cudaStream_t s) {
  Dev& D = c->L.D;
  const int B = D.B;
  // (4) upsample + next-byte decoder over the n candidates, head
  launch_nb_input(D, s);
  run_stack(c, c->L.nb, D.x_nb, D.r_v, B * n, B * n, 1, attn_splits(D, B, 1, c->kv_bytes_typ + n), s, nullptr, 0,
            &D.seq[0].t, false, 0, D.stk_nb);
  launch_head(D, D.x_nb, nullptr, D.r_v.M, B * n, D.nb_norm, D.nb_logits, D.nb_arg, D.nb_prob, s);
  // (5) accept + commit
  launch_commit(D, s);
}

// Capture one decode step into graph g (which may be the body of a WHILE node).
int capture_step(lca_ctx* c, cudaGraph_t g, int n, bool loop, cudaGraphConditionalHandle hwhile) {
  Dev& D = c->L.D;
  cudaStream_t s = c->cap;
  CK(cudaStreamBeginCaptureToGraph(s, g, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
  const long long l0 = g_launches;
  long long lm_launches = 0;
  enqueue_draft_encode(c, n, s);
  // segments closed by candidate boundaries -> LM rows; the LM runs only if there are any
  cudaStreamCaptureStatus st;
  cudaGraph_t cg;
  const cudaGraphNode_t* deps = nullptr;
  const cudaGraphEdgeData* edata = nullptr;
  size_t ndeps = 0;
  CK(cudaStreamGetCaptureInfo(s, &st, nullptr, &cg, nullptr, nullptr, nullptr));
  cudaGraphConditionalHandle hlm;
  CK(cudaGraphConditionalHandleCreate(&hlm, cg, 0, cudaGraphCondAssignDefault));
  launch_segment(D, hlm, 1, s);
  CK(cudaStreamGetCaptureInfo(s, &st, nullptr, &cg, &deps, &edata, &ndeps));
  cudaGraphNodeParams cp{};
  cp.type = cudaGraphNodeTypeConditional;
  cp.conditional.handle = hlm;
  cp.conditional.type = cudaGraphCondTypeIf;
  cp.conditional.size = 1;
  cudaGraphNode_t cnode;
  CK(cudaGraphAddNode(&cnode, cg, deps, edata, ndeps, &cp));
  cudaGraph_t body = cp.conditional.phGraph_out[0];
  {
    cudaStream_t s2 = c->cap2;
    CK(cudaStreamBeginCaptureToGraph(s2, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
    const long long b0 = g_launches;
    enqueue_lm(c, n, s2);
    lm_launches = g_launches - b0;
    cudaGraph_t tmp;
    CK(cudaStreamEndCapture(s2, &tmp));
  }
  CK(cudaStreamUpdateCaptureDependencies(s, &cnode, nullptr, 1, cudaStreamSetCaptureDependencies));
  enqueue_verify_commit(c, n, s);
  if (loop) launch_loop_ctl(D, hwhile, s);
  cudaGraph_t out;
  CK(cudaStreamEndCapture(s, &out));
  if (!loop) c->launches[n] = {g_launches - l0 - lm_launches, lm_launches};
  return LCA_OK;
}

// Holds a stream at a host node until release(): the launches (and profiling events) enqueued
// meanwhile then run back to back, so the event times of a profiled eager step measure the GPU,
// not the host's enqueue rate. The host-side wait is bounded (about five seconds).
struct HostGate {
  std::atomic<int> open{0};
  static void CUDART_CB wait_fn(void* p) {
    auto* g = static_cast<HostGate*>(p);
    for (int i = 0; i < 5000000 && !g->open.load(std::memory_order_acquire); ++i) std::this_thread::yield();
  }
  void hold(cudaStream_t s) { cudaLaunchHostFunc(s, wait_fn, this); }
  void release() { open.store(1, std::memory_order_release); }
};

// The same step as direct launches on the context stream; the LM decision is read back on
// the host. Used for per-kernel profiling (profilers cannot see kernels inside graphs with
// conditional nodes); results are identical to the graph. When profiling, each of the two
// segments is enqueued behind a host gate (see HostGate).
int run_step_eager(lca_ctx* c, int n) {
  Dev& D = c->L.D;
  cudaStream_t s = c->stream;
  const bool gate = g_prof != nullptr;
  HostGate g1, g2;
  // the step starts once the previous one has completed (as a graph launch does): kernels read the
  // committed cache prefix before their grid-dependency wait
  if (gate) g1.hold(s);
  else CK(cudaStreamSynchronize(s));
  enqueue_draft_encode(c, n, s);
  launch_segment(D, 0, 0, s);
  g1.release();
  int mlm = 0;
  CK(cudaMemcpyAsync(&mlm, D.r_lm.M, sizeof(int), cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  if (gate) g2.hold(s);
  if (mlm > 0) enqueue_lm(c, n, s);
  enqueue_verify_commit(c, n, s);
  g2.release();
  if (gate) CK(cudaStreamSynchronize(s));  // the gate's host node has run before g2 goes away
  CK(cudaGetLastError());
  return LCA_OK;
}

// Records CUDA events around each launch of an eager step and sums them per kind.
struct Profiler : ProfHook {
  struct Rec {
    int kind;
    double bytes;
    cudaEvent_t a, b;
  };
  std::vector<Rec> pool;
  size_t used = 0;
  double ms[PK_COUNT] = {0, 0, 0, 0};
  double bytes[PK_COUNT] = {0, 0, 0, 0};
  long long launches[PK_COUNT] = {0, 0, 0, 0};
  void begin(int kind, double by, cudaStream_t s) override {
    if (used == pool.size()) {
      Rec r{};
      cudaEventCreate(&r.a);
      cudaEventCreate(&r.b);
      pool.push_back(r);
    }
    Rec& r = pool[used];
    r.kind = kind;
    r.bytes = by;
    cudaEventRecord(r.a, s);
  }
  void end(cudaStream_t s) override { cudaEventRecord(pool[used++].b, s); }
  void collect() {
    for (size_t i = 0; i < used; ++i) {
      float t = 0.f;
      cudaEventSynchronize(pool[i].b);
      cudaEventElapsedTime(&t, pool[i].a, pool[i].b);
      ms[pool[i].kind] += t;
      bytes[pool[i].kind] += pool[i].bytes;
      launches[pool[i].kind] += 1;
    }
    used = 0;
  }
  ~Profiler() {
    for (auto& r : pool) {
      cudaEventDestroy(r.a);
      cudaEventDestroy(r.b);
    }
  }
};

// Destroy every captured step graph (they are captured again on next use).
void drop_graphs(lca_ctx* c) {
  cudaStreamSynchronize(c->stream);
  for (auto& kv : c->step_exec) cudaGraphExecDestroy(kv.second);
  for (auto& kv : c->gen_exec) cudaGraphExecDestroy(kv.second);
  c->step_exec.clear();
  c->gen_exec.clear();
  for (cudaGraph_t g : c->graphs) cudaGraphDestroy(g);
  c->graphs.clear();
}

int get_step_exec(lca_ctx* c, int n, cudaGraphExec_t* ex) {
  auto it = c->step_exec.find(n);
  if (it != c->step_exec.end()) {
    *ex = it->second;
    return LCA_OK;
  }
  cudaGraph_t g;
  CK(cudaGraphCreate(&g, 0));
  int st = capture_step(c, g, n, false, 0);
  if (st != LCA_OK) return st;
  cudaGraphExec_t e;
  CK(cudaGraphInstantiate(&e, g, 0));
  c->graphs.push_back(g);
  c->step_exec[n] = e;
  *ex = e;
  return LCA_OK;
}

int get_gen_exec(lca_ctx* c, int n, cudaGraphExec_t* ex) {
  auto it = c->gen_exec.find(n);
  if (it != c->gen_exec.end()) {
    *ex = it->second;
    return LCA_OK;
  }
  cudaGraph_t g;
  CK(cudaGraphCreate(&g, 0));
  cudaGraphConditionalHandle hw;
  CK(cudaGraphConditionalHandleCreate(&hw, g, 1, cudaGraphCondAssignDefault));
  cudaGraphNodeParams cp{};
  cp.type = cudaGraphNodeTypeConditional;
  cp.conditional.handle = hw;
  cp.conditional.type = cudaGraphCondTypeWhile;
  cp.conditional.size = 1;
  cudaGraphNode_t node;
  CK(cudaGraphAddNode(&node, g, nullptr, nullptr, 0, &cp));
  int st = capture_step(c, cp.conditional.phGraph_out[0], n, true, hw);
  if (st != LCA_OK) return st;
  cudaGraphExec_t e;
  CK(cudaGraphInstantiate(&e, g, 0));
  c->graphs.push_back(g);
  c->gen_exec[n] = e;
  *ex = e;
  return LCA_OK;
}

int read_err(lca_ctx* c) {
  int e = 0;
  CK(cudaMemcpyAsync(&e, c->L.D.err, sizeof(int), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  if (e) {
    CK(cudaMemsetAsync(c->L.D.err, 0, sizeof(int), c->stream));
    CK(cudaStreamSynchronize(c->stream));
  }
  if (e & ~15) fprintf(stderr, "lca: device error word 0x%x\n", e);
  if (e & kErrTimeout) return LCA_E_TIMEOUT;
  if (e & kErrNumeric) return LCA_E_NUMERIC;
  if (e & kErrPages) return LCA_E_CAPACITY;
  if (e & kErrIndex) return LCA_E_DEVICE_STATE;
  return LCA_OK;
}

struct WeightSpec {
  const void* ptr = nullptr;
  int64_t numel = 0;
  int dtype = 0;
};

int find_w(const std::map<std::string, WeightSpec>& m, const std::string& name, int64_t numel,
           int dtype, const void** out) {
  auto it = m.find(name);
  if (it == m.end() || !it->second.ptr) {
    fprintf(stderr, "lca: missing weight %s\n", name.c_str());
    return LCA_E_WEIGHTS;
  }
  if (it->second.numel != numel || it->second.dtype != dtype) {
    fprintf(stderr, "lca: weight %s has numel %lld dtype %d, expected %lld dtype %d\n", name.c_str(),
            (long long)it->second.numel, it->second.dtype, (long long)numel, dtype);
    return LCA_E_WEIGHTS;
  }
  *out = it->second.ptr;
  return LCA_OK;
}

int load_weights(lca_ctx* c, const lca_tensor* w, int nw) {
  std::map<std::string, WeightSpec> m;
  for (int i = 0; i < nw; ++i) {
    if (!w[i].name) return LCA_E_ARG;
    m[w[i].name] = WeightSpec{w[i].ptr, w[i].numel, w[i].dtype};
  }
  Dev& D = c->L.D;
  const int dt = c->cfg.dtype;
  const size_t tb = tw_bytes(dt);
  const int64_t d = D.d, F = D.F;
  cudaStream_t s = c->stream;
  const void* p;
  auto copy = [&](void* dst, const std::string& name, int64_t numel, int dtype) -> int {
    int st = find_w(m, name, numel, dtype, &p);
    if (st != LCA_OK) return st;
    CK(cudaMemcpyAsync(dst, p, numel * (dtype == LCA_BF16 ? 2 : 4), cudaMemcpyDeviceToDevice, s));
    return LCA_OK;
  };
#define TRY(x)                       \
  do {                               \
    int _s = (x);                    \
    if (_s != LCA_OK) return _s;     \
  } while (0)
  TRY(copy(D.embed, "embed", 256 * d, dt));
  TRY(copy(D.unembed, "unembed", 256 * d, dt));
  TRY(copy((void*)D.bos, "lm.bos", d, LCA_F32));
  TRY(copy((void*)D.nb_norm, "nb.norm", d, LCA_F32));
  TRY(copy((void*)D.mb_norm, "mb.norm", d, LCA_F32));
  auto stack = [&](std::vector<Block>& v, const char* pre) -> int {
    for (size_t l = 0; l < v.size(); ++l) {
      const std::string b = std::string(pre) + "." + std::to_string(l) + ".";
      Block& bk = v[l];
      TRY(copy((void*)bk.attn_norm, b + "attn_norm", d, LCA_F32));
      TRY(copy((void*)bk.mlp_norm, b + "mlp_norm", d, LCA_F32));
      TRY(copy((char*)bk.wqkv, b + "wq", d * d, dt));
      TRY(copy((char*)bk.wqkv + d * d * tb, b + "wk", d * d, dt));
      TRY(copy((char*)bk.wqkv + 2 * d * d * tb, b + "wv", d * d, dt));
      TRY(copy(bk.wo, b + "wo", d * d, dt));
      TRY(copy(bk.w2, b + "w2", d * F, dt));
      // interleave W1 and W3 rows: packed row 2j = W1_j, 2j+1 = W3_j
      TRY(find_w(m, b + "w1", F * d, dt, &p));
      launch_pack_rows(bk.w13, p, (int)F, (int)d, 0, 2, (int)tb, s);
      TRY(find_w(m, b + "w3", F * d, dt, &p));
      launch_pack_rows(bk.w13, p, (int)F, (int)d, 1, 2, (int)tb, s);
    }
    return LCA_OK;
  };
  TRY(stack(c->L.enc, "enc"));
  TRY(stack(c->L.lm, "lm"));
  TRY(stack(c->L.nb, "nb"));
  if (D.mb_kind == LCA_MB_LCA) {
    TRY(stack(c->L.mb, "mb"));
  } else {
    for (int l = 0; l < D.n_mb; ++l)
      for (int j = 0; j < D.n_mlp_heads; ++j)
        TRY(copy((char*)D.mlp_w + ((size_t)l * D.n_mlp_heads + j) * d * d * tb,
                 "mlp." + std::to_string(j) + "." + std::to_string(l) + ".w", d * d, dt));
  }
#undef TRY
  CK(cudaGetLastError());
  return LCA_OK;
}

}  // namespace

// ============================================================================ C ABI
extern "C" {

const char* lca_status_str(int s) {
  switch (s) {
    case LCA_OK: return "ok";
    case LCA_E_ARG: return "bad argument";
    case LCA_E_CAPACITY: return "capacity exceeded";
    case LCA_E_WEIGHTS: return "missing or malformed weights";
    case LCA_E_CUDA: return "CUDA error";
    case LCA_E_DEVICE_STATE: return "device index out of range";
    case LCA_E_NUMERIC: return "non-finite logits";
    case LCA_E_TIMEOUT: return "device wait timed out";
    case LCA_E_STATE: return "call out of order";
    default: return "unknown status";
  }
}

static size_t staging_bytes(const lca_config* c) {
  return ((size_t)c->max_batch * c->max_bytes + 255) / 256 * 256 + 4 * 256 +
         3 * (((size_t)c->max_batch * sizeof(int) + 255) / 256 * 256);
}

int lca_workspace_bytes(const lca_config* cfg, size_t* out) {
  int st = validate(cfg);
  if (st != LCA_OK) return st;
  if (!out) return LCA_E_ARG;
  Layout L;
  carve(*cfg, nullptr, L);
  *out = L.bytes + staging_bytes(cfg);
  return LCA_OK;
}

int lca_create(const lca_config* cfg, const lca_tensor* weights, int n_weights, void* workspace,
               size_t workspace_bytes, void* stream, lca_ctx** out) {
  int st = validate(cfg);
  if (st != LCA_OK) return st;
  if (!out || !workspace || !weights || n_weights <= 0) return LCA_E_ARG;
  if (reinterpret_cast<uintptr_t>(workspace) % 256) return LCA_E_ARG;
  size_t need = 0;
  lca_workspace_bytes(cfg, &need);
  if (workspace_bytes < need) return LCA_E_CAPACITY;
  lca_ctx* c = new lca_ctx();
  c->cfg = *cfg;
  c->ws = reinterpret_cast<char*>(workspace);
  c->ws_bytes = workspace_bytes;
  c->stream = reinterpret_cast<cudaStream_t>(stream);
  carve(*cfg, c->ws, c->L);
  {
    char* sb = c->ws + c->L.bytes;
    sb = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(sb) + 255) & ~uintptr_t(255));
    c->stg.bytes = reinterpret_cast<uint8_t*>(sb);
    sb += ((size_t)cfg->max_batch * cfg->max_bytes + 255) / 256 * 256 + 256;
    const size_t ib = ((size_t)cfg->max_batch * sizeof(int) + 255) / 256 * 256;
    c->stg.row0 = reinterpret_cast<int*>(sb);
    c->stg.lens = reinterpret_cast<int*>(sb + ib);
    c->stg.lm_row0 = reinterpret_cast<int*>(sb + 2 * ib);
  }
  auto fail = [&](int s) {
    lca_destroy(c);
    return s;
  };
  if (check(cudaStreamCreateWithFlags(&c->cap, cudaStreamNonBlocking), "stream") ||
      check(cudaStreamCreateWithFlags(&c->cap2, cudaStreamNonBlocking), "stream") ||
      check(cudaMallocHost(&c->h_params, sizeof(Params) * kParamSlots), "host params"))
    return fail(LCA_E_CUDA);
  kernel_attrs_linear();
  kernel_attrs_step();
  kernel_attrs_umma(&c->L.D);
  kernel_attrs_attn();
  Dev& D = c->L.D;
  {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    D.num_sms = sms > 0 ? sms : 148;
    const char* e = getenv("LCA_NO_TMA");
    D.use_tma = (e && e[0] == '1') ? 0 : 1;
    const char* um = getenv("LCA_NO_UMMA");
    D.use_umma = (um && um[0] == '1') ? 0 : 1;
    const char* sc = getenv("LCA_ATTN_SPLIT_CAP");
    D.attn_split_cap = sc ? std::max(1, std::min(16, atoi(sc))) : 16;
    const char* tr = getenv("LCA_TILED_MIN_ROWS");
    D.tiled_min_rows = tr ? std::max(0, atoi(tr)) : 32;
    const char* ap = getenv("LCA_ATTN_PIPE");
    D.attn_pipe = ap ? atoi(ap) : 2;
    const char* an = getenv("LCA_ATTN_NS");
    D.attn_ns = an ? atoi(an) : 8;
    const char* ant = getenv("LCA_ATTN_NS_T");
    D.attn_ns_t = ant ? atoi(ant) : 12;  // 12 stages: six compute warps (measured at batch 8-128)
    const char* atm = getenv("LCA_ATTN_TC_MIN");
    D.attn_tc_min = atm ? std::max(0, atoi(atm)) : 128;
    const char* gsw = getenv("LCA_GEMV_SPLIT");
    D.gemv_split = (gsw && gsw[0] == '0') ? 0 : 1;
    const char* kb = getenv("LCA_GEMV_KS_BIG");
    const char* ks = getenv("LCA_GEMV_KS_SMALL");
    auto pow2 = [](int v) { int p = 1; while (p * 2 <= v && p < kMaxKSplit) p *= 2; return p; };
    // measured at batch 1 and 32 (paper-size layers): a cluster reduction costs more than the
    // bandwidth of more CTAs buys for K = 1024 (Wo), and four ways are best for K = 4096 (W2)
    D.gemv_ks_big = kb ? pow2(std::max(2, atoi(kb))) : 4;
    D.gemv_ks_small = ks ? pow2(std::max(1, atoi(ks))) : 1;
    const char* sw = getenv("LCA_SPLIT_WRITE");
    D.split_write = (sw && sw[0] == '0') ? 0 : 1;
    const char* aw = getenv("LCA_ATTN_W");
    D.attn_w = (aw && aw[0] == '0') ? 0 : 1;
    const char* at = getenv("LCA_ATTN_T");
    D.attn_t = (at && at[0] == '0') ? 0 : 1;
    const char* mk = getenv("LCA_ATTN_MIN_KEYS");
    D.attn_min_keys = mk ? std::max(0, atoi(mk)) : 0;
    const char* pe = getenv("LCA_PERSIST");
    D.persist = (pe && pe[0] == '1') ? 1 : 0;
    D.stk_grid = D.num_sms;
    D.stk_splits = std::max(1, std::min(kMaxAttnSplit, D.num_sms / std::max(1, D.B * D.H)));
    if (D.stk_enc) kernel_attrs_stack(&D);
    else D.persist = 0;
  }
  // state and counters start at zero
  if (check(cudaMemsetAsync(c->ws, 0, c->L.bytes, c->stream), "memset")) return fail(LCA_E_CUDA);
  st = load_weights(c, weights, n_weights);
  if (st != LCA_OK) return fail(st);
  if (cfg->dtype == LCA_BF16) {
    auto add = [&](const void* W, long long rows, long long K) {
      TMapBlob blob;
      if (make_weight_tmap(blob.b, W, rows, K) == LCA_OK) c->tmaps[W] = blob;
    };
    for (auto* v : {&c->L.enc, &c->L.lm, &c->L.nb, &c->L.mb})
      for (auto& bk : *v) {
        add(bk.wqkv, 3LL * D.d, D.d);
        add(bk.wo, D.d, D.d);
        add(bk.w13, 2LL * D.F, D.d);
        add(bk.w2, D.d, D.F);
      }
    if (D.mlp_w)
      for (int l = 0; l < D.n_mb; ++l)
        add((char*)D.mlp_w + (size_t)l * D.n_mlp_heads * D.d * D.d * 2, (long long)D.n_mlp_heads * D.d, D.d);
    for (int K : {D.d, D.F})
      for (int buf = 0; buf < 2 && D.as_rows > 0; ++buf) {
        SplitMapBlob blob;
        if (make_split_tmaps(blob.b, D.as_hi[buf], D.as_lo[buf], D.as_rows, K) == LCA_OK)
          c->amaps[2 * K + buf] = blob;
      }
    if (D.hd == 64)
      for (auto* v : {&c->L.enc, &c->L.lm, &c->L.nb, &c->L.mb})
        for (auto& bk : *v) {
          SplitMapBlob blob;
          const long long rows = (long long)bk.kv.pages * D.H * kPage;
          // the kernels address rows with 32-bit coordinates
          if (rows <= 0x7fffffffLL && make_kv_tmaps(blob.b, bk.kv.k, bk.kv.v, rows) == LCA_OK) {
            c->kvmaps[bk.kv.k] = blob;
            bk.kv.tmaps = c->kvmaps[bk.kv.k].b;
          }
        }
  }
  if (D.stk_enc) {
    // the persistent stack kernel's view of each block
    auto table = [&](std::vector<Block>& v, StackLayer* dst) -> int {
      std::vector<StackLayer> h(v.size());
      for (size_t l = 0; l < v.size(); ++l) {
        h[l].wqkv = static_cast<const __nv_bfloat16*>(v[l].wqkv);
        h[l].wo = static_cast<const __nv_bfloat16*>(v[l].wo);
        h[l].w13 = static_cast<const __nv_bfloat16*>(v[l].w13);
        h[l].w2 = static_cast<const __nv_bfloat16*>(v[l].w2);
        h[l].attn_norm = v[l].attn_norm;
        h[l].mlp_norm = v[l].mlp_norm;
        h[l].k = v[l].kv.k;
        h[l].v = v[l].kv.v;
      }
      if (h.empty()) return LCA_OK;
      return check(cudaMemcpyAsync(dst, h.data(), sizeof(StackLayer) * h.size(), cudaMemcpyHostToDevice, c->stream),
                   "stack tables");
    };
    if (table(c->L.enc, D.stk_enc) || table(c->L.lm, D.stk_lm) || table(c->L.nb, D.stk_nb) ||
        table(c->L.mb, D.stk_mb) || check(cudaStreamSynchronize(c->stream), "stack tables"))
      return fail(LCA_E_CUDA);
  }
  launch_rope_table(D, cfg->rope_base, c->stream);
  if (check(cudaGetLastError(), "rope") || check(cudaStreamSynchronize(c->stream), "create sync"))
    return fail(LCA_E_CUDA);
  c->host_params = Params{};
  *out = c;
  return LCA_OK;
}

int lca_destroy(lca_ctx* c) {
  if (!c) return LCA_E_ARG;
  if (c->stream) cudaStreamSynchronize(c->stream);
  for (auto& kv : c->step_exec) cudaGraphExecDestroy(kv.second);
  for (auto& kv : c->gen_exec) cudaGraphExecDestroy(kv.second);
  for (auto g : c->graphs) cudaGraphDestroy(g);
  if (c->cap) cudaStreamDestroy(c->cap);
  if (c->cap2) cudaStreamDestroy(c->cap2);
  if (c->h_params) cudaFreeHost(c->h_params);
  delete c;
  return LCA_OK;
}

int lca_prefill(lca_ctx* c, int32_t batch, const uint8_t* const* prompts, const int32_t* lens) {
  if (!c || !prompts || !lens) return LCA_E_ARG;
  if (batch < 1 || batch > c->cfg.max_batch) return LCA_E_CAPACITY;
  Dev& D = c->L.D;
  cudaStream_t s = c->stream;
  std::vector<int> row0(batch), lm_row0(batch), K(batch);
  int M = 0, Mlm = 0, maxK = 0, maxlen = 0;
  for (int b = 0; b < batch; ++b) {
    if (!prompts[b] || lens[b] < 1) return LCA_E_ARG;
    if (lens[b] + c->cfg.max_n > c->cfg.max_bytes) return LCA_E_CAPACITY;
    row0[b] = M;
    M += lens[b];
    maxlen = std::max(maxlen, lens[b]);
    int k = 0;
    for (int p = 0; p < lens[b]; ++p) k += prompts[b][p] == c->cfg.boundary_byte;
    K[b] = k;
    maxK = std::max(maxK, k);
    lm_row0[b] = Mlm;
    Mlm += k + 1;
  }
  // host-built row descriptors (prompt structure is host data)
  std::vector<int> rb(M), rp(M), rs(M), rk(M), ss(D.B, M), sc(D.B, 0);
  std::vector<int> lb(Mlm), lp(Mlm), ls(D.B, Mlm), lc(D.B, 0);
  std::vector<uint8_t> bytes(M);
  for (int b = 0; b < batch; ++b) {
    ss[b] = row0[b];
    sc[b] = lens[b];
    for (int p = 0; p < lens[b]; ++p) {
      const int r = row0[b] + p;
      rb[r] = b;
      rp[r] = p;
      bytes[r] = prompts[b][p];
    }
    ls[b] = lm_row0[b];
    lc[b] = K[b] + 1;
    for (int k = 0; k <= K[b]; ++k) {
      lb[lm_row0[b] + k] = b;
      lp[lm_row0[b] + k] = k;
    }
  }
  std::vector<int> kv1(M), lkv1(Mlm);
  for (int r = 0; r < M; ++r) kv1[r] = rp[r] + 1;
  for (int r = 0; r < Mlm; ++r) lkv1[r] = lp[r] + 1;
  // pages of the prompts' positions and latents, in sequence order; those of later positions and
  // of the multi-byte windows are mapped by the decode steps
  std::vector<int> ptb((size_t)D.B * D.pt_ld_byte, -1), ptl((size_t)D.B * D.pt_ld_lm, -1),
      ptm((size_t)D.B * D.pt_ld_mb, -1);
  int npb = 0, npl = 0;
  for (int b = 0; b < batch; ++b) {
    for (int j = 0; j * kPage < lens[b]; ++j) ptb[(size_t)b * D.pt_ld_byte + j] = npb++;
    for (int j = 0; j * kPage < K[b] + 1; ++j) ptl[(size_t)b * D.pt_ld_lm + j] = npl++;
  }
  if (npb > D.pages_byte || npl > D.pages_lm) return LCA_E_CAPACITY;
  std::vector<int> rpg(M), lpg(Mlm);
  for (int r = 0; r < M; ++r) rpg[r] = ptb[(size_t)rb[r] * D.pt_ld_byte + rp[r] / kPage];
  for (int r = 0; r < Mlm; ++r) lpg[r] = ptl[(size_t)lb[r] * D.pt_ld_lm + lp[r] / kPage];
  const int pool_next[4] = {npb, npl, 0, 0};
  std::vector<int> last(batch);
  for (int b = 0; b < batch; ++b) last[b] = row0[b] + lens[b] - 1;
  auto up = [&](void* dst, const void* src, size_t n) {
    return check(cudaMemcpyAsync(dst, src, n, cudaMemcpyHostToDevice, s), "prefill upload");
  };
  if (up(c->stg.bytes, bytes.data(), M) || up(c->stg.row0, row0.data(), batch * 4) ||
      up(c->stg.lens, lens, batch * 4) || up(c->stg.lm_row0, lm_row0.data(), batch * 4) ||
      up(D.r_v.b, rb.data(), M * 4) || up(D.r_v.pos, rp.data(), M * 4) ||
      up(D.r_v.slot, rp.data(), M * 4) || up(D.r_v.page, rpg.data(), M * 4) || up(D.r_v.kvlen, kv1.data(), M * 4) ||
      up(D.r_v.seq_start, ss.data(), D.B * 4) || up(D.r_v.seq_count, sc.data(), D.B * 4) ||
      up(D.r_v.M, &M, 4) || up(D.r_lm.b, lb.data(), Mlm * 4) || up(D.r_lm.pos, lp.data(), Mlm * 4) ||
      up(D.r_lm.slot, lp.data(), Mlm * 4) || up(D.r_lm.page, lpg.data(), Mlm * 4) ||
      up(D.r_lm.kvlen, lkv1.data(), Mlm * 4) || up(D.pt_byte, ptb.data(), ptb.size() * 4) ||
      up(D.pt_lm, ptl.data(), ptl.size() * 4) || up(D.pt_mb, ptm.data(), ptm.size() * 4) ||
      up(D.pool_next, pool_next, sizeof(pool_next)) ||
      up(D.r_lm.seq_start, ls.data(), D.B * 4) || up(D.r_lm.seq_count, lc.data(), D.B * 4) ||
      up(D.r_lm.M, &Mlm, 4) || up(D.head_rows_v, last.data(), batch * 4) || up(D.M_head_v, &batch, 4))
    return LCA_E_CUDA;
  // inactive sequences
  {
    std::vector<SeqState> zs(D.B);
    for (auto& z : zs) memset(&z, 0, sizeof(z));
    if (up(D.seq, zs.data(), sizeof(SeqState) * D.B)) return LCA_E_CUDA;
  }
  const int qt = std::min(64, (maxlen + kAttnQT - 1) / kAttnQT);
  launch_prefill_embed(D, c->stg.bytes, M, s);
  run_stack(c, c->L.enc, D.x_enc, D.r_v, M, M, qt, 1, s);
  launch_prefill_segment(D, c->stg.bytes, c->stg.row0, c->stg.lens, batch, c->stg.lm_row0, s);
  launch_prefill_pool(D, c->stg.row0, c->stg.lens, c->stg.lm_row0, batch, maxK, s);
  const int lqt = std::min(64, (maxK + 1 + kAttnQT - 1) / kAttnQT);
  run_stack(c, c->L.lm, D.x_lm, D.r_lm, Mlm, Mlm, lqt, 1, s);
  launch_lm_scatter(D, s);
  launch_prefill_nb_input(D, M, s);
  run_stack(c, c->L.nb, D.x_nb, D.r_v, M, M, qt, 1, s);
  launch_head(D, D.x_nb, D.head_rows_v, D.M_head_v, batch, D.nb_norm, D.nb_logits, D.nb_arg,
              D.nb_prob, s);
  launch_prefill_finish(D, c->stg.row0, c->stg.lens, c->stg.lm_row0, batch, s);
  CK(cudaGetLastError());
  c->batch = batch;
  c->prefilled = true;
  c->t_host.assign(batch, 0);
  for (int b = 0; b < batch; ++b) c->t_host[b] = lens[b];
  c->host_params.batch = batch;
  c->pending_force_accept = c->pending_force_cand = 0;
  int e = read_err(c);
  if (e != LCA_OK) return e;
  // cache lengths for the attention key splits; step graphs captured for lengths more than twice
  // or less than half of these are dropped and captured again
  std::vector<SeqState> all(batch);
  CK(cudaMemcpy(all.data(), D.seq, sizeof(SeqState) * batch, cudaMemcpyDeviceToHost));
  int tb = 1, kl = 1;
  for (int b = 0; b < batch; ++b) {
    tb = std::max(tb, all[b].t);
    kl = std::max(kl, all[b].K);
  }
  auto far = [](int x, int y) { return x > 2 * y || y > 2 * x; };
  if (far(tb, c->kv_bytes_typ) || far(kl, c->kv_lat_typ)) drop_graphs(c);
  c->kv_bytes_typ = tb;
  c->kv_lat_typ = kl;
  return LCA_OK;
}

static int step_prep(lca_ctx* c, int n, float tau, int mode) {
  if (!c) return LCA_E_ARG;
  if (!c->prefilled) return LCA_E_STATE;
  if (n < 1 || n > c->cfg.max_n) return LCA_E_CAPACITY;
  if (mode != LCA_THRESH && mode != LCA_SPEC) return LCA_E_ARG;
  if (tau != tau) return LCA_E_ARG;
  Params& P = c->host_params;
  P.n = n;
  P.tau = tau;
  P.accept = mode;
  P.batch = c->batch;
  return LCA_OK;
}

int lca_mbp_step(lca_ctx* c, int32_t n, float tau, int32_t mode, uint8_t* out_bytes,
                 int32_t* out_counts) {
  int st = step_prep(c, n, tau, mode);
  if (st != LCA_OK) return st;
  for (int b = 0; b < c->batch; ++b)
    if (c->t_host[b] + n > c->cfg.max_bytes) return LCA_E_CAPACITY;
  if (c->pending_force_cand && c->pending_force_cand_n != n) return LCA_E_ARG;
  cudaGraphExec_t ex;
  st = get_step_exec(c, n, &ex);
  if (st != LCA_OK) return st;
  Params& P = c->host_params;
  P.gen = 0;
  P.force_accept = c->pending_force_accept;
  P.force_cand = c->pending_force_cand;
  st = upload_params(c);
  if (st != LCA_OK) return st;
  c->pending_force_accept = c->pending_force_cand = 0;
  if (c->eager) {
    st = run_step_eager(c, n);
    if (st != LCA_OK) return st;
  } else {
    CK(cudaGraphLaunch(ex, c->stream));
  }
  std::vector<int> cnt(c->batch);
  CK(cudaMemcpyAsync(cnt.data(), c->L.D.out_cnt, c->batch * sizeof(int), cudaMemcpyDeviceToHost,
                     c->stream));
  if (out_bytes)
    CK(cudaMemcpy2DAsync(out_bytes, n, c->L.D.out_step, c->L.D.NMAX, n, c->batch,
                         cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  c->last_n = n;
  for (int b = 0; b < c->batch; ++b) c->t_host[b] += cnt[b];
  if (out_counts) memcpy(out_counts, cnt.data(), c->batch * sizeof(int));
  return read_err(c);
}

int lca_mbp_step_async(lca_ctx* c, int32_t n, float tau, int32_t mode) {
  int st = step_prep(c, n, tau, mode);
  if (st != LCA_OK) return st;
  for (int b = 0; b < c->batch; ++b)
    if (c->t_host[b] + n > c->cfg.max_bytes) return LCA_E_CAPACITY;
  if (c->pending_force_cand && c->pending_force_cand_n != n) return LCA_E_ARG;
  cudaGraphExec_t ex;
  st = get_step_exec(c, n, &ex);
  if (st != LCA_OK) return st;
  Params& P = c->host_params;
  P.gen = 0;
  P.force_accept = c->pending_force_accept;
  P.force_cand = c->pending_force_cand;
  st = upload_params(c);
  if (st != LCA_OK) return st;
  c->pending_force_accept = c->pending_force_cand = 0;
  if (c->eager) {
    st = run_step_eager(c, n);
    if (st != LCA_OK) return st;
  } else {
    CK(cudaGraphLaunch(ex, c->stream));
  }
  c->last_n = n;
  for (int b = 0; b < c->batch; ++b) c->t_host[b] += n;  // upper bound until synced
  c->t_unsynced = true;
  return LCA_OK;
}

int lca_generate_async(lca_ctx* c, int32_t n, float tau, int32_t mode, int32_t max_new) {
  int st = step_prep(c, n, tau, mode);
  if (st != LCA_OK) return st;
  if (max_new < 1) return LCA_E_ARG;
  for (int b = 0; b < c->batch; ++b)
    if (c->t_host[b] + max_new + n > c->cfg.max_bytes) return LCA_E_CAPACITY;
  cudaGraphExec_t ex;
  st = get_gen_exec(c, n, &ex);
  if (st != LCA_OK) return st;
  Params& P = c->host_params;
  P.gen = 1;
  P.force_accept = 0;
  P.force_cand = 0;
  P.iter = 0;
  P.max_iter = max_new;
  st = upload_params(c);
  if (st != LCA_OK) return st;
  launch_gen_init(c->L.D, max_new, c->stream);
  CK(cudaGetLastError());
  CK(cudaGraphLaunch(ex, c->stream));
  c->gen_max_new = max_new;
  c->gen_n = n;
  c->last_n = n;
  for (int b = 0; b < c->batch; ++b) c->t_host[b] += max_new;
  return LCA_OK;
}

int lca_generate_fetch(lca_ctx* c, uint8_t* out, int32_t* out_len, int32_t* hist) {
  if (!c) return LCA_E_ARG;
  if (!c->gen_max_new) return LCA_E_STATE;
  Dev& D = c->L.D;
  const int mx = c->gen_max_new;
  if (out)
    CK(cudaMemcpy2DAsync(out, mx, D.out_gen, D.S, mx, c->batch, cudaMemcpyDeviceToHost, c->stream));
  std::vector<SeqState> ss(c->batch);
  CK(cudaMemcpyAsync(ss.data(), D.seq, sizeof(SeqState) * c->batch, cudaMemcpyDeviceToHost, c->stream));
  std::vector<int> h(D.NMAX);
  CK(cudaMemcpyAsync(h.data(), D.hist, sizeof(int) * D.NMAX, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  int st = LCA_OK;
  for (int b = 0; b < c->batch; ++b) {
    if (out_len) out_len[b] = ss[b].generated;
    if (ss[b].generated != mx) st = LCA_E_DEVICE_STATE;
  }
  if (hist) memcpy(hist, h.data(), sizeof(int) * c->gen_n);
  int e = read_err(c);
  return e != LCA_OK ? e : st;
}

int lca_generate(lca_ctx* c, int32_t n, float tau, int32_t mode, int32_t max_new, uint8_t* out,
                 int32_t* out_len, int32_t* hist) {
  int st = lca_generate_async(c, n, tau, mode, max_new);
  if (st != LCA_OK) return st;
  return lca_generate_fetch(c, out, out_len, hist);
}

int lca_debug_state(lca_ctx* c, int32_t b, lca_seq_state* out) {
  if (!c || !out) return LCA_E_ARG;
  if (!c->prefilled) return LCA_E_STATE;
  if (b < 0 || b >= c->batch) return LCA_E_ARG;
  Dev& D = c->L.D;
  SeqState s;
  CK(cudaMemcpyAsync(&s, D.seq + b, sizeof(s), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  if (c->t_unsynced) {
    std::vector<SeqState> all(c->batch);
    CK(cudaMemcpy(all.data(), D.seq, sizeof(SeqState) * c->batch, cudaMemcpyDeviceToHost));
    for (int i = 0; i < c->batch; ++i) c->t_host[i] = all[i].t;
    c->t_unsynced = false;
  }
  int g[2] = {-1, 0};
  if (s.K >= 1)
    CK(cudaMemcpyAsync(&g[0], D.gstart + (size_t)b * D.L + s.K - 1, 4, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaMemcpyAsync(&g[1], D.gstart + (size_t)b * D.L + s.K, 4, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  out->t = s.t;
  out->K = s.K;
  out->open_start = s.open_start;
  out->prev_group_start = g[0];
  out->group_start = g[1];
  out->next_byte = s.next_c1;
  out->generated = s.generated;
  out->pad = 0;
  return LCA_OK;
}

int lca_debug_logits(lca_ctx* c, float* nb, float* mb) {
  if (!c) return LCA_E_ARG;
  if (!c->last_n) return LCA_E_STATE;
  const int n = c->last_n;
  Dev& D = c->L.D;
  if (nb)
    CK(cudaMemcpyAsync(nb, D.nb_logits, sizeof(float) * 256 * c->batch * n, cudaMemcpyDeviceToHost,
                       c->stream));
  if (mb && n >= 2)
    CK(cudaMemcpyAsync(mb, D.mb_logits, sizeof(float) * 256 * c->batch * (n - 1),
                       cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  return LCA_OK;
}

int lca_debug_stats(lca_ctx* c, lca_stats* out) {
  if (!c || !out) return LCA_E_ARG;
  Stats s;
  CK(cudaMemcpyAsync(&s, c->L.D.stats, sizeof(s), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  out->steps = (int64_t)s.steps;
  out->lm_steps = (int64_t)s.lm_steps;
  out->lm_rows = (int64_t)s.lm_rows;
  out->mb_rows = (int64_t)s.mb_rows;
  out->committed = (int64_t)s.committed;
  auto it = c->launches.find(c->last_n);
  out->kernels_per_step = it == c->launches.end() ? 0 : it->second.first;
  out->kernels_per_lm_run = it == c->launches.end() ? 0 : it->second.second;
  out->workspace_bytes = (int64_t)c->ws_bytes;
  return LCA_OK;
}

int lca_debug_step_log(lca_ctx* c, int64_t first, int32_t count, uint8_t* out) {
  if (!c || !out || count < 0 || first < 0) return LCA_E_ARG;
  Stats s;
  CK(cudaMemcpyAsync(&s, c->L.D.stats, sizeof(s), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  const long long steps = (long long)s.steps;
  if (first + count > steps || steps - first > kStepLog) return LCA_E_ARG;
  std::vector<uint8_t> ring(kStepLog);
  CK(cudaMemcpy(ring.data(), c->L.D.step_log, kStepLog, cudaMemcpyDeviceToHost));
  for (int i = 0; i < count; ++i) out[i] = ring[(size_t)((first + i) % kStepLog)];
  return LCA_OK;
}

int lca_debug_accept_hist(lca_ctx* c, int32_t* out, int32_t reset) {
  if (!c) return LCA_E_ARG;
  Dev& D = c->L.D;
  if (out) CK(cudaMemcpyAsync(out, D.hist, sizeof(int) * D.NMAX, cudaMemcpyDeviceToHost, c->stream));
  if (reset) CK(cudaMemsetAsync(D.hist, 0, sizeof(int) * D.NMAX, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  return LCA_OK;
}

int lca_debug_page_table(lca_ctx* c, int32_t cache, int32_t* out, int64_t cap, int32_t* row_len, int32_t* used,
                         int32_t* pages) {
  if (!c || !row_len || !used || !pages || cache < 0 || cache > 2) return LCA_E_ARG;
  Dev& D = c->L.D;
  const int* pt = cache == 0 ? D.pt_byte : cache == 1 ? D.pt_lm : D.pt_mb;
  const int ld = cache == 0 ? D.pt_ld_byte : cache == 1 ? D.pt_ld_lm : D.pt_ld_mb;
  const int np = cache == 0 ? D.pages_byte : cache == 1 ? D.pages_lm : D.pages_mb;
  *row_len = ld;
  *pages = np;
  const size_t n = (size_t)D.B * ld;
  if (!out || cap < (int64_t)n) return LCA_E_CAPACITY;
  int next[4];
  CK(cudaMemcpyAsync(out, pt, n * 4, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaMemcpyAsync(next, D.pool_next, sizeof(next), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  *used = std::min(next[cache], np);
  return LCA_OK;
}

int lca_debug_set_eager(lca_ctx* c, int32_t on) {
  if (!c) return LCA_E_ARG;
  c->eager = on != 0;
  return LCA_OK;
}

int lca_debug_profile(lca_ctx* c, int32_t n, float tau, int32_t mode, int32_t steps,
                      lca_profile* out) {
  if (!out || steps < 1) return LCA_E_ARG;
  int st = step_prep(c, n, tau, mode);
  if (st != LCA_OK) return st;
  for (int b = 0; b < c->batch; ++b)
    if (c->t_host[b] + (long long)steps * n > c->cfg.max_bytes) return LCA_E_CAPACITY;
  Params& P = c->host_params;
  P.gen = 0;
  P.force_accept = 0;
  P.force_cand = 0;
  Profiler prof;
  for (int i = 0; i < steps; ++i) {
    st = upload_params(c);
    if (st != LCA_OK) return st;
    g_prof = &prof;
    st = run_step_eager(c, n);
    g_prof = nullptr;
    if (st != LCA_OK) return st;
    prof.collect();
  }
  c->last_n = n;
  std::vector<SeqState> all(c->batch);
  CK(cudaMemcpyAsync(all.data(), c->L.D.seq, sizeof(SeqState) * c->batch, cudaMemcpyDeviceToHost,
                     c->stream));
  CK(cudaStreamSynchronize(c->stream));
  for (int i = 0; i < c->batch; ++i) c->t_host[i] = all[i].t;
  for (int k = 0; k < PK_COUNT && k < 4; ++k) {
    out->launches[k] = prof.launches[k];
    out->ms[k] = prof.ms[k];
    out->bytes[k] = prof.bytes[k];
  }
  return read_err(c);
}

int lca_debug_bench_kernel(lca_ctx* c, int32_t kind, int32_t rows, int32_t iters, double* us,
                           double* bytes) {
  if (!c || !us || !bytes || iters < 1 || rows < 1) return LCA_E_ARG;
  if (!c->prefilled) return LCA_E_STATE;
  Dev& D = c->L.D;
  if (rows > std::min(D.R, 64)) return LCA_E_CAPACITY;
  std::vector<Block*> blocks;
  for (auto* v : {&c->L.enc, &c->L.lm, &c->L.nb, &c->L.mb})
    for (auto& b : *v) blocks.push_back(&b);
  if (blocks.empty()) return LCA_E_STATE;
  const double tb = tw_bytes(D.dtype);
  // rows [0, rows) of x_enc feed the kernels; r_v describes them (sequence 0, positions 0..)
  std::vector<int> z(rows, 0), pos(rows), kvl(rows);
  for (int i = 0; i < rows; ++i) {
    pos[i] = i;
    kvl[i] = std::min(c->t_host.empty() ? 1 : (int)c->t_host[0], D.S);
  }
  std::vector<int> ss(D.B, rows), sc(D.B, 0);
  ss[0] = 0;
  sc[0] = rows;
  cudaStream_t s = c->stream;
  CK(cudaMemcpyAsync(D.r_v.b, z.data(), rows * 4, cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(D.r_v.pos, pos.data(), rows * 4, cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(D.r_v.slot, pos.data(), rows * 4, cudaMemcpyHostToDevice, s));
  // slots [0, rows) of sequence 0 lie in its first page (rows <= 64), mapped by the prefill
  std::vector<int> pg0(rows);
  CK(cudaMemcpyAsync(pg0.data(), D.pt_byte, 4, cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  for (int i = 1; i < rows; ++i) pg0[i] = pg0[0];
  CK(cudaMemcpyAsync(D.r_v.page, pg0.data(), rows * 4, cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(D.r_v.kvlen, kvl.data(), rows * 4, cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(D.r_v.seq_start, ss.data(), D.B * 4, cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(D.r_v.seq_count, sc.data(), D.B * 4, cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(D.r_v.M, &rows, 4, cudaMemcpyHostToDevice, s));
  CK(cudaStreamSynchronize(s));
  double by = 0;
  cudaGraph_t g;
  CK(cudaStreamBeginCapture(c->cap, cudaStreamCaptureModeRelaxed));
  for (int i = 0; i < iters; ++i) {
    Block& bk = *blocks[i % blocks.size()];
    LinearArgs a{};
    a.groups = 1;
    a.eps = D.eps;
    a.M = D.r_v.M;
    a.M_cap = rows;
    a.x = D.x_enc;
    a.ldx = D.d;
    a.epi.mode = EPI_STORE;
    a.epi.y = D.mid;
    a.epi.ldy = 3 * D.d;
    a.epi.err = D.err;
    switch (kind) {
      case 0:  // RMSNorm + QKV (stored, no cache write)
        a.W = bk.wqkv; a.N = 3 * D.d; a.Kd = D.d; a.norm = bk.attn_norm;
        linear(D, a, false, c->cap);
        by = (double)a.N * a.Kd * tb;
        break;
      case 1:  // Wo
        a.W = bk.wo; a.N = D.d; a.Kd = D.d;
        linear(D, a, false, c->cap);
        by = (double)a.N * a.Kd * tb;
        break;
      case 2:  // RMSNorm + W1/W3 + SwiGLU
        a.W = bk.w13; a.N = 2 * D.F; a.Kd = D.d; a.norm = bk.mlp_norm;
        a.epi.mode = EPI_SWIGLU; a.epi.ldy = D.F;
        linear(D, a, false, c->cap);
        by = (double)a.N * a.Kd * tb;
        break;
      case 3:  // W2
        a.x = D.mid; a.ldx = D.F; a.W = bk.w2; a.N = D.d; a.Kd = D.F;
        a.epi.ldy = D.d; a.epi.y = D.att;
        linear(D, a, false, c->cap);
        by = (double)a.N * a.Kd * tb;
        break;
      case 4: {  // attention over the encoder cache of layer (i % n_enc)
        Block& eb = c->L.enc[i % c->L.enc.size()];
        attention(D, D.qbuf, D.att, eb.kv, D.r_v, D.B, 1, attn_splits(D, D.B, 1, kvl[0]), c->cap);
        by = 2.0 * D.H * (double)kvl[0] * D.hd * tb;
        break;
      }
      case 5:  // unembedding head
        launch_head(D, D.x_enc, nullptr, D.r_v.M, rows, D.nb_norm, D.nb_logits, D.nb_arg, D.nb_prob, c->cap);
        by = 256.0 * D.d * tb;
        break;
      default:  // a glue kernel (upsampling input of the next-byte decoder)
        launch_lm_scatter(D, c->cap);
        by = 0;
        break;
    }
  }
  CK(cudaStreamEndCapture(c->cap, &g));
  cudaGraphExec_t ex;
  CK(cudaGraphInstantiate(&ex, g, 0));
  cudaEvent_t e0, e1;
  CK(cudaEventCreate(&e0));
  CK(cudaEventCreate(&e1));
  for (int w = 0; w < 2; ++w) CK(cudaGraphLaunch(ex, s));
  CK(cudaEventRecord(e0, s));
  const int reps = 5;
  for (int r = 0; r < reps; ++r) CK(cudaGraphLaunch(ex, s));
  CK(cudaEventRecord(e1, s));
  CK(cudaEventSynchronize(e1));
  float ms = 0;
  CK(cudaEventElapsedTime(&ms, e0, e1));
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  cudaGraphExecDestroy(ex);
  cudaGraphDestroy(g);
  *us = ms * 1000.0 / (reps * iters);
  *bytes = by;
  c->prefilled = false;  // the row descriptors were overwritten: prefill again before stepping
  return read_err(c);
}

int lca_debug_trace(lca_ctx* c, int32_t n, float tau, int32_t mode, int32_t steps, void* out,
                    int32_t cap, int32_t* count) {
  if (!out || !count || cap < 1 || steps < 1) return LCA_E_ARG;
  int st = step_prep(c, n, tau, mode);
  if (st != LCA_OK) return st;
  for (int b = 0; b < c->batch; ++b)
    if (c->t_host[b] + (long long)steps * n > c->cfg.max_bytes) return LCA_E_CAPACITY;
  cudaGraphExec_t ex;
  st = get_step_exec(c, n, &ex);
  if (st != LCA_OK) return st;
  // the trace buffer borrows the split-K scratch (unused by the bf16 step)
  Dev& D = c->L.D;
  const size_t rec_cap = D.lin_part_floats * sizeof(float) / sizeof(TraceRec);
  const unsigned capu = (unsigned)std::min<size_t>(rec_cap, (size_t)cap);
  if (capu == 0) return LCA_E_CAPACITY;
  TraceRec* buf = reinterpret_cast<TraceRec*>(D.lin_part);
  unsigned* counter = reinterpret_cast<unsigned*>(D.lin_cnt);
  CK(cudaMemsetAsync(counter, 0, sizeof(unsigned), c->stream));
  CK(cudaStreamSynchronize(c->stream));
  trace_set_linear(buf, counter, capu);
  trace_set_attn(buf, counter, capu);
  trace_set_step(buf, counter, capu);
  trace_set_umma(buf, counter, capu);
  trace_set_stack(buf, counter, capu);
  Params& P = c->host_params;
  P.gen = 0;
  P.force_accept = 0;
  P.force_cand = 0;
  st = upload_params(c);
  if (st != LCA_OK) return st;
  for (int i = 0; i < steps; ++i) CK(cudaGraphLaunch(ex, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  trace_set_linear(nullptr, nullptr, 0);
  trace_set_attn(nullptr, nullptr, 0);
  trace_set_step(nullptr, nullptr, 0);
  trace_set_umma(nullptr, nullptr, 0);
  trace_set_stack(nullptr, nullptr, 0);
  unsigned got = 0;
  CK(cudaMemcpy(&got, counter, sizeof(unsigned), cudaMemcpyDeviceToHost));
  got = std::min(got, capu);
  CK(cudaMemcpy(out, buf, sizeof(TraceRec) * got, cudaMemcpyDeviceToHost));
  CK(cudaMemset(counter, 0, sizeof(unsigned)));
  *count = (int32_t)got;
  c->last_n = n;
  std::vector<SeqState> all(c->batch);
  CK(cudaMemcpy(all.data(), D.seq, sizeof(SeqState) * c->batch, cudaMemcpyDeviceToHost));
  for (int i = 0; i < c->batch; ++i) c->t_host[i] = all[i].t;
  return read_err(c);
}

int lca_debug_force_accept(lca_ctx* c, const int32_t* a) {
  if (!c) return LCA_E_ARG;
  if (!c->prefilled) return LCA_E_STATE;
  if (!a) {
    c->pending_force_accept = 0;
    return LCA_OK;
  }
  CK(cudaMemcpyAsync(c->L.D.forced_a, a, sizeof(int) * c->batch, cudaMemcpyHostToDevice, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  c->pending_force_accept = 1;
  return LCA_OK;
}

int lca_debug_force_candidates(lca_ctx* c, const uint8_t* cand, int32_t n) {
  if (!c) return LCA_E_ARG;
  if (!c->prefilled) return LCA_E_STATE;
  if (!cand) {
    c->pending_force_cand = 0;
    return LCA_OK;
  }
  if (n < 1 || n > c->cfg.max_n) return LCA_E_CAPACITY;
  Dev& D = c->L.D;
  std::vector<int> v((size_t)D.B * D.NMAX, 0);
  for (int b = 0; b < c->batch; ++b)
    for (int i = 0; i < n; ++i) v[(size_t)b * D.NMAX + i] = cand[(size_t)b * n + i];
  CK(cudaMemcpyAsync(D.forced_cand, v.data(), sizeof(int) * v.size(), cudaMemcpyHostToDevice, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  c->pending_force_cand = 1;
  c->pending_force_cand_n = n;
  return LCA_OK;
}

}  // extern "C"
