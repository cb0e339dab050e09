"""Thin ctypes binding of ``include/lca.h``: argument marshalling only.

Every step of the decode path runs in the CUDA library ``liblca.so``; torch provides the
device memory (workspace, weights) and the stream. There is no CPU fallback: if the
library is missing, loading raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liblca.so")

LCA_OK = 0
LCA_F32, LCA_BF16 = 0, 1
LCA_MB_LCA, LCA_MB_MLP = 0, 1
LCA_THRESH, LCA_SPEC = 0, 1
LCA_E_ARG, LCA_E_CAPACITY, LCA_E_DEVICE_STATE, LCA_E_TIMEOUT = -1, -2, -5, -7

STATUS = {0: "LCA_OK", -1: "LCA_E_ARG", -2: "LCA_E_CAPACITY", -3: "LCA_E_WEIGHTS", -4: "LCA_E_CUDA",
          -5: "LCA_E_DEVICE_STATE", -6: "LCA_E_NUMERIC", -7: "LCA_E_TIMEOUT", -8: "LCA_E_STATE"}

EXPORTS = ("lca_workspace_bytes", "lca_create", "lca_prefill", "lca_mbp_step", "lca_mbp_step_async",
           "lca_generate",
           "lca_generate_async", "lca_generate_fetch", "lca_debug_state", "lca_debug_stats",
           "lca_debug_set_eager", "lca_debug_profile", "lca_debug_bench_kernel", "lca_debug_trace",
           "lca_debug_logits",
           "lca_debug_force_accept", "lca_debug_force_candidates", "lca_destroy", "lca_status_str",
           "lca_debug_gemm", "lca_debug_gemm_scratch_bytes", "lca_debug_attn_diag",
           "lca_decode_attention_scratch_bytes", "lca_decode_attention", "lca_decode_attention_noalloc",
           "lca_decode_attention_noalloc_capacity", "lca_decode_attention_status",
           "lca_decode_attention_noalloc_status", "lca_debug_set_wait_spins",
           "lca_debug_step_log", "lca_debug_accept_hist", "lca_debug_page_table")


class LcaConfig(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("d_ff", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("n_enc", ctypes.c_int32), ("n_lm", ctypes.c_int32), ("n_nb", ctypes.c_int32),
                ("n_mb", ctypes.c_int32), ("mb_kind", ctypes.c_int32), ("n_mlp_heads", ctypes.c_int32),
                ("boundary_byte", ctypes.c_int32), ("rope_base", ctypes.c_float),
                ("rms_eps", ctypes.c_float), ("attn_scale", ctypes.c_float), ("dtype", ctypes.c_int32),
                ("max_batch", ctypes.c_int32), ("max_bytes", ctypes.c_int32), ("max_n", ctypes.c_int32),
                ("kv_pages", ctypes.c_int32), ("lm_pages", ctypes.c_int32), ("mb_pages", ctypes.c_int32)]


class LcaTensor(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("ptr", ctypes.c_void_p), ("numel", ctypes.c_int64),
                ("dtype", ctypes.c_int32)]


class LcaSeqState(ctypes.Structure):
    _fields_ = [("t", ctypes.c_int32), ("K", ctypes.c_int32), ("open_start", ctypes.c_int32),
                ("prev_group_start", ctypes.c_int32), ("group_start", ctypes.c_int32),
                ("next_byte", ctypes.c_int32), ("generated", ctypes.c_int32), ("pad", ctypes.c_int32)]


class LcaStats(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int64) for f in ("steps", "lm_steps", "lm_rows", "mb_rows", "committed",
                                              "kernels_per_step", "kernels_per_lm_run",
                                              "workspace_bytes")]


class LcaProfile(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64 * 4), ("ms", ctypes.c_double * 4), ("bytes", ctypes.c_double * 4)]


PROFILE_KINDS = ("linear", "attention", "head", "glue")


class LcaError(RuntimeError):
    def __init__(self, status, what):
        super().__init__(f"{what}: {STATUS.get(status, status)}")
        self.status = status


_lib = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load liblca.so (raises OSError when it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise OSError(f"CUDA library not built: {path} (run paper_2608_15454_gb300/build.py)")
    lib = ctypes.CDLL(path)
    P, I32, F32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_float
    sig = {
        "lca_workspace_bytes": [ctypes.POINTER(LcaConfig), ctypes.POINTER(ctypes.c_size_t)],
        "lca_create": [ctypes.POINTER(LcaConfig), ctypes.POINTER(LcaTensor), ctypes.c_int, P,
                       ctypes.c_size_t, P, ctypes.POINTER(P)],
        "lca_prefill": [P, I32, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(I32)],
        "lca_mbp_step": [P, I32, F32, I32, P, P],
        "lca_mbp_step_async": [P, I32, F32, I32],
        "lca_generate": [P, I32, F32, I32, I32, P, P, P],
        "lca_generate_async": [P, I32, F32, I32, I32],
        "lca_generate_fetch": [P, P, P, P],
        "lca_debug_state": [P, I32, ctypes.POINTER(LcaSeqState)],
        "lca_debug_stats": [P, ctypes.POINTER(LcaStats)],
        "lca_debug_logits": [P, P, P],
        "lca_debug_set_eager": [P, I32],
        "lca_debug_trace": [P, I32, F32, I32, I32, P, I32, ctypes.POINTER(I32)],
        "lca_debug_bench_kernel": [P, I32, I32, I32, ctypes.POINTER(ctypes.c_double),
                                   ctypes.POINTER(ctypes.c_double)],
        "lca_debug_profile": [P, I32, F32, I32, I32, ctypes.POINTER(LcaProfile)],
        "lca_debug_force_accept": [P, P],
        "lca_debug_force_candidates": [P, P, I32],
        "lca_destroy": [P],
        "lca_status_str": [ctypes.c_int],
        "lca_debug_gemm": [P, P, P, I32, I32, I32, P, I32, P, P, P],
        "lca_debug_gemm_scratch_bytes": [I32, I32],
        "lca_debug_attn_diag": [P],
        "lca_decode_attention_scratch_bytes": [I32, I32, I32, I32, ctypes.POINTER(ctypes.c_size_t)],
        "lca_decode_attention": [P, P, P, P, I32, I32, I32, I32, I32, I32, P, F32, I32, P,
                                 ctypes.c_size_t, P],
        "lca_decode_attention_noalloc": [P, P, P, P, I32, I32, I32, I32, I32, I32, P, F32, I32, P],
        "lca_decode_attention_noalloc_capacity": [],
        "lca_decode_attention_status": [P, P],
        "lca_decode_attention_noalloc_status": [P],
        "lca_debug_set_wait_spins": [I32],
        "lca_debug_step_log": [P, ctypes.c_int64, I32, P],
        "lca_debug_accept_hist": [P, P, I32],
        "lca_debug_page_table": [P, I32, P, ctypes.c_int64, P, P, P],
    }
    for name, args in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = (ctypes.c_char_p if name == "lca_status_str" else
                     ctypes.c_size_t if name in ("lca_decode_attention_noalloc_capacity",
                                                 "lca_debug_gemm_scratch_bytes") else ctypes.c_int)
    _lib = lib
    return lib


def make_config(model, max_batch: int, max_bytes: int, max_n: int, kv_pages: int = 0,
                lm_pages: int = 0, mb_pages: int = 0) -> LcaConfig:
    """lca_config from a synth.ModelConfig (kv_pages, lm_pages, mb_pages: pages of 64 slots in
    each byte-cache, LM-cache and window-cache layer's pool, 0 = enough for every sequence at
    max_bytes)."""
    return LcaConfig(model.d_model, model.n_heads, model.head_dim, model.d_ff, model.vocab,
                     model.n_enc, model.n_lm, model.n_nb, model.n_mb,
                     LCA_MB_MLP if model.mb_kind == "mlp" else LCA_MB_LCA, model.n_mlp_heads,
                     model.boundary_byte, model.rope_base, model.rms_eps, model.attn_scale,
                     LCA_BF16 if model.dtype == "bf16" else LCA_F32, max_batch, max_bytes, max_n,
                     kv_pages, lm_pages, mb_pages)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


class Context:
    """One lca_ctx: weights and workspace on a CUDA device, prompts and outputs on the host."""

    def __init__(self, model, weights: dict, max_batch: int, max_bytes: int, max_n: int,
                 device: str = "cuda", stream=None, kv_pages: int = 0, lm_pages: int = 0,
                 mb_pages: int = 0):
        import torch
        self.torch = torch
        self.lib = load_library()
        self.model = model
        self.device = torch.device(device)
        self.max_n = max_n
        self.cfg = make_config(model, max_batch, max_bytes, max_n, kv_pages, lm_pages, mb_pages)
        wdt = torch.bfloat16 if model.dtype == "bf16" else torch.float32
        self._weights = {}
        tensors = []
        for name, a in weights.items():
            is_f32 = name.endswith("norm") or name == "lm.bos"
            t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(self.device)
            t = t if is_f32 else t.to(wdt)
            t = t.contiguous()
            self._weights[name] = t
            tensors.append(LcaTensor(name.encode(), t.data_ptr(), t.numel(),
                                     LCA_F32 if (is_f32 or wdt == torch.float32) else LCA_BF16))
        arr = (LcaTensor * len(tensors))(*tensors)
        nbytes = ctypes.c_size_t(0)
        self._check(self.lib.lca_workspace_bytes(ctypes.byref(self.cfg), ctypes.byref(nbytes)),
                    "lca_workspace_bytes")
        self.workspace_bytes = nbytes.value
        self._ws = torch.empty(self.workspace_bytes + 256, dtype=torch.uint8, device=self.device)
        base = (self._ws.data_ptr() + 255) // 256 * 256
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        h = ctypes.c_void_p()
        self._check(self.lib.lca_create(ctypes.byref(self.cfg), arr, len(tensors), base,
                                        self.workspace_bytes, self.stream.cuda_stream, ctypes.byref(h)),
                    "lca_create")
        self.h = h
        self.batch = 0
        del self._weights  # repacked into the workspace

    def _check(self, st, what):
        if st != LCA_OK:
            raise LcaError(st, what)

    def close(self):
        if getattr(self, "h", None):
            self.lib.lca_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ------------------------------------------------------------------ calls
    def prefill(self, prompts):
        n = len(prompts)
        bufs = [ctypes.c_char_p(bytes(p)) for p in prompts]
        arr = (ctypes.c_char_p * n)(*bufs)
        lens = (ctypes.c_int32 * n)(*[len(p) for p in prompts])
        self._check(self.lib.lca_prefill(self.h, n, arr, lens), "lca_prefill")
        self.batch = n

    def step(self, n, tau, mode=LCA_THRESH):
        out = np.zeros((self.batch, n), dtype=np.uint8)
        cnt = np.zeros(self.batch, dtype=np.int32)
        self._check(self.lib.lca_mbp_step(self.h, n, tau, mode, _ptr(out), _ptr(cnt)), "lca_mbp_step")
        return [bytes(out[b, :cnt[b]]) for b in range(self.batch)], cnt

    def step_async(self, n, tau, mode=LCA_THRESH):
        self._check(self.lib.lca_mbp_step_async(self.h, n, tau, mode), "lca_mbp_step_async")

    def generate(self, n, tau, mode, max_new):
        out = np.zeros((self.batch, max_new), dtype=np.uint8)
        ln = np.zeros(self.batch, dtype=np.int32)
        hist = np.zeros(n, dtype=np.int32)
        self._check(self.lib.lca_generate(self.h, n, tau, mode, max_new, _ptr(out), _ptr(ln), _ptr(hist)),
                    "lca_generate")
        return [bytes(out[b, :ln[b]]) for b in range(self.batch)], hist

    def generate_async(self, n, tau, mode, max_new):
        self._check(self.lib.lca_generate_async(self.h, n, tau, mode, max_new), "lca_generate_async")
        self._gen = (n, max_new)

    def generate_fetch(self):
        n, max_new = self._gen
        out = np.zeros((self.batch, max_new), dtype=np.uint8)
        ln = np.zeros(self.batch, dtype=np.int32)
        hist = np.zeros(n, dtype=np.int32)
        self._check(self.lib.lca_generate_fetch(self.h, _ptr(out), _ptr(ln), _ptr(hist)),
                    "lca_generate_fetch")
        return [bytes(out[b, :ln[b]]) for b in range(self.batch)], hist

    def state(self, b):
        s = LcaSeqState()
        self._check(self.lib.lca_debug_state(self.h, b, ctypes.byref(s)), "lca_debug_state")
        return {f: getattr(s, f) for f, _ in LcaSeqState._fields_ if f != "pad"}

    def stats(self):
        s = LcaStats()
        self._check(self.lib.lca_debug_stats(self.h, ctypes.byref(s)), "lca_debug_stats")
        return {f: getattr(s, f) for f, _ in LcaStats._fields_}

    def step_log(self, first, count):
        """1 per decode step [first, first + count) that ran the LM module, else 0."""
        out = np.zeros(max(count, 1), dtype=np.uint8)
        self._check(self.lib.lca_debug_step_log(self.h, first, count, _ptr(out)), "lca_debug_step_log")
        return out[:count]

    def accept_hist(self, reset=False):
        """Steps (summed over sequences) by accepted drafts since the last reset, [max_n]."""
        out = np.zeros(self.max_n, dtype=np.int32)
        self._check(self.lib.lca_debug_accept_hist(self.h, _ptr(out), 1 if reset else 0), "lca_debug_accept_hist")
        return out

    def page_table(self, cache):
        """(table [max_batch][row_len] of pool pages or -1, pages mapped, pool pages) of cache kind
        0 (byte positions), 1 (LM latents) or 2 (multi-byte windows)."""
        ld, used, pages = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        self.lib.lca_debug_page_table(self.h, cache, None, 0, ctypes.byref(ld), ctypes.byref(used),
                                      ctypes.byref(pages))
        out = np.zeros(self.cfg.max_batch * ld.value, dtype=np.int32)
        self._check(self.lib.lca_debug_page_table(self.h, cache, _ptr(out), out.size, ctypes.byref(ld),
                                                  ctypes.byref(used), ctypes.byref(pages)),
                    "lca_debug_page_table")
        return out.reshape(self.cfg.max_batch, ld.value), used.value, pages.value

    def set_eager(self, on: bool):
        self._check(self.lib.lca_debug_set_eager(self.h, 1 if on else 0), "lca_debug_set_eager")

    def profile(self, n, tau, mode, steps):
        p = LcaProfile()
        self._check(self.lib.lca_debug_profile(self.h, n, tau, mode, steps, ctypes.byref(p)),
                    "lca_debug_profile")
        return {k: {"launches": p.launches[i], "ms": p.ms[i], "bytes": p.bytes[i]}
                for i, k in enumerate(PROFILE_KINDS)}

    TRACE_TAGS = {1: "gemv", 2: "gemv_f32", 3: "gemm", 4: "rowstats", 5: "attn", 6: "head",
                  7: "mb_plan", 8: "mb_fill", 9: "mlp_plan", 10: "verify_plan", 11: "segment",
                  12: "lm_scatter", 13: "nb_input", 14: "commit", 15: "loop_ctl", 16: "other",
                  17: "umma", 18: "split", 19: "sgemm", 20: "stack"}

    def trace(self, n, tau, mode, steps, cap=1 << 18):
        rec = np.zeros(cap, dtype=[("t0", "<u8"), ("t1", "<u8"), ("tw", "<u8"), ("tag", "<i4"),
                                   ("cta", "<i4"), ("sm", "<i4"), ("mark", "<i4"), ("mark2", "<i4"),
                                   ("mark3", "<i4")])
        cnt = ctypes.c_int32()
        self._check(self.lib.lca_debug_trace(self.h, n, tau, mode, steps, _ptr(rec), cap, ctypes.byref(cnt)),
                    "lca_debug_trace")
        return rec[:cnt.value]

    def bench_kernel(self, kind, rows, iters):
        us, by = ctypes.c_double(), ctypes.c_double()
        self._check(self.lib.lca_debug_bench_kernel(self.h, kind, rows, iters, ctypes.byref(us),
                                                    ctypes.byref(by)), "lca_debug_bench_kernel")
        return us.value, by.value

    def logits(self, n):
        nb = np.zeros((self.batch, n, 256), dtype=np.float32)
        mb = np.zeros((self.batch, max(n - 1, 0), 256), dtype=np.float32)
        self._check(self.lib.lca_debug_logits(self.h, _ptr(nb), _ptr(mb) if n > 1 else None),
                    "lca_debug_logits")
        return nb, mb

    def force_accept(self, a):
        if a is None:
            self._check(self.lib.lca_debug_force_accept(self.h, None), "force_accept")
            return
        arr = np.ascontiguousarray(a, dtype=np.int32)
        self._check(self.lib.lca_debug_force_accept(self.h, _ptr(arr)), "force_accept")

    def force_candidates(self, cand, n):
        if cand is None:
            self._check(self.lib.lca_debug_force_candidates(self.h, None, 0), "force_candidates")
            return
        arr = np.frombuffer(b"".join(bytes(c) for c in cand), dtype=np.uint8).copy()
        self._check(self.lib.lca_debug_force_candidates(self.h, _ptr(arr), n), "force_candidates")


def decode_attention(q, out, k_cache, v_cache, kv_len, scale, splits, scratch=None, stream=None,
                     noalloc=False):
    """Standalone decode attention on torch CUDA tensors (see include/lca.h).
    q/out: fp32 [batch*n_rows, heads*head_dim]; caches [batch, heads, slots, head_dim];
    kv_len: int32 [batch*n_rows]. Returns the status code."""
    import torch
    lib = load_library()
    batch, heads, slots, hd = k_cache.shape
    n_rows = q.shape[0] // batch
    dt = LCA_BF16 if k_cache.dtype == torch.bfloat16 else LCA_F32
    st = stream if stream is not None else torch.cuda.current_stream(q.device)
    args = [q.data_ptr(), out.data_ptr(), k_cache.data_ptr(), v_cache.data_ptr(), dt, batch, heads, hd,
            slots, n_rows, kv_len.data_ptr(), scale, splits]
    if noalloc:
        return lib.lca_decode_attention_noalloc(*args, st.cuda_stream)
    return lib.lca_decode_attention(*args, scratch.data_ptr(), scratch.numel(), st.cuda_stream)


def decode_attention_status(scratch=None, stream=None, noalloc=False, device=None):
    """Status the kernels of the last decode_attention call recorded (waits for the stream):
    0, LCA_E_DEVICE_STATE (-5) for a kv_len beyond the cache, or LCA_E_TIMEOUT (-7)."""
    import torch
    lib = load_library()
    st = stream if stream is not None else torch.cuda.current_stream(device)
    if noalloc:
        return lib.lca_decode_attention_noalloc_status(st.cuda_stream)
    return lib.lca_decode_attention_status(scratch.data_ptr(), st.cuda_stream)


def debug_gemm(x, W, y, M_dev, err_dev, rows_typ=0, scratch=None, stream=None):
    """y[:M] = x[:M] . W^T on the tensor cores (tcgen05, activations split into two bf16 halves).
    x fp32 [M,K], W bf16 [N,K], y fp32 [M,N], M_dev int32 [1] (rows actually used), err_dev
    int32 [1]; rows_typ: row count the launch shape is chosen for (0 = M); scratch: a uint8
    device tensor of debug_gemm_scratch_bytes(M, K) bytes (allocated here when None).
    Returns the status."""
    import torch
    st = stream if stream is not None else torch.cuda.current_stream(x.device)
    if scratch is None:
        scratch = torch.empty(debug_gemm_scratch_bytes(x.shape[0], W.shape[1]), dtype=torch.uint8,
                              device=x.device)
    return load_library().lca_debug_gemm(x.data_ptr(), W.data_ptr(), y.data_ptr(), x.shape[0], W.shape[0],
                                         W.shape[1], M_dev.data_ptr(), rows_typ, err_dev.data_ptr(),
                                         scratch.data_ptr(),
                                         st.cuda_stream)


def debug_gemm_scratch_bytes(M, K):
    return load_library().lca_debug_gemm_scratch_bytes(M, K)


def decode_attention_scratch_bytes(batch, heads, head_dim, splits):
    n = ctypes.c_size_t()
    st = load_library().lca_decode_attention_scratch_bytes(batch, heads, head_dim, splits, ctypes.byref(n))
    if st != LCA_OK:
        raise LcaError(st, "lca_decode_attention_scratch_bytes")
    return n.value


def status_str(st: int) -> str:
    return load_library().lca_status_str(st).decode()
