"""CPU oracle, part 2: the multi-byte-prediction decode loop (Algorithm 1), in fp64.

TEST INFRASTRUCTURE ONLY (see ``oracle/model.py``).

Two interchangeable implementations of one step:
  * ``generate_reference``: Algorithm 1 taken literally. Every step recomputes the
    whole forward over the committed bytes (its forward part), drafts with the MB head over
    the window (its drafting part) and accepts by threshold (Section 3.1, byte
    acceptance): the next-byte output is always kept, drafts are kept left to right
    while their probability is >= tau, and the first failure drops the rest.
  * ``IncrementalDecoder``: the same results with KV caches. Each step drafts, runs
    one forward over all n candidates (encoder, LM module on the segments the
    candidates close, next-byte decoder), then keeps the accepted prefix of the
    caches and drops the rest. Its equality with the reference is a test.

Speculative-decoding acceptance (Section 6.2, acceptance method (ii)) is the greedy variant: draft
d_i is kept while it equals the next-byte argmax at the position before it, so the
output equals plain next-byte decoding. Meaning of n (a reading): one next-byte
byte plus n-1 drafts per step, so 1..n bytes are emitted per step.

With a ``Sampling`` (``oracle/sampling.py``) both decoders draw c_1 and the drafts instead of
taking argmaxes, and speculative acceptance becomes the rejection rule of speculative sampling;
the first byte of the step after a rejection is drawn from the residual distribution.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from types import SimpleNamespace

import numpy as np

from .model import (Model, boundary_flags, causal_mask, forward_full, greedy, latent_index,
                    max_prob, mb_draft_logits, segments_of)
from .sampling import (ACCEPT, DRAFT, NEXT, Sampling, draw, residual_dist, sample_index,
                       sampling_dist, spec_keep)

THRESH = 0
SPEC = 1


@dataclass
class StepRecord:
    c1: int
    drafts: list
    probs: list
    a: int                       # accepted drafts (0..n-1) before the budget cut
    emitted: bytes               # committed bytes (1 + a, cut to the remaining budget)
    mb_logits: np.ndarray        # [n-1, V]
    nb_logits: np.ndarray | None  # [n, V] next-byte logits of the n candidate rows
    t: int = 0                   # committed length after the step
    K: int = 0                   # committed latent count after the step


def accept_count(mode, drafts, probs, nb_logits, tau, forced=None):
    """Accepted drafts a in [0, n-1], always a prefix (Section 3.1). ``drafts`` are the
    proposed bytes d_2..d_n, ``probs`` the drafter's probabilities of them."""
    if forced is not None:
        return int(forced)
    a = 0
    for i, d in enumerate(drafts):
        if mode == THRESH:
            ok = probs[i] >= tau
        elif mode == SPEC:
            ok = d == greedy(nb_logits[i])
        else:
            raise ValueError(mode)
        if not ok:
            break
        a += 1
    return a


def sampled_drafts(mbl, samp: Sampling, t, b):
    """Drafts d_2..d_n drawn from the MB head's sampling distributions (stream DRAFT at t), with
    the drafter's model probabilities softmax(l)[d] that threshold acceptance compares with tau."""
    drafts, probs = [], []
    for i, r in enumerate(mbl):
        q = sampling_dist(r, samp.temperature, samp.top_p)
        d = sample_index(q, draw(samp.seed, t, b, DRAFT, i))
        drafts.append(d)
        probs.append(max_prob(r, d))
    return drafts, probs


def sampled_accept(mode, drafts, probs, mbl, nbl, tau, samp: Sampling, t, b, forced=None):
    """(a, rejected): accepted drafts, a prefix, and whether the step ended on a draft that
    speculative acceptance rejected (threshold acceptance drops the rest without a correction)."""
    if forced is not None:
        return int(forced), False
    a = 0
    for i, d in enumerate(drafts):
        if mode == THRESH:
            ok = probs[i] >= tau
        elif mode == SPEC:
            P = sampling_dist(nbl[i], samp.temperature, samp.top_p)
            Q = sampling_dist(mbl[i], samp.temperature, samp.top_p)
            ok = spec_keep(P, Q, d, draw(samp.seed, t, b, ACCEPT, i))
        else:
            raise ValueError(mode)
        if not ok:
            return a, mode == SPEC
        a += 1
    return a, False


def carried_dist(rejected, a, e, mbl, nbl, samp: Sampling):
    """Distribution of the next step's c_1 when it is not the plain next-byte distribution of the
    last committed row: the residual norm(max(0, P_a - Q_a)) after a rejection at row a that the
    budget did not cut. None otherwise."""
    if not rejected or e - 1 != a:
        return None
    return residual_dist(sampling_dist(nbl[a], samp.temperature, samp.top_p),
                         sampling_dist(mbl[a], samp.temperature, samp.top_p))


def _force(force, step):
    if force is None:
        return None
    return force(step) if callable(force) else force[step % len(force)]


def generate_reference(model: Model, prompt, n, tau, mode, G, force=None, record_nb=False,
                       force_cand=None, samp: Sampling | None = None, b=0):
    """Algorithm 1 with a full recompute per step. Returns (generated bytes, [StepRecord]).
    force: accepted-draft counts per step (test hook); force_cand(step) -> n candidate bytes
    that replace c_1, d_2..d_n (test hook for driving boundaries through a step).
    samp: sample instead of taking argmaxes, with the draws of sequence index b."""
    x = bytearray(prompt)
    out = bytearray()
    recs = []
    step = 0
    carried = None
    while len(out) < G:
        F = forward_full(model, x)
        t = len(x)
        mbl = mb_draft_logits(model, F.Kp, F.o, F.u, t, n, x, y_last=F.y[t - 1])
        if samp is None:
            c1 = greedy(F.nb_logits[t - 1])
            drafts = [greedy(r) for r in mbl]
            probs = [max_prob(r, d) for r, d in zip(mbl, drafts)]
        else:
            p1 = carried if carried is not None else sampling_dist(
                F.nb_logits[t - 1], samp.temperature, samp.top_p)
            c1 = sample_index(p1, draw(samp.seed, t, b, NEXT, 0))
            drafts, probs = sampled_drafts(mbl, samp, t, b)
        cand = bytes([c1] + drafts)
        fc = force_cand(step) if force_cand is not None else None
        if fc is not None:
            cand = bytes(fc)
        nbl = None
        if mode == SPEC or record_nb:
            nbl = forward_full(model, bytes(x) + cand).nb_logits[t:t + n]
        if samp is None:
            a = accept_count(mode, list(cand[1:]), probs, nbl, tau, _force(force, step))
        else:
            a, rejected = sampled_accept(mode, list(cand[1:]), probs, mbl, nbl, tau, samp, t, b,
                                         _force(force, step))
        e = min(1 + a, G - len(out))
        if samp is not None:
            carried = carried_dist(rejected, a, e, mbl, nbl, samp)
        em = cand[:e]
        x += em
        out += em
        rec = StepRecord(c1, drafts, probs, a, em, mbl, nbl, t=len(x), K=_latents(model, x))
        recs.append(rec)
        step += 1
    return bytes(out), recs


def _latents(model: Model, x):
    """K(t-1) of bytes x: the closed segments (a forward for the learned predictor)."""
    if model.cfg.boundary == "learned":
        return int(forward_full(model, x).Kp[-1])
    return int(latent_index(model.cfg, x)[-1])


def greedy_decode(model: Model, prompt, G):
    """Plain next-byte greedy decoding, one byte per full forward."""
    x = bytearray(prompt)
    for _ in range(G):
        x.append(greedy(forward_full(model, x).nb_logits[-1]))
    return bytes(x[len(prompt):])


class IncrementalDecoder:
    """Cached decode of one sequence: prefill, then steps of draft / verify / accept /
    commit. All cache entries beyond the committed lengths are dropped at commit."""

    def __init__(self, model: Model):
        self.m = model
        self.cfg = model.cfg

    # -------------------------------------------------------------- prefill
    def prefill(self, prompt):
        F = forward_full(self.m, prompt, keep_caches=True)
        self.x = bytearray(prompt)
        self.b = [bool(f) for f in F.b]  # boundary flags of the committed bytes
        self.h_e = F.h_e
        self.Kp = list(int(k) for k in F.Kp)
        self.u = F.u
        self.o = F.o
        self.kv = {s: [[k, v] for k, v in F.caches[s]] for s in ("enc", "lm", "nb")}
        self.nb_last = F.nb_logits[-1]
        self.y_last = F.y[-1]
        self.carried = None  # c_1 distribution carried from a rejection (sampled decoding)
        return F

    @property
    def t(self):
        return len(self.x)

    @property
    def K(self):
        return self.Kp[-1] if self.Kp else 0

    def open_start(self):
        segs = segments_of(self.b)
        return segs[-1][1] + 1 if segs else 0

    def group_starts(self):
        """(start of group K(t-1)-1 or -1, start of group K(t-1))."""
        segs = segments_of(self.b)
        g = self.K

        def st(j):
            return 0 if j == 0 else segs[j - 1][1]
        return (st(g - 1) if g >= 1 else -1), st(g)

    # -------------------------------------------------------------- one step
    def _stack_cached(self, prefix, x, pos):
        caches = [(k, v) for k, v in self.kv[prefix]]
        T = x.shape[0]
        return self.m.run_stack(prefix, x, pos, lambda n_prev: causal_mask(n_prev, T), caches)

    def run_candidates(self, cand):
        """The forward part of a step over candidate bytes at positions t..t+len(cand)-1: encoder
        rows after the cached keys, the boundaries and the segments they close (mean pools over
        committed and candidate states), the LM module on those latents, the next-byte decoder
        over o_{K(p)} + h_e[p]. Nothing is kept until ``commit``; ``nbl`` of the result holds the
        next-byte logits of the candidate rows."""
        m, t, K, n = self.m, self.t, self.K, len(cand)
        pos = np.arange(t, t + n)
        # encoder over the candidates, appended after the cached keys
        h_c, enc_new = self._stack_cached("enc", m.embed(cand), pos)
        # segments closed by candidate boundaries (by the byte, or predicted from h_e of the
        # candidate); z over committed + candidate bytes
        cb = boundary_flags(m, cand, h_c)
        h_all = np.concatenate([self.h_e, h_c], axis=0)
        Kc, z_new, k_run = [], [], K
        seg_start = self.open_start()
        for i in range(n):
            if cb[i]:
                k_run += 1
                z_new.append(h_all[seg_start:t + i + 1].mean(axis=0))
                seg_start = t + i + 1
            Kc.append(k_run)
        u_ext, o_ext = self.u, self.o
        lm_new = None
        if z_new:
            z_new = np.stack(z_new)
            o_new, lm_new = self._stack_cached("lm", z_new, np.arange(K + 1, K + 1 + len(z_new)))
            u_ext = np.concatenate([self.u, z_new], axis=0)
            o_ext = np.concatenate([self.o, o_new], axis=0)
        # next-byte decoder over o_{K(p)} + h_e[p]
        y_c, nb_new = self._stack_cached("nb", o_ext[Kc] + h_c, pos)
        return SimpleNamespace(cand=bytes(cand), cb=cb, h_all=h_all, Kc=Kc, u=u_ext, o=o_ext,
                               enc=enc_new, lm=lm_new, nb=nb_new, y=y_c, nbl=m.head(y_c, "nb.norm"))

    def commit(self, P, e):
        """Keep the first e candidate rows of ``run_candidates``' result in every cache (and the
        latents their segments closed); drop the rest."""
        t, K = self.t, self.K
        self.x += P.cand[:e]
        self.b += [bool(f) for f in P.cb[:e]]
        self.h_e = P.h_all[:t + e]
        self.Kp += P.Kc[:e]
        K_new = self.Kp[-1]
        for s, new in (("enc", P.enc), ("nb", P.nb)):
            for l, (k, v) in enumerate(new):
                self.kv[s][l][0] = np.concatenate([self.kv[s][l][0], k[:e]], axis=0)
                self.kv[s][l][1] = np.concatenate([self.kv[s][l][1], v[:e]], axis=0)
        keep = K_new - K
        if keep > 0:
            for l, (k, v) in enumerate(P.lm):
                self.kv["lm"][l][0] = np.concatenate([self.kv["lm"][l][0], k[:keep]], axis=0)
                self.kv["lm"][l][1] = np.concatenate([self.kv["lm"][l][1], v[:keep]], axis=0)
        self.u = P.u[:K_new + 1]
        self.o = P.o[:K_new + 1]
        self.nb_last = P.nbl[e - 1]
        self.y_last = P.y[e - 1]

    def step(self, n, tau, mode, forced=None, budget=None, forced_cand=None,
             samp: Sampling | None = None, b=0):
        """One decode step. forced: accepted-draft count (test hook); forced_cand: n bytes
        replacing c_1, d_2..d_n (test hook); budget: cap on the committed bytes; samp: sample
        with the draws of sequence index b instead of taking argmaxes."""
        m, t = self.m, self.t
        # draft (Algorithm 1, drafting step)
        mbl = mb_draft_logits(m, self.Kp, self.o, self.u, t, n, self.x, y_last=self.y_last)
        if samp is None:
            c1 = greedy(self.nb_last)
            drafts = [greedy(r) for r in mbl]
            probs = [max_prob(r, d) for r, d in zip(mbl, drafts)]
        else:
            p1 = self.carried if self.carried is not None else sampling_dist(
                self.nb_last, samp.temperature, samp.top_p)
            c1 = sample_index(p1, draw(samp.seed, t, b, NEXT, 0))
            drafts, probs = sampled_drafts(mbl, samp, t, b)
        cand = bytes([c1] + drafts) if forced_cand is None else bytes(forced_cand)
        P = self.run_candidates(cand)
        nbl = P.nbl
        # accept (Algorithm 1, acceptance step) and commit the accepted prefix
        if samp is None:
            a = accept_count(mode, list(cand[1:]), probs, nbl, tau, forced)
        else:
            a, rejected = sampled_accept(mode, list(cand[1:]), probs, mbl, nbl, tau, samp, t, b,
                                         forced)
        e = 1 + a if budget is None else min(1 + a, budget)
        self.carried = None if samp is None else carried_dist(rejected, a, e, mbl, nbl, samp)
        self.commit(P, e)
        return StepRecord(c1, drafts, probs, a, cand[:e], mbl, nbl, t=self.t, K=self.K)


def generate_incremental(model: Model, prompt, n, tau, mode, G, force=None, force_cand=None,
                         samp: Sampling | None = None, b=0):
    """Cached decode loop with the same stopping rule as ``generate_reference``."""
    dec = IncrementalDecoder(model)
    dec.prefill(prompt)
    out = bytearray()
    recs = []
    step = 0
    while len(out) < G:
        fc = force_cand(step) if force_cand is not None else None
        r = dec.step(n, tau, mode, _force(force, step), budget=G - len(out), forced_cand=fc,
                     samp=samp, b=b)
        out += r.emitted
        recs.append(r)
        step += 1
    return bytes(out), recs
