"""CPU oracle, part 3: stochastic decoding, in fp64.

TEST INFRASTRUCTURE ONLY (see ``oracle/model.py``).

Section 4 samples one task's outputs with temperature 0.7 and top-p 0.9 and decodes the others
greedily; Section 6.2 names the two acceptance methods, the probability threshold of Algorithm 1
and speculative decoding after Leviathan et al. (2023). This module gives the sampled forms of
both; ``oracle/decode.py`` calls them when a ``Sampling`` is passed.

Random numbers come from Philox-4x32-10 (Salmon, Moraes, Dror and Shaw, "Parallel random numbers:
as easy as 1, 2, 3", SC 2011). The generator is counter-based: a draw is a pure function of its
key and its counter, so the device makes the same draws from the same definition and neither side
carries generator state. Key = the 64-bit seed (low word first). Counter of a draw = (t, b, kind,
j): t the committed length when the step starts, b the sequence index, kind one of DRAFT, ACCEPT,
NEXT, and j = w // 4 the block of word w of that kind's stream (w % 4 picks the output word).
A 32-bit word x becomes the uniform (x >> 8) * 2^-24 in [0, 1), exact in fp32 and fp64.

Readings (also listed with the design notes):
  * A head's sampling distribution is softmax(l / T), restricted to its top-p nucleus: the tokens
    taken in order of falling probability (lower byte first among equals) while the mass before
    them is below top_p, renormalised. T = 0 means greedy (all mass on the lowest argmax).
  * A byte is drawn from a distribution by its inverse CDF in byte order: the lowest j whose
    cumulative mass exceeds u.
  * Threshold acceptance compares the drafter's model probability softmax(l)[d] (T = 1, whole
    vocabulary) of the sampled draft d with tau; T and top-p only shape the draw. As T -> 0 this
    is the greedy threshold rule.
  * Speculative acceptance: draft d_{i+2}, drawn from Q_i (the MB head's sampling distribution of
    draft row i), is kept while u < P_i(d) / Q_i(d), where P_i is the next-byte sampling
    distribution of candidate row i (the row that predicts d's position). At the first rejection
    (row a) the following step's first byte c_1 is drawn from norm(max(0, P_a - Q_a)); when every
    draft is kept, from P_{n-1}. This is the rejection rule of speculative sampling, under which
    the emitted bytes are distributed as plain sampling from P.
  * c_1 of the step that starts at committed length t uses word 0 of kind NEXT at t; draft
    d_{i+2} word i of kind DRAFT, its acceptance word i of kind ACCEPT, both at the step's t.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

# Philox constants (Salmon et al. 2011): round multipliers and Weyl key increments.
PHILOX_M32 = (0xD2511F53, 0xCD9E8D57)
PHILOX_W32 = (0x9E3779B9, 0xBB67AE85)
PHILOX_M64 = (0xD2E7470EE14C6C93, 0xCA5A826395121157)
PHILOX_W64 = (0x9E3779B97F4A7C15, 0xBB67AE8584CAA73B)

# Streams of one step (third counter word).
DRAFT = 0
ACCEPT = 1
NEXT = 2


def philox4(ctr, key, width=32, rounds=10):
    """Philox-4xW-R block: four W-bit counter words and two key words -> four output words.
    Each round multiplies counter words 0 and 2 by the two round constants, takes the high halves
    XOR the other two counter words and the key, and the low halves as the new words 1 and 3;
    the key advances by the Weyl constants between rounds."""
    mask = (1 << width) - 1
    (m0, m1), (w0, w1) = (PHILOX_M32, PHILOX_W32) if width == 32 else (PHILOX_M64, PHILOX_W64)
    c0, c1, c2, c3 = (int(v) & mask for v in ctr)
    k0, k1 = (int(v) & mask for v in key)
    for r in range(rounds):
        if r:
            k0 = (k0 + w0) & mask
            k1 = (k1 + w1) & mask
        p0 = m0 * c0
        p1 = m1 * c2
        c0, c1, c2, c3 = (p1 >> width) ^ c1 ^ k0, p1 & mask, (p0 >> width) ^ c3 ^ k1, p0 & mask
    return c0, c1, c2, c3


def uniform24(word):
    """A 32-bit word as a uniform in [0, 1): its top 24 bits times 2^-24."""
    return float((int(word) & 0xFFFFFFFF) >> 8) * 2.0 ** -24


def draw(seed, t, b, kind, w):
    """Uniform w of stream `kind` of sequence b in the step that starts at committed length t."""
    key = (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    return uniform24(philox4((t, b, kind, w // 4), key)[w % 4])


@dataclass(frozen=True)
class Sampling:
    """Sampling settings of one decode. temperature 0: greedy (the draws are unused)."""
    temperature: float
    top_p: float = 1.0
    seed: int = 0


def sampling_dist(logits, temperature, top_p=1.0):
    """The distribution a byte is drawn from: softmax(l / T) restricted to its top-p nucleus."""
    l = np.asarray(logits, dtype=np.float64)
    V = l.shape[0]
    if temperature <= 0:
        p = np.zeros(V)
        p[int(np.argmax(l))] = 1.0
        return p
    z = l / temperature
    z = z - z.max()
    p = np.exp(z)
    p /= p.sum()
    if top_p < 1.0:
        order = sorted(range(V), key=lambda i: (-p[i], i))
        keep = np.zeros(V, dtype=bool)
        mass = 0.0
        for i in order:
            if mass >= top_p:
                break
            keep[i] = True
            mass += p[i]
        p = np.where(keep, p, 0.0)
        p /= p.sum()
    return p


def sample_index(p, u):
    """Inverse CDF in byte order: the lowest j with p_0 + ... + p_j > u (the last byte of
    nonzero mass if rounding leaves u above the total)."""
    c = 0.0
    last = -1
    for j in range(len(p)):
        if p[j] <= 0.0:
            continue
        c += p[j]
        last = j
        if u < c:
            return j
    return last


def residual_dist(p, q):
    """Distribution of the replacement byte after a rejected draft: norm(max(0, p - q)).
    p == q leaves no mass; then p itself."""
    r = np.maximum(np.asarray(p, dtype=np.float64) - np.asarray(q, dtype=np.float64), 0.0)
    s = r.sum()
    return np.asarray(p, dtype=np.float64) if s <= 0.0 else r / s


def spec_keep(p, q, d, u):
    """Speculative acceptance of draft d drawn from q: keep iff u < p(d) / q(d), i.e. with
    probability min(1, p(d) / q(d))."""
    return bool(u * q[d] < p[d])
