"""Mutant oracles for the separation checks of the bf16 attention tests.

A parity test at the bf16 tolerance (max-abs 2e-2) only means something if a
wrong kernel would fail it. Each mutant here is the oracle's cache, built by
`oracle.dmc_ref.update` (Algorithm 1) token by token, with one plausible kernel
mistake in the attention step (Eq. attn-softmax):

  uniform   the query ignored: softmax over all-zero scores, i.e. the plain
            mean of the head's slot values;
  noscale   scores without the 1/sqrt(d_h) factor;
  droppage  one 32-slot page of the head left out of the softmax (the page
            that carries the most softmax mass for the last token's first
            query, so that leaving it out matters).

`exact` is the same code with no mistake; the CPU tests pin it to the oracle's
own `run_head` / `prompt_attention`, so the mutants differ from the oracle by
their mistake only. The GPU tests require the CUDA result within the
tolerance of the oracle and farther than the tolerance from every mutant.
"""
from __future__ import annotations

import copy

import numpy as np

from oracle import dmc_ref as R

MODES = ("uniform", "noscale", "droppage")
PAGE = 32


class _Tracked:
    """An oracle HeadCache plus dense copies of its slots, updated in place
    (Algorithm 1 changes only the last slot or appends one)."""

    def __init__(self, d, cap, window=0):
        self.c = R.HeadCache(d)
        self.K = np.zeros((cap, d))
        self.V = np.zeros((cap, d))
        self.window = window

    def update(self, k, v, q0_group):
        R.update(self.c, k, v, int(R.decision(k[0])), float(R.importance(q0_group)), self.window)
        n = len(self.c)
        self.K[n - 1] = self.c.K[-1]
        self.V[n - 1] = self.c.V[-1]
        return n


def _attend(K, V, Q, mode, drop=None):
    """Outputs [G, d] of queries Q [G, d] over slots K, V [n, d] under `mode`."""
    d = K.shape[1]
    q = np.array(Q, dtype=np.float64)
    q[:, 0] = 0.0
    if drop is not None and drop * PAGE < K.shape[0]:
        keep = np.ones(K.shape[0], dtype=bool)
        keep[drop * PAGE:(drop + 1) * PAGE] = False
        if keep.any():
            K, V = K[keep], V[keep]
    S = K @ q.T                                     # [n, G]
    if mode == "uniform":
        S = np.zeros_like(S)
    elif mode != "noscale":
        S = S / np.sqrt(np.float64(d))
    S = S - S.max(axis=0, keepdims=True)
    P = np.exp(S)
    P = P / P.sum(axis=0, keepdims=True)
    return P.T @ V


def _heaviest_page(K, V, q):
    """The page with the most softmax mass for query q over slots K."""
    qq = np.array(q, dtype=np.float64)
    qq[0] = 0.0
    s = K @ qq / np.sqrt(np.float64(K.shape[1]))
    p = np.exp(s - s.max())
    mass = np.add.reduceat(p, np.arange(0, len(p), PAGE))
    return int(np.argmax(mass))


def decode_outputs(k_prompt, v_prompt, q0_prompt, k_dec, v_dec, q_dec, modes=MODES + ("exact",),
                   window=0):
    """Decode outputs [S, G, d] of one KV head under each mode: the prompt is
    compressed, then every decode token is compressed and its G queries
    attend (the oracle's run_head with the attention step mutated; window > 0:
    the window-grouping approximation)."""
    k_prompt, v_prompt = np.asarray(k_prompt, np.float64), np.asarray(v_prompt, np.float64)
    q0_prompt = np.asarray(q0_prompt, np.float64)
    k_dec, v_dec = np.asarray(k_dec, np.float64), np.asarray(v_dec, np.float64)
    q_dec = np.asarray(q_dec, np.float64)
    T, S = k_prompt.shape[0], k_dec.shape[0]
    d = k_dec.shape[1]
    G = q_dec.shape[1]
    tr = _Tracked(d, T + S + 1, window)
    for t in range(T):
        tr.update(k_prompt[t], v_prompt[t], q0_prompt[t])
    after_prompt = copy.deepcopy(tr)
    # the page to drop: from a first pass over the decode tokens
    for s in range(S):
        n = tr.update(k_dec[s], v_dec[s], q_dec[s, :, 0])
    drop = _heaviest_page(tr.K[:n], tr.V[:n], q_dec[S - 1, 0]) if S else 0
    out = {m: np.zeros((S, G, d)) for m in modes}
    tr = after_prompt
    for s in range(S):
        n = tr.update(k_dec[s], v_dec[s], q_dec[s, :, 0])
        for m in modes:
            out[m][s] = _attend(tr.K[:n], tr.V[:n], q_dec[s], "exact" if m == "droppage" else m,
                                drop if m == "droppage" else None)
    out["drop_page"] = drop
    return out


def prompt_outputs(k, v, q, modes=MODES + ("exact",)):
    """Prompt-attention outputs [T, G, d] of one KV head under each mode:
    every prompt token is compressed and its queries attend over the cache
    as it stands after that update (the oracle's prompt_attention with the
    attention step mutated)."""
    return decode_outputs(np.zeros((0, np.shape(k)[1])), np.zeros((0, np.shape(k)[1])),
                          np.zeros((0, np.shape(q)[1])), k, v, q, modes)


def separation(got, muts, modes=MODES):
    """max |got - mutant| per mode."""
    return {m: float(np.max(np.abs(np.asarray(got, np.float64) - muts[m]))) for m in modes}


def decode_separation(run, tol):
    """For a harness Run: per sampled head, the GPU decode outputs against each
    mutant. Returns (worst, failures): worst = smallest distance per mode over
    the heads where the mode applies (a head of one page has no page to drop),
    failures = the heads where a mutant lies within `tol`."""
    worst = {m: np.inf for m in MODES}
    bad = []
    for s in run.samples:
        I = run.inst[s]
        if not I["out"]:
            continue
        got = np.array(I["out"])
        muts = decode_outputs(I["k_prompt"], I["v_prompt"], I["q0_prompt"], np.array(I["k_dec"]),
                              np.array(I["v_dec"]), np.array(I["q_dec"]), window=run.window)
        n_slots = run.final_export[s][3]
        sep = separation(got, muts)
        for m in MODES:
            if m == "droppage" and n_slots <= PAGE:
                continue
            worst[m] = min(worst[m], sep[m])
            if not sep[m] > tol:
                bad.append(f"{s}: within {sep[m]:.4f} of the '{m}' mutant")
    return worst, bad
