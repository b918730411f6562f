"""Dynamic Memory Compression in plain numpy fp64: the oracle.

TEST INFRASTRUCTURE ONLY (see the package docstring). Nothing here is tuned:
every function is the paper's definition written out, one token at a time where
the paper's definition is sequential.

Notation follows the paper (arXiv 2403.09636):
  k_t, v_t, q_t  key, value, query of token t for one head (head dim d_h)
  alpha_t        append-or-accumulate decision,  omega_t importance
  K, V, z        the compressed cache of one KV head: slots K_j, V_j and the
                 running importance sum z_j of the tokens merged into slot j.

Readings the paper leaves open, fixed here and mirrored by the CUDA path:
  * alpha_t = round(sigmoid(k_t[0])) rounds a tie (k_t[0] = 0, sigmoid = 0.5)
    up to 1; NaN gives 0 (append).
  * The first token of an empty cache always opens slot 0 (the initial
    conditions z_0 = omega_0, k_0 = k_0 of Eq. partial-accumulation).
  * Grouped-query attention: one decision per KV head from its key; the
    importance is the sigmoid of the MEAN of the group's q[0]; every query of
    the group has its q[0] removed and attends over the shared slots.
  * The scale stays 1/sqrt(d_h) with d_h the full head dim (masking appendix).
  * A token attends over the cache AFTER its own update (Eq. attn-softmax sums
    up to t = i inclusive; the training mask has 0 on its diagonal).
"""
from __future__ import annotations

import numpy as np

f64 = np.float64


# --------------------------------------------------------------------------
# Eq. (reuse), Section 3.1: both gates are read from existing neurons.
# --------------------------------------------------------------------------

def sigmoid(x):
    """Logistic function, fp64."""
    x = np.asarray(x, dtype=f64)
    with np.errstate(over="ignore"):
        return 1.0 / (1.0 + np.exp(-x))


def decision(k0):
    """alpha_t = round(sigmoid(k_t[0])) -- Eq. (reuse), first step of Algorithm 1.

    Rounded to the closest integer; sigmoid = 0.5 exactly rounds up (reading).
    NaN compares false and yields 0 (append)."""
    return (sigmoid(k0) >= 0.5).astype(np.int64)


def omega_logit(q0_group):
    """The pre-sigmoid importance of one token from its queries' first neuron.

    MHA passes one value; GQA passes the G values of the group, and the
    reading here is their mean (the paper does not say how a group shares
    omega). Shape [..., G] -> [...]."""
    return np.mean(np.asarray(q0_group, dtype=f64), axis=-1)


def importance(q0_group):
    """omega_t = sigmoid(q_t[0]) -- Eq. (reuse), second step of Algorithm 1."""
    return sigmoid(omega_logit(q0_group))


# --------------------------------------------------------------------------
# Formulation A: Algorithm 1, one token at a time, then attention (Sec. 3.1).
# --------------------------------------------------------------------------

class HeadCache:
    """The variable-length compressed cache of one (layer, sequence, KV head)."""

    def __init__(self, d: int):
        self.d = d
        self.K: list[np.ndarray] = []
        self.V: list[np.ndarray] = []
        self.z: list[float] = []
        # tokens (k with k[0] cleared, v, omega) of the open segment, for the
        # window-grouping approximation
        self.seg: list[tuple] = []

    def __len__(self) -> int:
        return len(self.K)

    def arrays(self):
        d = self.d
        K = np.array(self.K, dtype=f64).reshape(-1, d)
        V = np.array(self.V, dtype=f64).reshape(-1, d)
        return K, V, np.array(self.z, dtype=f64)


def update(cache: HeadCache, k_t, v_t, alpha_t: int, omega_t: float, window: int = 0) -> None:
    """Algorithm 1: single-head KV cache update with DMC.

    k_t[0] is cleared first (Algorithm 1, third step). With alpha_t = 1 the
    token is merged into the last slot as the omega-weighted running mean,
    z_t = z_{t-1} + omega_t; with alpha_t = 0 it opens a new slot, z_t = omega_t.
    An empty cache always receives a new slot.

    window = w > 0: the window-grouping approximation (Sec. 3.3), where
    Eq. partial-accumulation runs over the last w tokens only: the last slot
    is the omega-weighted mean of the last min(segment length, w) tokens of
    its segment and z their summed omega."""
    k = np.array(k_t, dtype=f64)
    k[0] = 0.0
    v = np.array(v_t, dtype=f64)
    if window > 0:
        if alpha_t == 1 and len(cache) > 0:
            cache.seg = (cache.seg + [(k, v, float(omega_t))])[-window:]
            w = np.array([t[2] for t in cache.seg])
            cache.K[-1] = (w[:, None] * np.array([t[0] for t in cache.seg])).sum(0) / w.sum()
            cache.V[-1] = (w[:, None] * np.array([t[1] for t in cache.seg])).sum(0) / w.sum()
            cache.z[-1] = float(w.sum())
        else:
            cache.seg = [(k, v, float(omega_t))]
            cache.K.append(k)
            cache.V.append(v)
            cache.z.append(float(omega_t))
        return
    if alpha_t == 1 and len(cache) > 0:
        z_prev = cache.z[-1]
        z_t = z_prev + omega_t
        cache.K[-1] = (cache.K[-1] * z_prev + k * omega_t) / z_t
        cache.V[-1] = (cache.V[-1] * z_prev + v * omega_t) / z_t
        cache.z[-1] = z_t
    else:
        cache.K.append(k)
        cache.V.append(v)
        cache.z.append(float(omega_t))


def attend(cache: HeadCache, q_t) -> np.ndarray:
    """Eq. (attn-softmax) for one query over the compressed cache.

    q_t[0] is removed (Algorithm 1, third step) and the score is
    q[1:]^T K_j[1:] / sqrt(d_h) (masking appendix). Softmax in fp64 with the
    maximum subtracted."""
    q = np.array(q_t, dtype=f64)
    q[0] = 0.0
    K, V, _ = cache.arrays()
    s = (K @ q) / np.sqrt(f64(cache.d))
    s = s - np.max(s)
    p = np.exp(s)
    p = p / np.sum(p)
    return p @ V


def run_head(k_prompt, v_prompt, q0_prompt, k_dec, v_dec, q_dec, cache=None, window: int = 0):
    """One KV head through a prompt and then decode tokens (formulation A).

    k_prompt, v_prompt [T, d]; q0_prompt [T, G] (first neuron of each query of
    the group); k_dec, v_dec [S, d]; q_dec [S, G, d]. Prompt tokens are only
    compressed into the cache; every decode token is compressed and then each
    of its G queries attends over the updated cache.

    Returns dict with the cache after the prompt (K, V, z copies), the decode
    outputs [S, G, d], the lengths after each decode token, and the cache."""
    k_prompt = np.asarray(k_prompt, dtype=f64)
    v_prompt = np.asarray(v_prompt, dtype=f64)
    q0_prompt = np.asarray(q0_prompt, dtype=f64)
    k_dec = np.asarray(k_dec, dtype=f64)
    v_dec = np.asarray(v_dec, dtype=f64)
    q_dec = np.asarray(q_dec, dtype=f64)
    d = k_prompt.shape[1] if k_prompt.size else k_dec.shape[1]
    if cache is None:
        cache = HeadCache(d)
    for t in range(k_prompt.shape[0]):
        update(cache, k_prompt[t], v_prompt[t],
               int(decision(k_prompt[t, 0])), float(importance(q0_prompt[t])), window)
    Kp, Vp, zp = cache.arrays()
    S = k_dec.shape[0]
    G = q_dec.shape[1] if S else 0
    out = np.zeros((S, G, d), dtype=f64)
    lens = np.zeros(S, dtype=np.int64)
    for s in range(S):
        update(cache, k_dec[s], v_dec[s],
               int(decision(k_dec[s, 0])), float(importance(q_dec[s, :, 0])), window)
        for g in range(G):
            out[s, g] = attend(cache, q_dec[s, g])
        lens[s] = len(cache)
    return {"prompt_K": Kp, "prompt_V": Vp, "prompt_z": zp,
            "prompt_len": Kp.shape[0], "out": out, "lens": lens,
            "cache": cache}


def prompt_attention(k, v, q, cache=None, window: int = 0):
    """Attention outputs of every prompt token at inference (formulation A).

    Sec. 3.2 (intermediate compression steps): at inference the last slot
    changes in place, so each prompt token sees the cache as it stands after
    its own update: the closed slots and its segment's running state. That is
    the decode step applied to the prompt tokens one by one (Algorithm 1, then
    Eq. attn-softmax), which is what this returns; `masked_attention` is the
    training-time statement of the same thing. k, v [T, d]; q [T, G, d]; an
    existing `cache` is continued. Returns [T, G, d]."""
    d = np.asarray(k).shape[1]
    G = np.asarray(q).shape[1]
    empty = np.zeros((0, d))
    return run_head(empty, empty, np.zeros((0, G)), k, v, q, cache=cache, window=window)["out"]


def decode_lengths(k0_tokens, start_len: int = 0) -> np.ndarray:
    """Cache length after each token, from the decisions alone (Sec. 3.1:
    l = sum_t (1 - alpha_t), with an empty cache's first token always opening
    a slot). k0_tokens [n] -> int64 [n]."""
    lens = np.zeros(len(k0_tokens), dtype=np.int64)
    cur = start_len
    for t, x in enumerate(np.asarray(k0_tokens, dtype=f64)):
        if cur == 0 or decision(x) == 0:
            cur += 1
        lens[t] = cur
    return lens


# --------------------------------------------------------------------------
# Formulation C: closed form of a compressed prompt (Eq. partial-accumulation
# with binary alpha): slot j is the omega-weighted mean of segment j.
# --------------------------------------------------------------------------

def segment_ids(k0_tokens) -> np.ndarray:
    """Segment index of every token of a prompt compressed into an empty cache.

    A token with alpha = 0 opens a new segment; the first token opens segment 0
    (Eq. partial-accumulation: z_0 = omega_0, k_0 = k_0)."""
    alpha = decision(np.asarray(k0_tokens, dtype=f64))
    opens = 1 - alpha
    opens[0] = 1
    return np.cumsum(opens) - 1


def segment_slots(k_prompt, v_prompt, q0_prompt, window: int = 0):
    """Slots of a prompt compressed into an empty cache, as segment means.

    K_j = sum_{t in seg j} omega_t k'_t / z_j, V_j likewise, z_j = sum omega_t,
    where k'_t is k_t with its first component cleared. With window = w > 0
    (window grouping) only the last min(|seg j|, w) tokens of each segment
    count. Returns K, V, z."""
    k = np.array(k_prompt, dtype=f64)
    v = np.array(v_prompt, dtype=f64)
    k[:, 0] = 0.0
    seg = segment_ids(np.asarray(k_prompt, dtype=f64)[:, 0])
    w = importance(q0_prompt)
    if window > 0:
        # position of each token counted from its segment's end
        from_end = np.zeros(len(seg), dtype=np.int64)
        for t in range(len(seg) - 2, -1, -1):
            from_end[t] = from_end[t + 1] + 1 if seg[t + 1] == seg[t] else 0
        w = np.where(from_end < window, w, 0.0)
    n = int(seg[-1]) + 1
    z = np.zeros(n, dtype=f64)
    Ks = np.zeros((n, k.shape[1]), dtype=f64)
    Vs = np.zeros((n, v.shape[1]), dtype=f64)
    np.add.at(z, seg, w)
    np.add.at(Ks, seg, w[:, None] * k)
    np.add.at(Vs, seg, w[:, None] * v)
    return Ks / z[:, None], Vs / z[:, None], z


# --------------------------------------------------------------------------
# Formulation B: the training-time view (Sec. 3.2). Every intermediate state of
# Eq. partial-accumulation is kept, and the additive mask of the masking figure
# (0 on the diagonal, log(1 - alpha_{j+1}) below it, -inf above) decides which
# states a query sees. With binary alpha this reproduces inference exactly.
# --------------------------------------------------------------------------

def unrolled_states(k, v, q0_group):
    """Eq. partial-accumulation for every token i of one sequence.

    z_0 = omega_0, k~_0 = k_0;  z_i = z_{i-1} alpha_i + omega_i,
    k~_i = (alpha_i k~_{i-1} z_{i-1} + k_i omega_i) / z_i  (v~ likewise).
    k_i has its first component cleared. Returns k~ [n, d], v~ [n, d], z [n],
    alpha [n] (float)."""
    k = np.array(k, dtype=f64)
    v = np.array(v, dtype=f64)
    alpha = decision(k[:, 0]).astype(f64)
    k[:, 0] = 0.0
    w = importance(q0_group)
    n, d = k.shape
    kt = np.zeros((n, d), dtype=f64)
    vt = np.zeros((n, d), dtype=f64)
    z = np.zeros(n, dtype=f64)
    z[0], kt[0], vt[0] = w[0], k[0], v[0]
    for i in range(1, n):
        z[i] = z[i - 1] * alpha[i] + w[i]
        kt[i] = (alpha[i] * kt[i - 1] * z[i - 1] + k[i] * w[i]) / z[i]
        vt[i] = (alpha[i] * vt[i - 1] * z[i - 1] + v[i] * w[i]) / z[i]
    return kt, vt, z, alpha


def unrolled_states_window(k, v, q0_group, window: int):
    """The window-grouping approximation of Eq. partial-accumulation (Sec. 3.3):
    the state of token i is the recurrence run independently over the window
    of the last w tokens up to i, started afresh at the window's first token
    (z = omega, k~ = k there). Same returns as unrolled_states."""
    k = np.array(k, dtype=f64)
    v = np.array(v, dtype=f64)
    alpha = decision(k[:, 0]).astype(f64)
    k[:, 0] = 0.0
    w = importance(q0_group)
    n, d = k.shape
    kt = np.zeros((n, d), dtype=f64)
    vt = np.zeros((n, d), dtype=f64)
    z = np.zeros(n, dtype=f64)
    for i in range(n):
        s0 = max(0, i - window + 1)
        zi, ki, vi = w[s0], k[s0].copy(), v[s0].copy()
        for j in range(s0 + 1, i + 1):
            zj = zi * alpha[j] + w[j]
            ki = (alpha[j] * ki * zi + k[j] * w[j]) / zj
            vi = (alpha[j] * vi * zi + v[j] * w[j]) / zj
            zi = zj
        z[i], kt[i], vt[i] = zi, ki, vi
    return kt, vt, z, alpha


def training_mask(alpha) -> np.ndarray:
    """Additive mask of the masking figure for binary alpha: row i (query),
    column j (state): 0 if j == i, log(1 - alpha_{j+1}) if j < i, -inf if j > i."""
    n = len(alpha)
    with np.errstate(divide="ignore"):
        lg = np.log(1.0 - np.asarray(alpha, dtype=f64))
    M = np.full((n, n), -np.inf, dtype=f64)
    for i in range(n):
        M[i, i] = 0.0
        for j in range(i):
            M[i, j] = lg[j + 1]
    return M


def masked_attention(k, v, q, window: int = 0):
    """Outputs of every token of one sequence, training formulation.

    k, v [n, d]; q [n, G, d]. The score of query i against state j is
    q_i[1:]^T k~_j[1:] / sqrt(d_h) + M[i, j] (masking appendix). Returns
    [n, G, d]."""
    q = np.array(q, dtype=f64)
    if window > 0:
        kt, vt, _, alpha = unrolled_states_window(k, v, q[:, :, 0], window)
    else:
        kt, vt, _, alpha = unrolled_states(k, v, q[:, :, 0])
    q[:, :, 0] = 0.0
    M = training_mask(alpha)
    n, G, d = q.shape
    out = np.zeros((n, G, d), dtype=f64)
    for g in range(G):
        S = (q[:, g, :] @ kt.T) / np.sqrt(f64(d)) + M
        S = S - S.max(axis=1, keepdims=True)
        P = np.exp(S)
        P = P / P.sum(axis=1, keepdims=True)
        out[:, g, :] = P @ vt
    return out
