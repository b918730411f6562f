"""The mutant oracles of the separation checks (CPU): with no mistake they are
the oracle itself, and each mistake changes the result."""
import numpy as np

from oracle import dmc_ref as R
from tests import mutants as M


def _stream(rng, n, d, G, p_append=0.4, qs=3.0):
    k = rng.normal(size=(n, d))
    k[:, 0] = np.where(rng.random(n) < p_append, -1, 1) * (np.abs(rng.normal(size=n)) + 0.1)
    v = rng.normal(size=(n, d)) + np.repeat(rng.normal(size=((n + 15) // 16, d)), 16, axis=0)[:n]
    q = rng.normal(size=(n, G, d)) * qs
    return k, v, q


def test_exact_mode_is_the_oracle_decode():
    rng = np.random.default_rng(0)
    d, G, T, S = 16, 3, 90, 12
    k, v, q = _stream(rng, T + S, d, G)
    ref = R.run_head(k[:T], v[:T], q[:T, :, 0], k[T:], v[T:], q[T:])
    got = M.decode_outputs(k[:T], v[:T], q[:T, :, 0], k[T:], v[T:], q[T:])
    np.testing.assert_allclose(got["exact"], ref["out"], rtol=0, atol=1e-12)
    for m in M.MODES:
        assert np.max(np.abs(got[m] - ref["out"])) > 1e-3, m


def test_exact_mode_is_the_oracle_prompt_attention():
    rng = np.random.default_rng(1)
    d, G, T = 16, 2, 150
    k, v, q = _stream(rng, T, d, G)
    ref = R.prompt_attention(k, v, q)
    got = M.prompt_outputs(k, v, q)
    np.testing.assert_allclose(got["exact"], ref, rtol=0, atol=1e-12)
    for m in M.MODES:
        assert np.max(np.abs(got[m] - ref)) > 1e-3, m


def test_uniform_mutant_is_the_mean_of_the_slots():
    rng = np.random.default_rng(2)
    d, G, T, S = 8, 1, 40, 3
    k, v, q = _stream(rng, T + S, d, G)
    got = M.decode_outputs(k[:T], v[:T], q[:T, :, 0], k[T:], v[T:], q[T:])
    cache = R.HeadCache(d)
    for t in range(T + S):
        R.update(cache, k[t], v[t], int(R.decision(k[t, 0])), float(R.importance(q[t, :, 0])))
    _, V, _ = cache.arrays()
    np.testing.assert_allclose(got["uniform"][-1, 0], V.mean(axis=0), rtol=0, atol=1e-12)


def test_droppage_mutant_leaves_out_one_page():
    rng = np.random.default_rng(3)
    d, G, T, S = 8, 1, 200, 2
    k, v, q = _stream(rng, T + S, d, G, p_append=1.0)  # every token its own slot
    got = M.decode_outputs(k[:T], v[:T], q[:T, :, 0], k[T:], v[T:], q[T:])
    p = got["drop_page"]
    kk, vv = k.copy(), v.copy()
    kk[:, 0] = 0.0
    keep = np.ones(T + S, dtype=bool)
    keep[p * 32:(p + 1) * 32] = False
    qq = q[-1, 0].copy()
    qq[0] = 0.0
    s = kk[keep] @ qq / np.sqrt(d)
    w = np.exp(s - s.max())
    np.testing.assert_allclose(got["droppage"][-1, 0], (w / w.sum()) @ vv[keep], rtol=0, atol=1e-12)
