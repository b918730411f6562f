"""The C ABI on the CPU: libdmc.so builds and loads, exports every function
include/dmc.h declares, and rejects bad configs and arguments on the host
(no GPU needed: these paths return before any CUDA call)."""
import ctypes as C
import os
import re

import pytest

import paper_2403_09636_gb300 as P
from paper_2403_09636_gb300 import build as B

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "dmc.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return P.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w]+\s*\*?\s*(dmc_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_binding_names():
    assert declared_functions() == sorted(P.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def _cfg(**kw):
    base = dict(num_layers=2, batch=3, num_q_heads=8, num_kv_heads=4, head_dim=128,
                dtype=P.DMC_BF16, page_size=32, max_slots_per_head=100, num_pages=50,
                max_prefill_tokens=1000, window=0)
    base.update(kw)
    return P.dmc_cache_config(*[base[f] for f, _ in P.dmc_cache_config._fields_])


def test_required_bytes_accounts_for_the_page_pool(lib):
    a = P.dmc_cache_required_bytes(_cfg(num_pages=50))
    b = P.dmc_cache_required_bytes(_cfg(num_pages=150))
    page = 2 * 32 * 128 * 2 + 32 * 4  # K and V rows plus z
    assert a > 0 and b - a == pytest.approx(100 * page, abs=1024)


@pytest.mark.parametrize("bad", [dict(head_dim=96), dict(page_size=16), dict(num_q_heads=6),
                                 dict(dtype=7), dict(num_layers=0), dict(num_pages=0),
                                 dict(num_q_heads=132, num_kv_heads=4), dict(window=33), dict(window=-1),
                                 dict(batch=4096, num_kv_heads=8)])
def test_invalid_configs_need_zero_bytes(lib, bad):
    assert P.dmc_cache_required_bytes(_cfg(**bad)) == 0


def test_create_rejects_bad_arena_on_the_host(lib):
    cfg = _cfg()
    n = P.dmc_cache_required_bytes(cfg)
    assert P.dmc_cache_create(cfg, 0, n, 0)[0] == P.DMC_ERR_INVALID_ARG
    assert P.dmc_cache_create(cfg, 256 + 8, n, 0)[0] == P.DMC_ERR_INVALID_ARG   # misaligned
    assert P.dmc_cache_create(cfg, 4096, n - 1, 0)[0] == P.DMC_ERR_ARENA_TOO_SMALL
    assert P.dmc_cache_create(_cfg(head_dim=80), 4096, n, 0)[0] == P.DMC_ERR_INVALID_ARG


def test_null_handle_is_rejected(lib):
    assert P.dmc_decode_step(None, 0, 16, 16, 16, 16, 0) == P.DMC_ERR_INVALID_ARG
    assert P.dmc_cache_lengths(None, 0, 16, 0) == P.DMC_ERR_INVALID_ARG
    assert P.dmc_prefill_attention(None, 0, 0, 1, 16, 16, 16, 16, 1, 1, 16, 0) == P.DMC_ERR_INVALID_ARG
    assert P.dmc_cache_destroy(None) == P.DMC_OK


def test_status_strings(lib):
    for s in range(6):
        assert P.dmc_status_string(s) and P.dmc_status_string(s) != "unknown status"
    assert P.dmc_status_string(99) == "unknown status"


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(P, "_lib", None)
    monkeypatch.setattr(P, "LIB_PATH", str(tmp_path / "libdmc.so"))
    with pytest.raises(RuntimeError, match="missing"):
        P.lib()


@pytest.mark.parametrize("U", [1, 2, 5, 37, 1000, 4097])
@pytest.mark.parametrize("nb", [1, 3, 152, 304, 1024])
def test_unit_partition_inverse(U, nb):
    """The decode kernel gives block b the unit range [b*U//nb, (b+1)*U//nb)
    and finds the block holding unit u as ((u+1)*nb - 1)//U."""
    owner = {}
    for b in range(nb):
        for u in range(b * U // nb, (b + 1) * U // nb):
            owner[u] = b
    assert sorted(owner) == list(range(U))
    for u in range(U):
        assert ((u + 1) * nb - 1) // U == owner[u]
    # a run of units [a, b) is split over exactly the non-empty blocks between
    # the blocks holding its first and last unit (the combine's contributor set)
    start = lambda b: b * U // nb
    for a in range(0, U, max(1, U // 13)):
        for b in (a + 1, min(U, a + 7), U):
            want = {owner[u] for u in range(a, b)}
            bf, bl = ((a + 1) * nb - 1) // U, (b * nb - 1) // U
            got = {c for c in range(bf, bl + 1) if start(c) < start(c + 1)}
            assert got == want
