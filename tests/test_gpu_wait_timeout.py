"""The bounded in-kernel wait gives up cleanly (GPU).

The prompt-attention kernel waits for its tensor-core commits through
`mbar_wait` (dmc_internal.cuh), which gives up after a time limit, sets
DMC_FAULT_WAIT_TIMEOUT and returns, so that a lost completion cannot hang the
GPU. A test-only kernel (tests/csrc/wait_timeout_probe.cu), built here with the
limit shortened to 2 ms, waits on an mbarrier that nobody arrives at: it must
return within the limit plus scheduling noise, report failure on every thread
and set the fault bit. With the one expected arrival made first, the same
wait must succeed and leave the bit clear. No tensor-core work is in flight.
"""
import ctypes as C
import os
import subprocess

import pytest
import torch

from paper_2403_09636_gb300 import DMC_FAULT_WAIT_TIMEOUT
from paper_2403_09636_gb300 import build as B

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "csrc", "wait_timeout_probe.cu")
OUT = os.path.join(HERE, "_build", "libwaitprobe.so")
LIMIT_NS = 2_000_000


def _probe():
    os.makedirs(os.path.dirname(OUT), exist_ok=True)
    deps = [SRC, os.path.join(B.CSRC, "dmc_internal.cuh")]
    if not os.path.exists(OUT) or any(os.path.getmtime(d) > os.path.getmtime(OUT) for d in deps):
        tmp = OUT + f".tmp{os.getpid()}"
        subprocess.check_call([B.nvcc()] + B.ARCH + B.FLAGS +
                              [f"-DDMC_WAIT_LIMIT_NS={LIMIT_NS}ull", "-shared", SRC, "-o", tmp])
        os.replace(tmp, OUT)
    lib = C.CDLL(OUT)
    lib.dmc_wait_probe.argtypes = [C.c_int, C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
    return lib


@pytest.mark.parametrize("threads", [32, 256])
def test_wait_on_a_barrier_nobody_arrives_at_gives_up(cuda_dev, threads):
    lib = _probe()
    s = torch.cuda.current_stream().cuda_stream
    for arrive_first in (0, 1):
        err = torch.zeros(1, dtype=torch.int32, device=cuda_dev)
        ok = torch.full((threads,), -1, dtype=torch.int32, device=cuda_dev)
        ns = torch.zeros(1, dtype=torch.int64, device=cuda_dev)
        assert lib.dmc_wait_probe(arrive_first, threads, err.data_ptr(), ok.data_ptr(),
                                  ns.data_ptr(), s) == 0
        torch.cuda.synchronize()
        bits, waited = int(err.item()), int(ns.item())
        if arrive_first:
            assert bool((ok == 1).all()), ok.tolist()
            assert bits == 0
            assert waited < LIMIT_NS
        else:
            assert bool((ok == 0).all()), ok.tolist()
            assert bits & DMC_FAULT_WAIT_TIMEOUT
            assert LIMIT_NS <= waited < 100 * LIMIT_NS, waited
    # the context is still usable
    x = torch.ones(1024, device=cuda_dev)
    assert float(x.sum()) == 1024.0
