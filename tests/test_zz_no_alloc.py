"""dmc_decode_step_static_scratch against dmc_decode_step (GPU).

The static-scratch entry point serves callers that cannot allocate device
memory of their own (a plugin handed only its input and output buffers by a
framework that owns every allocation, or a loop that must not pay cudaMalloc's
implicit synchronisation): its split-K scratch lives in the library's static
device array instead. It must give the same results as the regular entry
point. This file is collected last so that a failure here does not hide any
other test; it passes alone in a fresh process and after the other tests.
"""
import numpy as np
import pytest
import torch

import paper_2403_09636_gb300 as P

pytestmark = pytest.mark.gpu

TOL_BF16 = 2e-2  # the bf16 tolerance of the parity tests


def _inputs(seed, n, B, H, d, p_append):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    k = torch.randn((n, H, d), generator=g, device="cuda") * 0.5
    v = torch.randn((n, H, d), generator=g, device="cuda") * 0.5
    q = torch.randn((n, H, d), generator=g, device="cuda") * 0.5
    sign = torch.where(torch.rand((n, H), generator=g, device="cuda") < p_append, -1.0, 1.0)
    k[:, :, 0] = sign * 0.5 * (torch.randn((n, H), generator=g, device="cuda").abs() + 0.1)
    return q.bfloat16(), k.bfloat16(), v.bfloat16()


def _cache(B, H, d, T, q, k, v):
    c = P.DmcCache(1, B, H, H, d, torch.bfloat16, T + 8, B * H * (T // 32 + 2), B * T)
    cu = torch.arange(0, B * T + 1, T, dtype=torch.int32, device="cuda")
    c.prefill(0, q[:, :, 0], k, v, cu, T)
    return c


def test_static_scratch_matches_regular_decode_two_calls(cuda_dev):
    # long heads (3000 slots at CR ~1.1) are split over many blocks, so the
    # partial softmax states in the scratch carry real data
    B, H, d, T = 2, 4, 128, 3000
    q, k, v = _inputs(21, B * T, B, H, d, 0.9)
    ref = _cache(B, H, d, T, q, k, v)
    tst = _cache(B, H, d, T, q, k, v)
    s = torch.cuda.current_stream().cuda_stream
    for step in range(2):
        qd, kd, vd = (t.reshape(B, H, d) for t in _inputs(100 + step, B, B, H, d, 0.5))
        qd, kd, vd = qd.contiguous(), kd.contiguous(), vd.contiguous()
        out_ref = torch.empty_like(qd)
        out_tst = torch.full_like(qd, float("nan"))
        assert P.dmc_decode_step(ref.handle, 0, qd.data_ptr(), kd.data_ptr(), vd.data_ptr(),
                                 out_ref.data_ptr(), s) == P.DMC_OK
        assert P.dmc_decode_step_static_scratch(tst.handle, 0, qd.data_ptr(), kd.data_ptr(),
                                                vd.data_ptr(), out_tst.data_ptr(), s) == P.DMC_OK
        torch.cuda.synchronize()
        err = (out_ref.float() - out_tst.float()).abs().max().item()
        assert np.isfinite(err) and err <= TOL_BF16, (step, err)
        assert torch.equal(ref.lengths(0), tst.lengths(0))
    assert ref.status()[0] == P.DMC_OK and tst.status()[0] == P.DMC_OK


def test_static_scratch_rejects_null_handle():
    assert P.dmc_decode_step_static_scratch(None, 0, 16, 16, 16, 16, 0) == P.DMC_ERR_INVALID_ARG
