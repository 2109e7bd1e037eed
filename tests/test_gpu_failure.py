"""Failure detection on the GPU without a fault: the attention kernel's
bounded pipeline wait is made to run out (through the test hook the first
value tile is never loaded), the call reports HSA_ERR_TIMEOUT through the device error
word, and the same CUDA context then runs a normal call correctly."""
import time

import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hsa():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2605_06892_gb300 as m
    m.lib()
    torch.cuda.set_device(0)
    assert m.hsa_get_device_error() == 0
    return m


def test_attention_wait_timeout_is_reported_and_context_survives(hsa):
    N, H, D, n = 256, 1, 128, 200
    q = synth.normal((n, H, D), 1, "bf16").cuda()
    kc = synth.normal((N, H, D), 2, "bf16").cuda()
    vc = synth.normal((N, H, D), 3, "bf16").cuda()
    out = torch.empty((n, H, D), dtype=torch.bfloat16, device="cuda")
    assert hsa.hsa_test_inject_attention_stall(1) == 0
    try:
        t0 = time.time()
        hsa.hsa_active_attention(q, None, n, kc, vc, out)
        status = hsa.hsa_get_device_error()          # synchronises
        elapsed = time.time() - t0
    finally:
        hsa.hsa_test_inject_attention_stall(0)
    assert status == -7                               # HSA_ERR_TIMEOUT
    assert elapsed < 30.0
    # the context is intact: a normal call on it matches the oracle
    hsa.hsa_active_attention(q, None, n, kc, vc, out)
    assert hsa.hsa_get_device_error() == 0
    ref = oracle.attention(q.cpu(), kc.cpu(), vc.cpu())
    assert (out.cpu().double() - ref).abs().max() <= 2e-2


def test_inject_hook_rejects_unknown_mode(hsa):
    with pytest.raises(hsa.HsaError):
        hsa.hsa_test_inject_attention_stall(5)
    assert hsa.hsa_test_inject_attention_stall(0) == 0
