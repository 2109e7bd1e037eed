"""GPU parity of the rotary embedding of active rows (Sec. 2.3): rotation in
place and inside the KV-cache scatter, bit-exact against the oracle's fp32
mirror (same table, same fused multiply-adds, same bf16 rounding)."""
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def hsa():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2605_06892_gb300 as m
    m.lib()
    torch.cuda.set_device(0)
    assert m.hsa_get_device_error() == 0
    return m


@pytest.mark.parametrize("name", ["wan13b", "ltx", "tiny_f32", "wan14b_boxes"])
def test_rope_rows_and_scatter(hsa, name):
    w = synth.WORKLOADS[name]
    table = oracle.rope_table(w.grid, w.D)
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    idx, _ = oracle.active_set(g, w.T, w.budgets, 1)
    n = idx.numel()
    q = synth.normal((n, w.H, w.D), 1, "bf16")
    q_d = q.to(DEV)
    tab_d = table.to(DEV)
    hsa.hsa_rope_rows(q_d, idx.to(DEV), n, tab_d)
    assert torch.equal(q_d.cpu(), oracle.rope_rows(q, idx, table))
    kc = synth.normal((w.N, w.H, w.D), 2, "bf16")
    vc = synth.normal((w.N, w.H, w.D), 3, "bf16")
    kf = synth.normal((n, w.H, w.D), 4, "bf16")
    vf = synth.normal((n, w.H, w.D), 5, "bf16")
    kc_d, vc_d = kc.to(DEV), vc.to(DEV)
    hsa.hsa_kv_sync_scatter_rope(kc_d, vc_d, kf.to(DEV), vf.to(DEV), idx.to(DEV), n, tab_d)
    oracle.kv_scatter(kc, vc, oracle.rope_rows(kf, idx, table), vf, idx)
    assert torch.equal(kc_d.cpu(), kc) and torch.equal(vc_d.cpu(), vc)
    assert hsa.hsa_get_device_error() == 0


def test_rope_bad_index(hsa):
    table = oracle.rope_table((1, 2, 2), 64).to(DEV)
    x = torch.ones((2, 1, 64), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_rope_rows(x, torch.tensor([1, 9], dtype=torch.int32, device=DEV), 2, table)
    assert hsa.hsa_get_device_error() == -6
    assert torch.all(x[1] == 1.0)
