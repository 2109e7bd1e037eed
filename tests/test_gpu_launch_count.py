"""The library's launch counter (hsa_launch_count) on the GPU: each entry point
adds the number of kernels it enqueues, which is what the bench reports as its
launch count.  Partition of a layer of at most 360448 tokens is one launch (a
ranking up to 12032 tokens, then a boundary select on one cluster of 8 CTAs);
larger layers take the 4-pass radix sort (key, then histogram + scan + scatter
per pass) plus the group assignment.  The active set is one launch at any
size.  bf16 attention with a workspace
adds a combine launch exactly when its last wave is split along the keys."""
import pytest
import torch

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
    return m


def _delta(hsa, fn):
    c0 = hsa.hsa_launch_count()
    fn()
    torch.cuda.synchronize()
    return hsa.hsa_launch_count() - c0


def test_launch_counts(hsa):
    N, H, D, T = 4096, 2, 128, 8
    budgets, counts = (8, 4), (1024, 3072)
    stat = synth.lognormal_stat(N, 1.0, 3).to(DEV)
    g = torch.empty(N, dtype=torch.int32, device=DEV)
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(N), dtype=torch.uint8, device=DEV)
    # up to 360448 tokens the partition takes one launch (rank by count, then
    # the cluster boundary select); beyond, the radix sort takes fourteen
    assert _delta(hsa, lambda: hsa.hsa_partition(stat, T, budgets, counts, g, ws)) == 1
    for Nb, launches in ((20000, 1), (75600, 1), (360448, 1), (360449, 14)):
        stat_b = synth.lognormal_stat(Nb, 1.0, 4).to(DEV)
        g_b = torch.empty(Nb, dtype=torch.int32, device=DEV)
        ws_b = torch.empty(hsa.hsa_partition_workspace_bytes(Nb), dtype=torch.uint8, device=DEV)
        assert _delta(hsa, lambda: hsa.hsa_partition(stat_b, T, budgets,
                                                     (Nb // 4, Nb - Nb // 4), g_b,
                                                     ws_b)) == launches
    idx = torch.empty(N, dtype=torch.int32, device=DEV)
    pos = torch.empty(N, dtype=torch.int32, device=DEV)
    assert _delta(hsa, lambda: hsa.hsa_partition_active(g, T, budgets, 0, idx, pos)) == 1
    Nl = 2097153                                     # above the one-cluster active set
    g_l = torch.zeros(Nl, dtype=torch.int32, device=DEV)
    i_l = torch.empty(Nl, dtype=torch.int32, device=DEV)
    assert _delta(hsa, lambda: hsa.hsa_partition_active(g_l, T, budgets, 1, i_l, None)) == 1
    n = N
    rows = synth.normal((N, H * D), 1, "bf16").to(DEV)
    out = torch.empty_like(rows)
    assert _delta(hsa, lambda: hsa.hsa_gather_active(rows, idx, n, out)) == 1
    kc, vc = (synth.normal((N, H, D), s, "bf16").to(DEV) for s in (2, 3))
    kf, vf = (synth.normal((N, H, D), s, "bf16").to(DEV) for s in (4, 5))
    assert _delta(hsa, lambda: hsa.hsa_kv_sync_scatter(kc, vc, kf, vf, idx, n)) == 1
    assert _delta(hsa, lambda: hsa.hsa_kv_sync_scatter(kc, vc, kf, vf, idx, 0)) == 0
    x, vh = synth.normal((N, 16), 6).to(DEV), synth.normal((N, 16), 7).to(DEV)
    vfr = synth.normal((N, 16), 8).to(DEV)
    assert _delta(hsa, lambda: hsa.hsa_cached_euler(x, vh, vfr, pos, -0.1)) == 1
    q = synth.normal((N, H, D), 9, "bf16").to(DEV)
    o = torch.empty((N, H, D), dtype=torch.bfloat16, device=DEV)
    # 4096 rows x 2 heads = 32 units of 256 rows: one partial wave on any GPU
    # with more SMs than units, so with a workspace its keys are split
    wsa = torch.empty(hsa.hsa_active_attention_workspace_bytes(N, N, H, D), dtype=torch.uint8,
                      device=DEV)
    assert _delta(hsa, lambda: hsa.hsa_active_attention(q, None, N, kc, vc, o)) == 1
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    expect = 2 if sms > 32 else 1
    assert _delta(hsa, lambda: hsa.hsa_active_attention(q, None, N, kc, vc, o,
                                                        workspace=wsa)) == expect
    assert hsa.hsa_get_device_error() == 0
