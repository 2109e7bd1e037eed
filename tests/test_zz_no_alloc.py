"""GPU check of hsa_partition_static, the partition entry point that takes no
workspace: it serves callers that cannot allocate device memory themselves
(for example a plugin inside a framework that owns all device memory, or a
loop that must not call cudaMalloc because it can synchronise the device).

Through the C ABI it must give exactly what hsa_partition gives with a
caller-provided workspace, on calls in a row (the second with a smaller
input, so anything left in the shared scratch by the first call would show,
the third at a size served by another partition path),
and it must refuse inputs larger than its fixed scratch before launching.
This file is collected last on purpose.
"""
import ctypes

import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hsa():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2605_06892_gb300 as m
    m.lib()
    torch.cuda.set_device(0)
    return m


def _with_workspace(hsa, stat, T, budgets, counts):
    g = torch.full((stat.numel(),), -1, dtype=torch.int32, device="cuda")
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(stat.numel()), dtype=torch.uint8,
                     device="cuda")
    hsa.hsa_partition(stat, T, budgets, counts, g, ws)
    return g


def _static_c_abi(hsa, stat, T, budgets, counts):
    """Direct ctypes call of the C entry point (no Python wrapper)."""
    N = stat.numel()
    g = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    b = (ctypes.c_int * len(budgets))(*budgets)
    c = (ctypes.c_int * len(counts))(*counts)
    st = hsa.lib().hsa_partition_static(stat.data_ptr(), N, T, b, c, len(budgets),
                                        g.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert st == 0, hsa.hsa_status_string(st)
    return g


def test_static_partition_matches_workspace_partition_twice(hsa):
    w = synth.WORKLOADS["wan14b_720p"]
    stat1, counts1 = synth.stat_for(w)
    stat1 = stat1.cuda()
    ref1 = _with_workspace(hsa, stat1, w.T, w.budgets, counts1)
    got1 = _static_c_abi(hsa, stat1, w.T, w.budgets, counts1)
    torch.cuda.synchronize()
    assert torch.equal(got1, ref1)

    # second call: fewer tokens, heavy ties, different groups
    N2 = 5003
    g = torch.Generator().manual_seed(2)
    stat2 = torch.tensor([-0.0, 0.0, 1.0, 2.0])[torch.randint(0, 4, (N2,), generator=g)].cuda()
    budgets2, counts2 = (20, 10, 5), (1000, 2003, 2000)
    ref2 = _with_workspace(hsa, stat2, 20, budgets2, counts2)
    got2 = _static_c_abi(hsa, stat2, 20, budgets2, counts2)
    torch.cuda.synchronize()
    assert torch.equal(got2, ref2)

    # third call: a size the one-block boundary select serves
    N3 = 30000
    stat3 = synth.lognormal_stat(N3, 1.0, 5).cuda()
    budgets3, counts3 = (40, 20, 10, 5), (7000, 8000, 9000, 6000)
    ref3 = _with_workspace(hsa, stat3, 40, budgets3, counts3)
    got3 = _static_c_abi(hsa, stat3, 40, budgets3, counts3)
    torch.cuda.synchronize()
    assert torch.equal(got3, ref3)
    assert hsa.hsa_get_device_error() == 0


def test_static_partition_rejects_oversize(hsa):
    N = hsa.HSA_PARTITION_STATIC_MAX_TOKENS + 1
    stat = torch.rand(N, device="cuda")
    g = torch.empty(N, dtype=torch.int32, device="cuda")
    with pytest.raises(hsa.HsaError) as e:
        hsa.hsa_partition_static(stat, 8, (8,), (N,), g)
    assert e.value.status == -4
