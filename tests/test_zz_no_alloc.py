"""GPU check of hsa_partition_static, the partition entry point that takes no
workspace: it serves callers that cannot allocate device memory themselves
(for example a plugin inside a framework that owns all device memory, or a
loop that must not call cudaMalloc because it can synchronise the device).

Through the C ABI it must give exactly what hsa_partition gives with a
caller-provided workspace, on calls in a row: the first large enough for the
radix sort that works in the fixed scratch, the second a smaller sort in the
same scratch (anything the first left there would show), then sizes served by
the paths that need no scratch, and a sort again; and it must refuse inputs
larger than its fixed scratch before launching.
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
    # first call: the largest size accepted, a radix sort in the fixed scratch
    N0 = hsa.HSA_PARTITION_STATIC_MAX_TOKENS
    stat0 = synth.lognormal_stat(N0, 1.0, 9).cuda()
    budgets0, counts0 = (40, 20, 10, 5), (N0 // 4, N0 // 4, N0 // 4, N0 - 3 * (N0 // 4))
    ref0 = _with_workspace(hsa, stat0, 40, budgets0, counts0)
    got0 = _static_c_abi(hsa, stat0, 40, budgets0, counts0)
    torch.cuda.synchronize()
    assert torch.equal(got0, ref0)

    # a smaller sort in the same scratch, with ties across group boundaries
    Ns = 400003
    g = torch.Generator().manual_seed(3)
    stats = torch.rand(Ns, generator=g)
    stats[1000:90000] = stats[5]
    stats = stats.cuda()
    budgets_s, counts_s = (40, 10), (150001, 250002)
    ref_s = _with_workspace(hsa, stats, 40, budgets_s, counts_s)
    got_s = _static_c_abi(hsa, stats, 40, budgets_s, counts_s)
    torch.cuda.synchronize()
    assert torch.equal(got_s, ref_s)

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

    # a size the cluster boundary select serves
    N3 = 30000
    stat3 = synth.lognormal_stat(N3, 1.0, 5).cuda()
    budgets3, counts3 = (40, 20, 10, 5), (7000, 8000, 9000, 6000)
    ref3 = _with_workspace(hsa, stat3, 40, budgets3, counts3)
    got3 = _static_c_abi(hsa, stat3, 40, budgets3, counts3)
    torch.cuda.synchronize()
    assert torch.equal(got3, ref3)

    # and a sort in the scratch again after the paths that do not use it
    got4 = _static_c_abi(hsa, stat0, 40, budgets0, counts0)
    torch.cuda.synchronize()
    assert torch.equal(got4, ref0)
    assert hsa.hsa_get_device_error() == 0


def test_static_partition_rejects_oversize(hsa):
    N = hsa.HSA_PARTITION_STATIC_MAX_TOKENS + 1
    stat = torch.rand(N, device="cuda")
    g = torch.empty(N, dtype=torch.int32, device="cuda")
    with pytest.raises(hsa.HsaError) as e:
        hsa.hsa_partition_static(stat, 8, (8,), (N,), g)
    assert e.value.status == -4
