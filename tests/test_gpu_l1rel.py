"""GPU parity of hsa_cached_euler_l1rel: the cached Euler step fused with the
velocity statistic of the dynamic token selection (App. B, Eq. 7).

Bars: x and the velocity cache bit-exact against the oracle's fp32 Euler
mirror; the statistic within 5e-5 relative of the fp64 oracle (fp32 sums of C
absolute values, one division and one fused multiply-add per step)."""
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu
DEV = "cuda"
RTOL = 5e-5


@pytest.fixture(scope="module")
def hsa():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2605_06892_gb300 as m
    m.lib()
    torch.cuda.set_device(0)
    assert m.hsa_get_device_error() == 0
    return m


def _step(hsa, x, vh, vfr, pos, ds, stat_d, stat_ref, weight):
    x_d, vh_d = x.to(DEV), vh.to(DEV)
    hsa.hsa_cached_euler_l1rel(x_d, vh_d, vfr.to(DEV), pos.to(DEV), ds, stat_d, weight)
    oracle.l1rel_accumulate(vh, vfr, pos, weight, stat_ref)
    oracle.cached_euler_f32(x, vh, vfr, pos, ds)
    assert torch.equal(x_d.cpu(), x) and torch.equal(vh_d.cpu(), vh)


@pytest.mark.parametrize("N,C", [(1024, 16), (6144, 128), (777, 12), (300, 20), (500, 256)])
def test_l1rel_step_parity(hsa, N, C):
    x, vh = synth.normal((N, C), 1), synth.normal((N, C), 2)
    idx = synth.uniform_subset(N, N // 2, 3)
    pos = torch.full((N,), -1, dtype=torch.int32)
    pos[idx.long()] = torch.arange(idx.numel(), dtype=torch.int32)
    stat_d = torch.full((N,), 0.25, device=DEV)
    stat_ref = torch.full((N,), 0.25, dtype=torch.float64)
    for s in range(3):
        vfr = synth.normal((idx.numel(), C), 10 + s)
        _step(hsa, x, vh, vfr, pos, -0.025, stat_d, stat_ref, 1.0 / 3.0)
    got = stat_d.cpu().double()
    assert torch.all((got - stat_ref).abs() <= RTOL * stat_ref.abs() + 1e-7)
    skipped = pos < 0
    assert torch.all(got[skipped] == 0.25)
    assert hsa.hsa_get_device_error() == 0


def test_l1rel_zero_denominator(hsa):
    N, C = 64, 16
    x, vh = torch.zeros(N, C), synth.normal((N, C), 5)
    vh[:32] = 0.0
    pos = torch.arange(N, dtype=torch.int32)
    vfr = torch.zeros(N, C)
    stat_d = torch.zeros(N, device=DEV)
    stat_ref = torch.zeros(N, dtype=torch.float64)
    _step(hsa, x, vh, vfr, pos, -0.1, stat_d, stat_ref, 1.0)
    got = stat_d.cpu()
    assert torch.all(got[:32] == 0.0)
    assert torch.all(got[32:] == torch.tensor(3.4028234663852886e38, dtype=torch.float32))


def test_dynamic_selection_pipeline(hsa):
    """The first m = 10 iterations run every token (window 50 %, T = 40); the
    statistic accumulates over steps 1..9 with weight 1/9 and then drives the
    partition.  The GPU statistic matches the oracle's; partitioning the GPU
    statistic on the GPU equals the oracle's partition of the same values."""
    w = synth.WORKLOADS["ltx"]
    N, C, T = w.N, w.C, w.T
    m = oracle.margin(T, 50)
    sig = oracle.sigmas(T, w.shift)
    x, vh = synth.normal((N, C), 1), torch.zeros(N, C)
    pos = torch.arange(N, dtype=torch.int32)
    stat_d = torch.zeros(N, device=DEV)
    stat_ref = torch.zeros(N, dtype=torch.float64)
    base = synth.normal((N, C), 2)
    for i in range(m):
        # velocities drifting at token-dependent rates
        vfr = base + 0.05 * i * synth.normal((N, C), 100 + i) * (torch.arange(N) % 7).unsqueeze(1)
        ds = float(sig[i + 1] - sig[i])
        if i == 0:
            x_d, vh_d = x.to(DEV), vh.to(DEV)
            hsa.hsa_cached_euler(x_d, vh_d, vfr.to(DEV), pos.to(DEV), ds)
            oracle.cached_euler_f32(x, vh, vfr, pos, ds)
            assert torch.equal(x_d.cpu(), x)
        else:
            _step(hsa, x, vh, vfr, pos, ds, stat_d, stat_ref, 1.0 / (m - 1))
    got = stat_d.cpu()
    assert torch.all((got.double() - stat_ref).abs() <= RTOL * stat_ref.abs() + 1e-7)
    g = torch.empty(N, dtype=torch.int32, device=DEV)
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(N), dtype=torch.uint8, device=DEV)
    hsa.hsa_partition(stat_d, T, w.budgets, w.counts, g, ws)
    assert torch.equal(g.cpu(), oracle.partition(got, T, w.budgets, w.counts))
    assert hsa.hsa_get_device_error() == 0
