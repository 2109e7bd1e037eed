"""The hot path inside a CUDA graph.  The library allocates nothing and does
all of its host work (argument checks, tensor-map encoding, the tail plan)
before enqueueing, so a whole step (partition, then one iteration's active
set, gather, KV-sync scatter, attention with the split-tail workspace and
cached Euler) can be captured once and replayed.  A replay must give exactly
the eager results, which are themselves checked against the oracle."""
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


@pytest.mark.parametrize("D,it", [(128, 1), (64, 0)])
def test_step_replayed_from_cuda_graph(hsa, D, it):
    N, H, C, T = 3001, 3, 16, 8
    budgets, counts = (8, 4, 2), (601, 900, 1500)
    stat = synth.lognormal_stat(N, 1.0, 40 + D)
    g_ref = oracle.partition(stat, T, budgets, counts)
    idx_ref, pos_ref = oracle.active_set(g_ref, T, budgets, it)
    n = idx_ref.numel()
    sig = oracle.sigmas(T)
    ds = float(sig[it + 1] - sig[it])

    hid = synth.normal((N, H * D), 41, "bf16").to(DEV)
    q = synth.normal((N, H, D), 42, "bf16").to(DEV)
    kc0, vc0 = synth.normal((N, H, D), 43, "bf16"), synth.normal((N, H, D), 44, "bf16")
    kf = synth.normal((n, H, D), 45, "bf16").to(DEV)
    vf = synth.normal((n, H, D), 46, "bf16").to(DEV)
    x0, vh0 = synth.normal((N, C), 47), synth.normal((N, C), 48)
    vfr = synth.normal((n, C), 49).to(DEV)
    stat_d = stat.to(DEV)

    state = dict(kc=kc0.to(DEV), vc=vc0.to(DEV), x=x0.to(DEV), vh=vh0.to(DEV))
    outs = dict(g=torch.empty(N, dtype=torch.int32, device=DEV),
                idx=torch.empty(N, dtype=torch.int32, device=DEV),
                pos=torch.empty(N, dtype=torch.int32, device=DEV),
                gathered=torch.empty((n, H * D), dtype=torch.bfloat16, device=DEV),
                att=torch.empty((n, H, D), dtype=torch.bfloat16, device=DEV))
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(N), dtype=torch.uint8, device=DEV)
    ws_att = torch.empty(hsa.hsa_active_attention_workspace_bytes(n, N, H, D),
                         dtype=torch.uint8, device=DEV)

    def reset():
        state["kc"].copy_(kc0)
        state["vc"].copy_(vc0)
        state["x"].copy_(x0)
        state["vh"].copy_(vh0)
        for t in outs.values():
            t.fill_(-7)

    def step():
        hsa.hsa_partition(stat_d, T, budgets, counts, outs["g"], ws)
        hsa.hsa_partition_active(outs["g"], T, budgets, it, outs["idx"], outs["pos"])
        hsa.hsa_gather_active(hid, outs["idx"], n, outs["gathered"])
        hsa.hsa_kv_sync_scatter(state["kc"], state["vc"], kf, vf, outs["idx"], n)
        hsa.hsa_active_attention(q, outs["idx"], n, state["kc"], state["vc"], outs["att"],
                                 workspace=ws_att)
        hsa.hsa_cached_euler(state["x"], state["vh"], vfr, outs["pos"], ds, n)

    # eager pass (also the warm-up that resolves per-device setup)
    reset()
    step()
    torch.cuda.synchronize()
    assert hsa.hsa_get_device_error() == 0
    eager = {k: v.clone() for k, v in {**outs, **state}.items()}

    # the eager pass against the oracle
    assert torch.equal(eager["g"].cpu(), g_ref)
    assert torch.equal(eager["idx"][:n].cpu(), idx_ref)
    assert torch.equal(eager["pos"].cpu(), pos_ref)
    assert torch.equal(eager["gathered"].cpu(), oracle.gather(hid.cpu(), idx_ref))
    kc_ref, vc_ref = kc0.clone(), vc0.clone()
    oracle.kv_scatter(kc_ref, vc_ref, kf.cpu(), vf.cpu(), idx_ref)
    assert torch.equal(eager["kc"].cpu(), kc_ref) and torch.equal(eager["vc"].cpu(), vc_ref)
    x_ref, vh_ref = x0.clone(), vh0.clone()
    oracle.cached_euler_f32(x_ref, vh_ref, vfr.cpu(), pos_ref, ds)
    assert torch.equal(eager["x"].cpu(), x_ref) and torch.equal(eager["vh"].cpu(), vh_ref)
    rows = torch.arange(0, n, max(1, n // 40))
    ref = oracle.attention(q.cpu(), kc_ref, vc_ref, q_idx=idx_ref[rows])
    got = eager["att"][rows].double().cpu()
    assert (got - ref).abs().max().item() <= 2e-2
    assert ((got - ref).norm() / ref.norm()).item() <= 1e-2

    # capture once, replay twice from the reset state: bit-identical to eager
    reset()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for _ in range(2):
        reset()
        torch.cuda.synchronize()
        graph.replay()
        torch.cuda.synchronize()
        assert hsa.hsa_get_device_error() == 0
        for k in eager:
            got = {**outs, **state}[k]
            assert torch.equal(got, eager[k]), k
