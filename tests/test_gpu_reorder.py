"""GPU parity of token reordering (Sec. 2.5): the permutation is bit-exact
against the oracle; attention over the cached non-baseline prefix followed by
the fresh baseline K/V matches the oracle's attention over those keys; a whole
schedule run in reordered form gives, permuted back, the same attention
outputs as the oracle's run over the full cache."""
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


def _check(got, ref, dtype):
    got = got.double().cpu()
    err = (got - ref).abs().max().item()
    if dtype == "f32":
        assert err <= 1e-4, err
    else:
        rl2 = ((got - ref).norm() / ref.norm()).item()
        assert err <= 2e-2 and rl2 <= 1e-2, (err, rl2)


def _gpu_reorder(hsa, g, n_base, offset=0):
    N = g.numel()
    buf = torch.zeros(N + offset, dtype=torch.int32, device=DEV)
    buf[offset:] = g.to(DEV)
    order = torch.full((N,), -1, dtype=torch.int32, device=DEV)
    where = torch.full((N,), -1, dtype=torch.int32, device=DEV)
    gn = torch.full((N,), -1, dtype=torch.int32, device=DEV)
    hsa.hsa_reorder_tokens(buf[offset:], n_base, order, where, gn)
    return order.cpu(), where.cpu(), gn.cpu()


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_reorder_workloads(hsa, name):
    w = synth.WORKLOADS[name]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    order, where, gn, M = oracle.reorder(g)
    for offset in (0, 1):
        got = _gpu_reorder(hsa, g, counts[0], offset)
        assert torch.equal(got[0], order) and torch.equal(got[1], where)
        assert torch.equal(got[2], gn)
    assert hsa.hsa_get_device_error() == 0


@pytest.mark.parametrize("N", [1, 5, 4097, 70001])
def test_reorder_ragged(hsa, N):
    g = torch.randint(0, 3, (N,), generator=torch.Generator().manual_seed(N), dtype=torch.int32)
    order, where, gn, M = oracle.reorder(g)
    got = _gpu_reorder(hsa, g, N - M)
    assert torch.equal(got[0], order) and torch.equal(got[1], where) and torch.equal(got[2], gn)
    assert hsa.hsa_get_device_error() == 0


def test_reorder_inconsistent_count_is_reported(hsa):
    g = torch.tensor([0, 1, 0, 2], dtype=torch.int32)
    _gpu_reorder(hsa, g, 3)          # only two baseline tokens exist
    assert hsa.hsa_get_device_error() == -6


@pytest.mark.parametrize("M,B,H,D,n_act,dtype,indexed", [
    (1000, 300, 2, 128, 700, "bf16", True),
    (257, 129, 3, 64, 386, "bf16", False),
    (0, 500, 1, 128, 500, "bf16", False),        # every token in the baseline group
    (640, 0, 2, 128, 200, "bf16", True),         # no baseline tokens
    (4000, 1000, 2, 128, 2345, "bf16", True),
    (300, 100, 2, 64, 200, "f32", True),
])
def test_prefix_attention(hsa, M, B, H, D, n_act, dtype, indexed):
    N = M + B
    q = synth.normal((N if indexed else n_act, H, D), 1, dtype)
    kc, vc = synth.normal((M, H, D), 2, dtype), synth.normal((M, H, D), 3, dtype)
    kb, vb = synth.normal((B, H, D), 4, dtype), synth.normal((B, H, D), 5, dtype)
    idx = synth.uniform_subset(N, n_act, 6) if indexed else None
    ref = oracle.attention(q, torch.cat([kc, kb]).contiguous(), torch.cat([vc, vb]).contiguous(),
                           q_idx=idx)
    for ws_on in (False, True):
        ws = None
        if ws_on:
            nb = hsa.hsa_active_attention_workspace_bytes(n_act, N, H, D,
                                                          0 if dtype == "bf16" else 1)
            ws = torch.empty(max(nb, 1), dtype=torch.uint8, device=DEV)
        out = torch.full((n_act, H, D), 5.0, device=DEV).to(q.dtype)
        hsa.hsa_active_attention_prefix(q.to(DEV), None if idx is None else idx.to(DEV), n_act,
                                        kc.to(DEV), vc.to(DEV), kb.to(DEV), vb.to(DEV), out,
                                        workspace=ws)
        assert hsa.hsa_get_device_error() == 0
        _check(out, ref, dtype)


@pytest.mark.parametrize("D", [128, 64])
def test_prefix_attention_reversed_waves(hsa, D):
    """Enough units (8 heads x 24 query blocks = 192) that those past the first wave
    of CTAs walk their keys backwards, starting in the ragged last tile of the second
    source; both sources end in a ragged tile (5000 = 39 x 128 + 8 cache rows, 1500
    = 11 x 128 + 92 fresh rows).  The oracle checks sampled rows of a head whose
    units run forwards (0), one whose units are split between the two directions
    (6) and one whose units all run backwards (7), with and without the split-tail
    workspace."""
    M, B, H, n_act = 5000, 1500, 8, 6000
    N = M + B
    q = synth.normal((N, H, D), 41, "bf16")
    kc, vc = synth.normal((M, H, D), 42, "bf16"), synth.normal((M, H, D), 43, "bf16")
    kb, vb = synth.normal((B, H, D), 44, "bf16"), synth.normal((B, H, D), 45, "bf16")
    idx = synth.uniform_subset(N, n_act, 46)
    k_all, v_all = torch.cat([kc, kb]), torch.cat([vc, vb])
    g = torch.Generator().manual_seed(47)
    rows = torch.unique(torch.cat([torch.randperm(n_act, generator=g)[:24],
                                   torch.arange(n_act - 12, n_act), torch.arange(0, 4)]))
    outs = []
    for ws_on in (False, True):
        ws = None
        if ws_on:
            nb = hsa.hsa_active_attention_workspace_bytes(n_act, N, H, D, 0)
            ws = torch.empty(max(nb, 1), dtype=torch.uint8, device=DEV)
        out = torch.full((n_act, H, D), 5.0, device=DEV).to(torch.bfloat16)
        hsa.hsa_active_attention_prefix(q.to(DEV), idx.to(DEV), n_act, kc.to(DEV), vc.to(DEV),
                                        kb.to(DEV), vb.to(DEV), out, workspace=ws)
        assert hsa.hsa_get_device_error() == 0
        outs.append(out.cpu())
    for h in (0, 6, 7):
        ref = oracle.attention(q[:, h:h + 1].contiguous(), k_all[:, h:h + 1].contiguous(),
                               v_all[:, h:h + 1].contiguous(), q_idx=idx[rows])
        for out in outs:
            _check(out[rows, h:h + 1], ref, "bf16")


def test_reordered_schedule_matches_full_cache(hsa):
    """T = 40 schedule with four groups.  GPU, reordered: gather of the token
    rows by `order`, prefix-only cache, scatter of the active non-baseline
    K/V, attention over cache + fresh baseline K/V.  Oracle, not reordered:
    full N-row cache.  Attention outputs agree (rows permuted back)."""
    N, H, D, T = 1500, 2, 128, 40
    budgets, counts = (40, 20, 10, 5), (300, 300, 400, 500)
    stat = synth.lognormal_stat(N, 1.0, 21)
    g = oracle.partition(stat, T, budgets, counts)
    order_ref, where_ref, gn_ref, M = oracle.reorder(g)
    order, where, gn = (t.to(DEV) for t in _gpu_reorder(hsa, g, counts[0]))
    # initial full cache (oracle) and its reordered prefix (GPU, via gather)
    kc_full, vc_full = synth.normal((N, H, D), 31, "bf16"), synth.normal((N, H, D), 32, "bf16")
    kc_pre = torch.empty((M, H, D), dtype=torch.bfloat16, device=DEV)
    vc_pre = torch.empty_like(kc_pre)
    hsa.hsa_gather_active(kc_full.to(DEV), order, M, kc_pre)
    hsa.hsa_gather_active(vc_full.to(DEV), order, M, vc_pre)
    idx = torch.empty(N, dtype=torch.int32, device=DEV)
    ws = torch.empty(hsa.hsa_active_attention_workspace_bytes(N, N, H, D), dtype=torch.uint8,
                     device=DEV)
    for it in range(T):
        kf = synth.normal((N, H, D), 1000 + it, "bf16")     # fresh K/V/Q, old order
        vf = synth.normal((N, H, D), 2000 + it, "bf16")
        q = synth.normal((N, H, D), 3000 + it, "bf16")
        idx_old, _ = oracle.active_set(g, T, budgets, it)
        oracle.kv_scatter(kc_full, vc_full, kf[idx_old.long()].contiguous(),
                          vf[idx_old.long()].contiguous(), idx_old)
        # GPU in reordered form
        n = hsa.hsa_active_count(budgets, counts, T, it)
        hsa.hsa_partition_active(gn, T, budgets, it, idx)
        nb = n - counts[0]
        new_idx = idx[:n].cpu().long()
        old_rows = order_ref[new_idx].long()                 # tokens of A_i, new order
        kf_new = kf[old_rows].contiguous().to(DEV)
        vf_new = vf[old_rows].contiguous().to(DEV)
        hsa.hsa_kv_sync_scatter(kc_pre, vc_pre, kf_new[:nb].contiguous(),
                                vf_new[:nb].contiguous(), idx[:nb].contiguous(), nb)
        out = torch.empty((n, H, D), dtype=torch.bfloat16, device=DEV)
        hsa.hsa_active_attention_prefix(q[old_rows].contiguous().to(DEV), None, n, kc_pre, vc_pre,
                                        kf_new[nb:].contiguous(), vf_new[nb:].contiguous(), out,
                                        workspace=ws)
        if it % 7 == 0:
            ref = oracle.attention(q, kc_full, vc_full, q_idx=idx_old)
            perm = torch.argsort(old_rows)                   # new-order rows -> old order
            _check(out.cpu()[perm], ref, "bf16")
    # the prefix cache equals the full cache's non-baseline rows
    assert torch.equal(kc_pre.cpu(), kc_full[order_ref[:M].long()])
    assert torch.equal(vc_pre.cpu(), vc_full[order_ref[:M].long()])
    assert hsa.hsa_get_device_error() == 0
