"""GPU parity of every libhsa call against the CPU oracle, through the C ABI.

Bars: bit-exact for the partition, the active set, gather, scatter and the
cached Euler step (against the oracle's fp32 mirror, one fused multiply-add per
element); the cached Euler step also within 1e-6 of the fp64 oracle, scaled by
the condition |x| + |v dsigma|; bf16 attention within max |err| <= 2e-2 and
relative L2 error <= 1e-2 of the fp64 oracle fed the same bf16 inputs; fp32
attention within 1e-4.
"""

import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

ATOL_BF16, RL2_BF16, ATOL_F32 = 2e-2, 1e-2, 1e-4


@pytest.fixture(scope="module")
def hsa():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2605_06892_gb300 as m
    m.lib()
    torch.cuda.set_device(0)
    assert m.hsa_get_device_error() == 0
    return m


DEV = "cuda"


def _no_device_error(hsa):
    assert hsa.hsa_get_device_error() == 0


def _check_attention(got, ref, dtype):
    got = got.double().cpu()
    err = (got - ref).abs().max().item()
    rl2 = ((got - ref).norm() / ref.norm()).item()
    if dtype == "f32":
        assert err <= ATOL_F32, err
    else:
        assert err <= ATOL_BF16 and rl2 <= RL2_BF16, (err, rl2)
    return err, rl2


# --------------------------------------------------------------- partition

def _gpu_partition(hsa, stat, T, budgets, counts):
    N = stat.numel()
    g = torch.full((N,), -7, dtype=torch.int32, device=DEV)
    ws = torch.empty(max(1, hsa.hsa_partition_workspace_bytes(N)), dtype=torch.uint8, device=DEV)
    hsa.hsa_partition(stat.to(DEV), T, budgets, counts, g, ws)
    return g.cpu()


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_partition_workloads(hsa, name):
    w = synth.WORKLOADS[name]
    stat, counts = synth.stat_for(w)
    assert torch.equal(_gpu_partition(hsa, stat, w.T, w.budgets, counts),
                       oracle.partition(stat, w.T, w.budgets, counts))
    _no_device_error(hsa)


@pytest.mark.parametrize("N", [1, 2, 31, 4095, 4096, 4097, 12289, 100003])
def test_partition_ties_signed_zero_ragged(hsa, N):
    g = torch.Generator().manual_seed(N)
    pool = torch.tensor([-0.0, 0.0, 1.0, -1.0, 2.5e-38, -3.4e38, 3.4e38, 1e-45, -1e-45])
    stat = pool[torch.randint(0, pool.numel(), (N,), generator=g)]
    budgets = (40, 20, 10, 5)
    cut = sorted(torch.randint(0, N + 1, (3,), generator=g).tolist())
    b = [0] + cut + [N]
    counts = tuple(b[k + 1] - b[k] for k in range(4))
    assert torch.equal(_gpu_partition(hsa, stat, 40, budgets, counts),
                       oracle.partition(stat, 40, budgets, counts))
    _no_device_error(hsa)


@pytest.mark.parametrize("N", [12032, 12033, 20000, 49153, 75600, 360448, 360449, 500001])
def test_partition_paths_many_and_empty_groups(hsa, N):
    """Each of the three partition paths (rank by count up to 12032 tokens, a
    cluster of 8 CTAs selecting the group boundaries up to 360448, the radix
    sort beyond) against the oracle: 1 to 32 groups with random cuts, a run of
    equal values straddling boundaries (and the CTAs' token ranges), and empty
    groups at either end."""
    g = torch.Generator().manual_seed(N)
    stat = synth.lognormal_stat(N, 1.0, 11)
    stat[N // 3: N // 3 + 3000] = stat[7]             # ties across several boundaries
    c = (((N + 7) // 8) + 3) & ~3                     # first token of the second CTA's range
    stat[max(8, c - 1500): c + 1500] = stat[7]        # ties across the CTAs' ranges
    stat[5] = -0.0
    stat[6] = 0.0
    for K in (1, 2, 5, 32):
        budgets = (40,) * K
        cut = sorted(torch.randint(0, N + 1, (K - 1,), generator=g).tolist())
        b = [0] + cut + [N]
        counts = tuple(b[k + 1] - b[k] for k in range(K))
        assert torch.equal(_gpu_partition(hsa, stat, 40, budgets, counts),
                           oracle.partition(stat, 40, budgets, counts)), (K, counts)
    lo = int((stat < stat[7]).sum())                  # a cut inside the run of ties
    for counts in ((0, N, 0), (N, 0, 0), (0, 0, N), (N - lo - 1000, 1000, lo)):
        assert torch.equal(_gpu_partition(hsa, stat, 40, (40, 20, 10), counts),
                           oracle.partition(stat, 40, (40, 20, 10), counts)), counts
    _no_device_error(hsa)


def test_partition_single_group_and_empty_groups(hsa):
    stat = synth.lognormal_stat(5000, 1.0, 3)
    for budgets, counts in (((8,), (5000,)), ((8, 4, 2), (0, 5000, 0)), ((8, 1), (4999, 1))):
        assert torch.equal(_gpu_partition(hsa, stat, 8, budgets, counts),
                           oracle.partition(stat, 8, budgets, counts))


def test_partition_errors(hsa):
    stat = torch.rand(100).to(DEV)
    g = torch.empty(100, dtype=torch.int32, device=DEV)
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(100), dtype=torch.uint8, device=DEV)
    for budgets, counts, code in (((40, 15), (50, 50), -2), ((20, 10), (50, 50), -1),
                                  ((40, 10), (50, 49), -3), ((40, 10), (-1, 101), -3)):
        with pytest.raises(hsa.HsaError) as e:
            hsa.hsa_partition(stat, 40, budgets, counts, g, ws)
        assert e.value.status == code
    with pytest.raises(hsa.HsaError) as e:
        hsa.hsa_partition(stat, 40, (40, 10), (50, 50), g, ws[:16])
    assert e.value.status == -9
    bad = stat.clone()
    bad[17] = float("nan")
    hsa.hsa_partition(bad, 40, (40, 10), (50, 50), g, ws)
    assert hsa.hsa_get_device_error() == -5
    bad[17] = float("-inf")
    hsa.hsa_partition(bad, 40, (40, 10), (50, 50), g, ws)
    assert hsa.hsa_get_device_error() == -5
    for n_big in (20000, 300000, 400000):            # the select and radix paths
        big = torch.rand(n_big).to(DEV)
        big[n_big - 3] = float("nan")
        gb = torch.empty(n_big, dtype=torch.int32, device=DEV)
        wsb = torch.empty(hsa.hsa_partition_workspace_bytes(n_big), dtype=torch.uint8, device=DEV)
        hsa.hsa_partition(big, 40, (40, 10), (n_big // 2, n_big - n_big // 2), gb, wsb)
        assert hsa.hsa_get_device_error() == -5
    _no_device_error(hsa)


@pytest.mark.parametrize("name", ["wan13b", "ltx", "wan14b_720p", "tiny_f32"])
def test_allocation_strategies_u_and_f(hsa, name):
    """U and F statistics match the oracle bit for bit and give the same
    partitions (App. B)."""
    w = synth.WORKLOADS[name]
    counts = w.counts
    st = torch.empty(w.N, device=DEV)
    hsa.hsa_uniform_stat(st)
    ref = oracle.uniform_stat(w.N)
    assert torch.equal(st.cpu(), ref)
    assert torch.equal(_gpu_partition(hsa, st.cpu(), w.T, w.budgets, counts),
                       oracle.partition(ref, w.T, w.budgets, counts))
    frame = w.grid[1] * w.grid[2]
    if counts[0] >= frame:
        rnd = torch.rand(w.N, generator=torch.Generator().manual_seed(w.cid))
        st = rnd.to(DEV)
        hsa.hsa_reserve_first_frame(st, frame)
        ref_f = oracle.reserve_frame(rnd, frame)
        assert torch.equal(st.cpu(), ref_f)
        g = _gpu_partition(hsa, st.cpu(), w.T, w.budgets, counts)
        assert torch.equal(g, oracle.partition(ref_f, w.T, w.budgets, counts))
        assert torch.all(g[:frame] == 0)
    _no_device_error(hsa)


# -------------------------------------------------------------- active set

@pytest.mark.parametrize("name", list(synth.WORKLOADS))
@pytest.mark.parametrize("window", [100, 80, 50])
def test_active_set_workloads(hsa, name, window):
    w = synth.WORKLOADS[name]
    stat, counts = synth.stat_for(w)
    g_ref = oracle.partition(stat, w.T, w.budgets, counts)
    g = g_ref.to(DEV)
    idx = torch.full((w.N,), -7, dtype=torch.int32, device=DEV)
    pos = torch.full((w.N,), -7, dtype=torch.int32, device=DEV)
    for it in range(w.T):
        idx_ref, pos_ref = oracle.active_set(g_ref, w.T, w.budgets, it, window)
        n = hsa.hsa_active_count(w.budgets, counts, w.T, it, window)
        assert n == idx_ref.numel()
        hsa.hsa_partition_active(g, w.T, w.budgets, it, idx, pos, window)
        assert torch.equal(idx[:n].cpu(), idx_ref)
        assert torch.equal(pos.cpu(), pos_ref)
    _no_device_error(hsa)


@pytest.mark.parametrize("N", [1, 7, 1000, 4096, 4097, 70001, 700001, 2097152, 2097153])
def test_active_set_ragged_and_unaligned(hsa, N):
    g_ref = torch.randint(0, 3, (N,), generator=torch.Generator().manual_seed(N),
                          dtype=torch.int32)
    budgets = (12, 6, 3)
    for offset in (0, 1):        # offset 1: group_of not 16-byte aligned
        buf = torch.zeros(N + 1, dtype=torch.int32, device=DEV)
        buf[offset:offset + N] = g_ref.to(DEV)
        g = buf[offset:offset + N]
        idx = torch.empty(N, dtype=torch.int32, device=DEV)
        pos = torch.empty(N, dtype=torch.int32, device=DEV)
        for it in (0, 1, 2, 4):
            idx_ref, pos_ref = oracle.active_set(g_ref, 12, budgets, it)
            hsa.hsa_partition_active(g, 12, budgets, it, idx, pos)
            assert torch.equal(idx[:idx_ref.numel()].cpu(), idx_ref)
            assert torch.equal(pos.cpu(), pos_ref)
    _no_device_error(hsa)


def test_active_set_bad_group(hsa):
    g = torch.zeros(50, dtype=torch.int32, device=DEV)
    g[7] = 5
    idx = torch.empty(50, dtype=torch.int32, device=DEV)
    hsa.hsa_partition_active(g, 4, (4, 2), 0, idx, None)
    assert hsa.hsa_get_device_error() == -6


# ------------------------------------------------------------------ gather

@pytest.mark.parametrize("rows,row_elems,dtype,n_act", [
    (1024, 16, "f32", 256),         # tiny latent rows, 64 B
    (1000, 12, "f32", 333),         # 48 B rows: 3 vectors, not a power of two
    (777, 4, "f32", 777),           # 16 B rows, all active
    (32760, 1536, "bf16", 8190),    # Wan-1.3B hidden rows, 3072 B
    (6144, 2048, "bf16", 1536),     # LTX hidden rows, 4096 B
    (5000, 5120, "bf16", 1),        # 10240 B rows, a single active token
    (300, 128, "f32", 0),
])
def test_gather(hsa, rows, row_elems, dtype, n_act):
    src = synth.normal((rows, row_elems), rows + row_elems, dtype)
    idx = synth.uniform_subset(rows, n_act, 5)
    dst = torch.full((max(n_act, 1), row_elems), 3.0, device=DEV).to(src.dtype)
    hsa.hsa_gather_active(src.to(DEV), idx.to(DEV), n_act, dst)
    if n_act:
        assert torch.equal(dst[:n_act].cpu(), oracle.gather(src, idx))
    _no_device_error(hsa)


def test_gather_full_size_720p(hsa):
    w = synth.WORKLOADS["wan14b_720p"]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    idx, _ = oracle.active_set(g, w.T, w.budgets, 2)
    src = synth.normal((w.N, w.H * w.D), 77, "bf16")
    dst = torch.empty((idx.numel(), w.H * w.D), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_gather_active(src.to(DEV), idx.to(DEV), idx.numel(), dst)
    assert torch.equal(dst.cpu(), oracle.gather(src, idx))


def test_gather_bad_index_skips_row(hsa):
    src = torch.arange(40, dtype=torch.float32).reshape(10, 4).to(DEV)
    idx = torch.tensor([3, 10, -1, 0], dtype=torch.int32, device=DEV)
    dst = torch.full((4, 4), -5.0, device=DEV)
    hsa.hsa_gather_active(src, idx, 4, dst)
    assert hsa.hsa_get_device_error() == -6
    assert torch.equal(dst[0].cpu(), src[3].cpu()) and torch.equal(dst[3].cpu(), src[0].cpu())
    assert torch.all(dst[1:3] == -5.0)


def test_gather_rejects_bad_args(hsa):
    src = torch.zeros(10, 3, device=DEV)        # 12-byte rows
    idx = torch.zeros(2, dtype=torch.int32, device=DEV)
    with pytest.raises(hsa.HsaError) as e:
        hsa.hsa_gather_active(src, idx, 2, torch.zeros(2, 3, device=DEV))
    assert e.value.status == -1


# ----------------------------------------------------------------- scatter

@pytest.mark.parametrize("name,frac_iter", [("tiny_f32", 1), ("wan13b", 0), ("wan13b", 1),
                                            ("ltx", 2), ("wan14b_boxes", 2),
                                            ("wan14b_720p", 1)])
def test_scatter_workloads(hsa, name, frac_iter):
    w = synth.WORKLOADS[name]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    idx, _ = oracle.active_set(g, w.T, w.budgets, frac_iter)
    n = idx.numel()
    kc = synth.normal((w.N, w.H, w.D), 101, w.dtype)
    vc = synth.normal((w.N, w.H, w.D), 102, w.dtype)
    kf = synth.normal((n, w.H, w.D), 103, w.dtype)
    vf = synth.normal((n, w.H, w.D), 104, w.dtype)
    kc_d, vc_d = kc.to(DEV), vc.to(DEV)
    hsa.hsa_kv_sync_scatter(kc_d, vc_d, kf.to(DEV), vf.to(DEV), idx.to(DEV), n)
    oracle.kv_scatter(kc, vc, kf, vf, idx)
    assert torch.equal(kc_d.cpu(), kc) and torch.equal(vc_d.cpu(), vc)
    _no_device_error(hsa)


def test_scatter_canaries_and_bad_index(hsa):
    N, H, D = 257, 3, 64
    kc = torch.full((N, H, D), 9.0, dtype=torch.bfloat16, device=DEV)
    vc = torch.full((N, H, D), -9.0, dtype=torch.bfloat16, device=DEV)
    idx = torch.tensor([0, 256, 100, 300], dtype=torch.int32)
    kf = synth.normal((4, H, D), 1, "bf16")
    vf = synth.normal((4, H, D), 2, "bf16")
    hsa.hsa_kv_sync_scatter(kc, vc, kf.to(DEV), vf.to(DEV), idx.to(DEV), 4)
    assert hsa.hsa_get_device_error() == -6
    for j in range(3):
        assert torch.equal(kc[idx[j]].cpu(), kf[j]) and torch.equal(vc[idx[j]].cpu(), vf[j])
    keep = torch.ones(N, dtype=torch.bool)
    keep[idx[:3].long()] = False
    assert torch.all(kc.cpu()[keep] == 9.0) and torch.all(vc.cpu()[keep] == -9.0)


# --------------------------------------------------------------- attention

def _workspace(hsa, n_act, N, H, D, dtype):
    nbytes = hsa.hsa_active_attention_workspace_bytes(n_act, N, H, D,
                                                      0 if dtype == "bf16" else 1)
    return torch.empty(max(nbytes, 1), dtype=torch.uint8, device=DEV)


def _attention_case(hsa, N, H, D, n_act, dtype, indexed, seed):
    """Both launch plans: without a workspace (every unit whole) and with one
    (last wave split along the keys and combined)."""
    q = synth.normal((N if indexed else n_act, H, D), seed, dtype)
    kc = synth.normal((N, H, D), seed + 1, dtype)
    vc = synth.normal((N, H, D), seed + 2, dtype)
    idx = synth.uniform_subset(N, n_act, seed + 3) if indexed else None
    ref = oracle.attention(q, kc, vc, q_idx=idx)
    res = None
    for ws in (None, _workspace(hsa, n_act, N, H, D, dtype)):
        out = torch.full((n_act, H, D), 777.0, device=DEV).to(q.dtype)
        hsa.hsa_active_attention(q.to(DEV), None if idx is None else idx.to(DEV), n_act,
                                 kc.to(DEV), vc.to(DEV), out, workspace=ws)
        _no_device_error(hsa)
        res = _check_attention(out, ref, dtype)
    return res


@pytest.mark.parametrize("N,H,D,n_act,dtype,indexed", [
    (1024, 4, 64, 256, "f32", True),       # tiny fp32 workload
    (1024, 2, 128, 256, "f32", False),
    (130, 1, 64, 77, "f32", True),         # ragged keys and queries
    (1024, 4, 64, 256, "bf16", True),
    (1000, 2, 128, 333, "bf16", True),     # ragged N (7 full tiles + 104 keys)
    (1000, 3, 64, 1000, "bf16", False),    # every token active, compact Q
    (129, 1, 128, 1, "bf16", True),        # one query, one key past a tile
    (1, 1, 64, 1, "bf16", False),          # N = 1: output is v_0
    (5000, 2, 128, 4999, "bf16", True),    # queries end one row short of N
    (2304, 2, 64, 513, "bf16", True),      # 2 full Q blocks + 1 row
])
def test_attention_small(hsa, N, H, D, n_act, dtype, indexed):
    _attention_case(hsa, N, H, D, n_act, dtype, indexed, seed=N + n_act)


def test_attention_closed_forms_gpu(hsa):
    """Identical keys give the mean of V; one dominant key gives its value."""
    N, H, D = 700, 2, 128
    q = synth.normal((64, H, D), 1, "bf16")
    k = synth.normal((1, H, D), 2, "bf16").expand(N, H, D).contiguous()
    v = synth.normal((N, H, D), 3, "bf16")
    out = torch.empty((64, H, D), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_active_attention(q.to(DEV), None, 64, k.to(DEV), v.to(DEV), out)
    mean = v.double().mean(0).expand(64, H, D)
    assert (out.cpu().double() - mean).abs().max() < 2e-2


def test_attention_large_scores_rescale(hsa):
    """Scores far above 2^8 in log2 units force the lazy rescale path."""
    N, H, D = 1500, 1, 64
    q = (synth.normal((N, H, D), 5) * 4).to(torch.bfloat16)
    kc = (synth.normal((N, H, D), 6) * 4).to(torch.bfloat16)
    vc = synth.normal((N, H, D), 7, "bf16")
    idx = synth.uniform_subset(N, 300, 8)
    out = torch.empty((300, H, D), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_active_attention(q.to(DEV), idx.to(DEV), 300, kc.to(DEV), vc.to(DEV), out)
    _check_attention(out, oracle.attention(q, kc, vc, q_idx=idx), "bf16")


@pytest.mark.parametrize("D,pos,lift", [(128, 192, 1.8), (128, 64 + 3 * 128 + 5, 1.8),
                                        (128, 739, 1.8), (128, 192, 3.0), (128, 130, 1.8),
                                        (64, 192, 2.1), (64, 739, 2.1), (64, 739, 3.0),
                                        (64, 700, 3.0), (128, 739, 3.0)])
def test_attention_late_half_peak(hsa, D, pos, lift):
    """One key whose score lies 25-45 log2 units above the scores of the
    tiles before it, in the second 64-key half of a key tile (739: of the
    ragged last tile, 100 keys; 130: in a first half instead).  Against the
    running reference of the earlier tiles its probability is 2^25 to 2^45:
    below the 2^32 bound of a tile's row sum the fast path keeps those large
    values, above it the exact path rescales O; both must give the softmax.
    With the peak in the last key tile (lift 3) every row rescales O there,
    the rows of the second Q tile too (300 queries: two Q tiles)."""
    N, H, n = 740, 1, 300
    u = synth.normal((1, H, D), 81)
    q = (u + 0.3 * synth.normal((n, H, D), 82)).to(torch.bfloat16)
    kc = synth.normal((N, H, D), 83)
    kc[pos] = lift * u[0]
    kc = kc.to(torch.bfloat16)
    vc = synth.normal((N, H, D), 84, "bf16")
    out = torch.empty((n, H, D), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_active_attention(q.to(DEV), None, n, kc.to(DEV), vc.to(DEV), out)
    _no_device_error(hsa)
    _check_attention(out, oracle.attention(q, kc, vc), "bf16")


@pytest.mark.parametrize("trend", ["growing", "shrinking"])
def test_attention_score_trends(hsa, trend):
    """Key norms that grow (or shrink) along the sequence: with growing keys
    later tiles exceed the first tile's reference maximum by a wide margin
    (large probabilities, and the exact path once a row sum passes 2^32);
    with shrinking keys the first tile's reference dominates."""
    N, H, D, n = 3000, 2, 128, 500
    ramp = torch.linspace(0.2, 3.0, N) if trend == "growing" else torch.linspace(3.0, 0.2, N)
    q = synth.normal((n, H, D), 71, "bf16")
    kc = (synth.normal((N, H, D), 72) * ramp.view(N, 1, 1)).to(torch.bfloat16)
    vc = synth.normal((N, H, D), 73, "bf16")
    out = torch.empty((n, H, D), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_active_attention(q.to(DEV), None, n, kc.to(DEV), vc.to(DEV), out)
    _no_device_error(hsa)
    _check_attention(out, oracle.attention(q, kc, vc), "bf16")


def _sampled_rows(n_act, k, seed):
    """k random rows plus rows of the last Q block: its first 4 and last 12
    (its tail is ragged whenever n_act is not a multiple of 256)."""
    g = torch.Generator().manual_seed(seed)
    rows = set(torch.randperm(n_act, generator=g)[:k].tolist())
    last = (n_act - 1) // 256 * 256
    rows.update(range(last, min(last + 4, n_act)))
    rows.update(range(max(last, n_act - 12), n_act))
    return sorted(rows)


def _attention_full_size(hsa, name, it, n_rows=24, n_heads=2, seed=0):
    """Full-size layer, launch as the benchmark does; the oracle checks a
    sample of (row, head) pairs against all N keys, plus the last Q block."""
    w = synth.WORKLOADS[name]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    idx, _ = oracle.active_set(g, w.T, w.budgets, it)
    n = idx.numel()
    q = synth.normal((w.N, w.H, w.D), 201, w.dtype)
    kc = synth.normal((w.N, w.H, w.D), 202, w.dtype)
    vc = synth.normal((w.N, w.H, w.D), 203, w.dtype)
    q_d, kc_d, vc_d, idx_d = q.to(DEV), kc.to(DEV), vc.to(DEV), idx.to(DEV)
    outs = []
    # the benchmark's launch (with the split-tail workspace) and the plain one
    for ws in (_workspace(hsa, n, w.N, w.H, w.D, w.dtype), None):
        out = torch.empty((n, w.H, w.D), dtype=q.dtype, device=DEV)
        hsa.hsa_active_attention(q_d, idx_d, n, kc_d, vc_d, out, workspace=ws)
        _no_device_error(hsa)
        outs.append(out.cpu())
    del q_d, kc_d, vc_d
    rows = torch.tensor(_sampled_rows(n, n_rows, seed), dtype=torch.long)
    # The units split along the keys (with a workspace) are the last query
    # blocks of the last head: sample rows there too.
    lo = max(0, n - 16 * 256)
    g = torch.Generator().manual_seed(seed + 1)
    tail = torch.unique(torch.cat([lo + torch.randperm(n - lo, generator=g)[:16],
                                   torch.tensor(_sampled_rows(n, 0, seed))]))
    heads = torch.randperm(w.H, generator=torch.Generator().manual_seed(seed))[:n_heads]
    heads = sorted(set(heads.tolist()) | {w.H - 1})
    for h in heads:
        kh, vh = kc[:, h:h + 1].contiguous(), vc[:, h:h + 1].contiguous()
        qh = q[:, h:h + 1].contiguous()
        r = rows if h != w.H - 1 else torch.unique(torch.cat([rows, tail]))
        ref = oracle.attention(qh, kh, vh, q_idx=idx[r])
        for out in outs:
            _check_attention(out[r, h:h + 1], ref, w.dtype)


@pytest.mark.parametrize("it", [0, 2, 1])
def test_attention_wan13b_full_size(hsa, it):
    _attention_full_size(hsa, "wan13b", it)


def test_attention_wan14b_boxes_full_size(hsa):
    _attention_full_size(hsa, "wan14b_boxes", 1)


def test_attention_ltx_full_size(hsa):
    _attention_full_size(hsa, "ltx", 0, n_rows=64, n_heads=4)


def test_attention_wan14b_720p_full_size(hsa):
    _attention_full_size(hsa, "wan14b_720p", 1, n_rows=12, n_heads=1)


def test_dense_equivalence_all_active(hsa):
    """All tokens active: scatter of fresh K/V + active attention = dense
    attention of the fresh Q, K, V (both through libhsa; one oracle)."""
    N, H, D, T = 2000, 2, 128, 8
    budgets, counts = (8, 4), (500, 1500)
    g = oracle.partition(synth.lognormal_stat(N, 1.0, 1), T, budgets, counts)
    idx, _ = oracle.active_set(g, T, budgets, 0)
    assert idx.numel() == N
    q, kf, vf = (synth.normal((N, H, D), s, "bf16") for s in (11, 12, 13))
    kc = torch.zeros((N, H, D), dtype=torch.bfloat16, device=DEV)
    vc = torch.zeros_like(kc)
    hsa.hsa_kv_sync_scatter(kc, vc, kf.to(DEV), vf.to(DEV), idx.to(DEV), N)
    o_hsa = torch.empty((N, H, D), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_active_attention(q.to(DEV), idx.to(DEV), N, kc, vc, o_hsa)
    o_dense = torch.empty_like(o_hsa)
    hsa.hsa_active_attention(q.to(DEV), None, N, kf.to(DEV), vf.to(DEV), o_dense)
    assert torch.equal(o_hsa, o_dense)
    _check_attention(o_dense, oracle.attention(q, kf, vf), "bf16")


def test_attention_bad_query_index(hsa):
    N, H, D = 300, 1, 64
    q = synth.normal((N, H, D), 1, "bf16").to(DEV)
    kc = synth.normal((N, H, D), 2, "bf16").to(DEV)
    idx = torch.tensor([5, 300], dtype=torch.int32, device=DEV)
    out = torch.empty((2, H, D), dtype=torch.bfloat16, device=DEV)
    hsa.hsa_active_attention(q, idx, 2, kc, kc, out)
    assert hsa.hsa_get_device_error() == -6


def test_attention_rejects_unsupported(hsa):
    q = torch.zeros((10, 1, 96), dtype=torch.bfloat16, device=DEV)
    out = torch.zeros_like(q)
    with pytest.raises(hsa.HsaError) as e:
        hsa.hsa_active_attention(q, None, 10, q, q, out)
    assert e.value.status == -4


# ------------------------------------------------------------- cached Euler

def _euler_step_check(hsa, x, vh, vfr, pos, ds):
    x_d, vh_d = x.to(DEV), vh.to(DEV)
    hsa.hsa_cached_euler(x_d, vh_d, None if vfr is None else vfr.to(DEV),
                         None if pos is None else pos.to(DEV), ds)
    x64, vh64 = x.double(), vh.double()
    oracle.cached_euler_f64(x64, vh64, None if vfr is None else vfr.double(), pos, ds)
    oracle.cached_euler_f32(x, vh, vfr, pos, ds)
    assert torch.equal(x_d.cpu(), x) and torch.equal(vh_d.cpu(), vh)
    cond = x64.abs() + (vh64 * ds).abs() + 1e-30
    assert torch.all((x_d.cpu().double() - x64).abs() <= 1e-6 * cond)


@pytest.mark.parametrize("name", ["tiny_f32", "ltx", "wan14b_720p", "wan13b"])
def test_cached_euler_workloads(hsa, name):
    w = synth.WORKLOADS[name]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    sig = oracle.sigmas(w.T, w.shift)
    x = synth.normal((w.N, w.C), 301)
    vh = synth.normal((w.N, w.C), 302)
    for it in (0, 1, 2, w.T - 1):
        idx, pos = oracle.active_set(g, w.T, w.budgets, it)
        vfr = synth.normal((idx.numel(), w.C), 303 + it)
        _euler_step_check(hsa, x, vh, vfr, pos, float(sig[it + 1] - sig[it]))
    _euler_step_check(hsa, x, vh, None, None, float(sig[1] - sig[0]))
    _no_device_error(hsa)


@pytest.mark.parametrize("N,C", [(777, 12), (1000, 20), (5, 4), (33333, 8)])
def test_cached_euler_odd_widths(hsa, N, C):
    """C/4 not a power of two (division path), tiny N, ragged N."""
    g = torch.Generator().manual_seed(N)
    x = synth.normal((N, C), 1)
    vh = synth.normal((N, C), 2)
    idx = synth.uniform_subset(N, max(1, N // 3), 3)
    pos = torch.full((N,), -1, dtype=torch.int32)
    pos[idx.long()] = torch.arange(idx.numel(), dtype=torch.int32)
    vfr = synth.normal((idx.numel(), C), 4)
    _euler_step_check(hsa, x, vh, vfr, pos, -0.0625)
    _no_device_error(hsa)


def test_cached_euler_skip4_telescopes(hsa):
    """Tiny workload, skip length 4: four cached steps of the GPU equal the
    fp32 mirror bit for bit and one fp64 Euler step from sigma_i to
    sigma_{i+4} within the fp32 rounding of four updates."""
    w = synth.WORKLOADS["tiny_f32"]
    sig = oracle.sigmas(w.T)
    x = synth.normal((w.N, w.C), 1)
    v = synth.normal((w.N, w.C), 2)
    idx = synth.uniform_subset(w.N, w.n_active, 3)
    pos = torch.full((w.N,), -1, dtype=torch.int32)
    pos[idx.long()] = torch.arange(idx.numel(), dtype=torch.int32)
    vh = synth.normal((w.N, w.C), 4)
    vfr = v[idx.long()].contiguous()
    x_d, vh_d = x.to(DEV), vh.to(DEV)
    i0 = 8
    hsa.hsa_cached_euler(x_d, vh_d, vfr.to(DEV), pos.to(DEV), float(sig[i0 + 1] - sig[i0]))
    for i in range(i0 + 1, i0 + w.skip):
        hsa.hsa_cached_euler(x_d, vh_d, None, None, float(sig[i + 1] - sig[i]))
    vh_exp = vh.clone()
    vh_exp[idx.long()] = vfr
    one = x.double() + vh_exp.double() * float(sig[i0 + w.skip] - sig[i0])
    got = x_d.cpu().double()
    bound = 4 * 2 * 2.0 ** -24 * (x.double().abs() + vh_exp.double().abs() * 0.1)
    assert torch.all((got - one).abs() <= bound)
    x32, vh32 = x.clone(), vh.clone()
    oracle.cached_euler_f32(x32, vh32, vfr, pos, float(sig[i0 + 1] - sig[i0]))
    for i in range(i0 + 1, i0 + w.skip):
        oracle.cached_euler_f32(x32, vh32, None, None, float(sig[i + 1] - sig[i]))
    assert torch.equal(x_d.cpu(), x32)


def test_cached_euler_bad_pos(hsa):
    x = torch.zeros((10, 4), device=DEV)
    vh = torch.ones((10, 4), device=DEV)
    pos = torch.full((10,), -1, dtype=torch.int32, device=DEV)
    pos[3] = 2                                  # only 2 fresh rows exist
    hsa.hsa_cached_euler(x, vh, torch.ones((2, 4), device=DEV), pos, 0.5)
    assert hsa.hsa_get_device_error() == -6
    assert torch.all(x.cpu() == 0.5)


@pytest.mark.parametrize("bad", [-2, -5, -(2 ** 31)])
def test_cached_euler_negative_pos(hsa, bad):
    """Only -1 means 'no fresh row': any other negative pos is reported as an
    index error and that token keeps its cached velocity (plain and fused)."""
    x = torch.zeros((10, 4), device=DEV)
    vh = torch.ones((10, 4), device=DEV)
    vfr = torch.full((2, 4), 3.0, device=DEV)
    pos = torch.full((10,), -1, dtype=torch.int32, device=DEV)
    pos[1] = 0
    pos[4] = bad
    hsa.hsa_cached_euler(x, vh, vfr, pos, 0.5)
    assert hsa.hsa_get_device_error() == -6
    exp = torch.full((10, 4), 0.5)
    exp[1] = 1.5
    assert torch.equal(x.cpu(), exp)
    x.zero_()
    vh.fill_(1.0)
    stat = torch.zeros(10, device=DEV)
    hsa.hsa_cached_euler_l1rel(x, vh, vfr, pos, 0.5, stat, 1.0)
    assert hsa.hsa_get_device_error() == -6
    assert torch.equal(x.cpu(), exp)
    assert stat.cpu()[4].item() == 0.0


def test_check_indices(hsa):
    """Opt-in index check: a valid active set passes; a repeated id or one out
    of range is reported as HSA_ERR_INDEX (Sec. 2.2: groups are disjoint)."""
    N = 70001
    ws = torch.empty(hsa.hsa_check_indices_workspace_bytes(N), dtype=torch.uint8, device=DEV)
    idx = synth.uniform_subset(N, 30000, 5)
    d = idx.to(DEV)
    hsa.hsa_check_indices(d, idx.numel(), N, ws)
    assert hsa.hsa_get_device_error() == 0
    perm = torch.randperm(N, generator=torch.Generator().manual_seed(3)).to(torch.int32)
    hsa.hsa_check_indices(perm.to(DEV), N, N, ws)          # a permutation, any order
    assert hsa.hsa_get_device_error() == 0
    dup = idx.clone()
    dup[20000] = dup[123]                                   # one repeated token
    hsa.hsa_check_indices(dup.to(DEV), dup.numel(), N, ws)
    assert hsa.hsa_get_device_error() == -6
    hsa.hsa_check_indices(d, idx.numel(), N, ws)            # the bitmap is cleared per call
    assert hsa.hsa_get_device_error() == 0
    oob = idx.clone()
    oob[-1] = N
    hsa.hsa_check_indices(oob.to(DEV), oob.numel(), N, ws)
    assert hsa.hsa_get_device_error() == -6
    # the active set the library writes passes the check
    g = torch.randint(0, 3, (N,), generator=torch.Generator().manual_seed(4),
                      dtype=torch.int32).to(DEV)
    a_idx = torch.empty(N, dtype=torch.int32, device=DEV)
    hsa.hsa_partition_active(g, 40, (40, 20, 10), 2, a_idx, None)
    torch.cuda.synchronize()
    n = int((g.cpu() <= 1).sum())
    hsa.hsa_check_indices(a_idx, n, N, ws)
    assert hsa.hsa_get_device_error() == 0


# ------------------------------------------------------- whole schedule

def test_full_schedule_small(hsa):
    """Every iteration of a T=40, K=4 schedule on a small layer: partition,
    active set, gather, scatter, attention and cached Euler on the GPU track
    the oracle's run of the same loop (exact except attention)."""
    N, H, D, C, T = 700, 2, 64, 16, 40
    budgets, counts = (40, 20, 10, 5), (100, 150, 200, 250)
    stat = synth.lognormal_stat(N, 1.0, 11)
    sig = oracle.sigmas(T, 3.0)
    g_ref = oracle.partition(stat, T, budgets, counts)
    g = torch.empty(N, dtype=torch.int32, device=DEV)
    ws = torch.empty(hsa.hsa_partition_workspace_bytes(N), dtype=torch.uint8, device=DEV)
    hsa.hsa_partition(stat.to(DEV), T, budgets, counts, g, ws)
    kc, vc = synth.normal((N, H, D), 1, "bf16"), synth.normal((N, H, D), 2, "bf16")
    hid = synth.normal((N, H * D), 3, "bf16")
    x, vh = synth.normal((N, C), 4), torch.zeros((N, C))
    d = {k: t.to(DEV) for k, t in dict(kc=kc, vc=vc, hid=hid, x=x, vh=vh).items()}
    idx = torch.empty(N, dtype=torch.int32, device=DEV)
    pos = torch.empty(N, dtype=torch.int32, device=DEV)
    for it in range(T):
        idx_ref, pos_ref = oracle.active_set(g_ref, T, budgets, it, 80)
        n = hsa.hsa_active_count(budgets, counts, T, it, 80)
        hsa.hsa_partition_active(g, T, budgets, it, idx, pos, 80)
        h_act = torch.empty((n, H * D), dtype=torch.bfloat16, device=DEV)
        hsa.hsa_gather_active(d["hid"], idx, n, h_act)
        kf = synth.normal((n, H, D), 1000 + it, "bf16")
        vf = synth.normal((n, H, D), 2000 + it, "bf16")
        qf = synth.normal((n, H, D), 3000 + it, "bf16")
        hsa.hsa_kv_sync_scatter(d["kc"], d["vc"], kf.to(DEV), vf.to(DEV), idx, n)
        oracle.kv_scatter(kc, vc, kf, vf, idx_ref)
        o = torch.empty((n, H, D), dtype=torch.bfloat16, device=DEV)
        hsa.hsa_active_attention(qf.to(DEV), None, n, d["kc"], d["vc"], o)
        if it % 9 == 0:
            _check_attention(o, oracle.attention(qf, kc, vc), "bf16")
        vfr = synth.normal((n, C), 4000 + it)
        ds = float(sig[it + 1] - sig[it])
        hsa.hsa_cached_euler(d["x"], d["vh"], vfr.to(DEV), pos, ds)
        oracle.cached_euler_f32(x, vh, vfr, pos_ref, ds)
        assert torch.equal(h_act.cpu(), oracle.gather(hid, idx_ref))
    assert torch.equal(d["kc"].cpu(), kc) and torch.equal(d["vc"].cpu(), vc)
    assert torch.equal(d["x"].cpu(), x) and torch.equal(d["vh"].cpu(), vh)
    _no_device_error(hsa)
