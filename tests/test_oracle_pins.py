"""Pins of the CPU oracle against what the paper and mathematics fix.

None of these tests compares the oracle with a retyped copy of its own
formula: each one checks a printed value of the paper, a closed form, an
invariant the paper states, a library routine the definition reduces to, or a
brute-force enumeration on tiny inputs.
"""
import itertools
import math
import os

import pytest
import torch

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------------ presets

def _presets():
    rows = []
    with open(os.path.join(GOLDEN, "presets.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if not line:
                continue
            name, runtime, alloc, window, strategy = line.split()
            groups = [tuple(int(v) for v in g.split("@")) for g in alloc.split("+")]
            rows.append((name, float(runtime), groups, int(window), strategy))
    return rows


@pytest.mark.parametrize("preset", _presets(), ids=lambda p: p[0])
def test_preset_runtimes_match_paper(preset):
    """App. C prints each preset's runtime as a percentage of FM (T=40).
    Counting active token-steps with the modular rule (Sec. 2.2) and the
    caching-window margin (Sec. 2.5) must reproduce those labels.  HSA-25 has
    no 40-step group, so its baseline budget 20 is its T (s_1 = T, Sec. 2.2)."""
    name, runtime, groups, window, _ = preset
    budgets = [s for _, s in groups]
    counts = [pct for pct, _ in groups]          # 100 tokens in total
    T = budgets[0]
    assert sum(counts) == 100
    token_steps = sum(oracle.active_count(budgets, counts, T, i, window) for i in range(T))
    pct = 100.0 * token_steps / (100 * 40)
    assert abs(pct - runtime) <= 0.5, (name, pct)


def test_window_margin_integer_reading():
    """Sec. 2.5: m = floor((1-k) T / 2).  k = 50% and 80% at T = 40 give
    m = 10 and 4; in floating point (1-0.8)*40/2 falls just below 4."""
    assert oracle.margin(40, 50) == 10
    assert oracle.margin(40, 80) == 4
    assert math.floor((1 - 0.8) * 40 / 2) == 3      # why the reading is integer
    assert oracle.margin(40, 100) == 0
    assert oracle.margin(40, 0) == 20
    assert oracle.margin(20, 80) == 2


# -------------------------------------------------------- modular activity

@pytest.mark.parametrize("T", [1, 6, 12, 20, 40])
def test_budget_is_number_of_active_iterations(T):
    """Without a window, a group with budget s is active in exactly s of the
    T iterations (the meaning of 'step budget', Sec. 2.2), and the gap between
    its active iterations is T/s, the maximum KV lag stated in Sec. 2.3."""
    for s in [d for d in range(1, T + 1) if T % d == 0]:
        active = [i for i in range(T) if oracle.is_active(i, T, s, 0)]
        assert len(active) == s
        assert active[0] == 0
        gaps = [b - a for a, b in zip(active, active[1:])] + [T - active[-1]]
        assert all(g == T // s for g in gaps)


def test_mean_active_fraction_is_effective_steps():
    """Eq. 4: s_bar = sum_k |G_k|/N s_k.  Averaged over the T iterations,
    |A_i|/N equals s_bar/T, so the speedup T/s_bar of Eq. 4 is the ratio of
    token-steps."""
    for w in synth.WORKLOADS.values():
        if w.counts is None:
            continue
        sbar = sum(c / w.N * s for c, s in zip(w.counts, w.budgets))
        tot = sum(oracle.active_count(w.budgets, w.counts, w.T, i, 100) for i in range(w.T))
        assert abs(tot / (w.N * w.T) - sbar / w.T) < 1e-12


def test_window_margins_are_full_passes():
    """Sec. 2.5: the first m and last m iterations treat every token as active."""
    budgets, counts, T = (40, 20, 10, 5), (3, 4, 5, 6), 40
    for k in (50, 80):
        m = oracle.margin(T, k)
        for i in list(range(m)) + list(range(T - m, T)):
            assert oracle.active_count(budgets, counts, T, i, k) == sum(counts)
        assert oracle.active_count(budgets, counts, T, m + 1, k) < sum(counts)


def test_active_set_is_union_of_active_groups():
    """A_i = union of the active groups (Fig. 1 caption), listed ascending,
    with pos the inverse map; on the Wan-1.3B split the active fractions are
    100/50/25% at i = 0, 2, 1 (the three measured iterations)."""
    w = synth.WORKLOADS["wan13b"]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    for i, frac in ((0, 1.0), (2, 0.5), (1, 0.25)):
        idx, pos = oracle.active_set(g, w.T, w.budgets, i)
        assert idx.numel() == round(frac * w.N)
        assert torch.all(idx[1:] > idx[:-1])
        act = torch.tensor([oracle.is_active(i, w.T, w.budgets[int(k)], 0) for k in g])
        assert torch.equal(torch.nonzero(act).flatten().to(torch.int32), idx)
        assert torch.equal(pos[idx.long()], torch.arange(idx.numel(), dtype=torch.int32))
        assert int((pos >= 0).sum()) == idx.numel()
        assert oracle.active_count(w.budgets, counts, w.T, i) == idx.numel()


# ----------------------------------------------------------------- partition

def _brute_force_partition(stat, counts):
    """Every assignment with the given group sizes such that each token of a
    lower-budget group ranks below each token of a higher-budget group in the
    (value, index) order.  App. B: small change -> low budget, sizes fixed."""
    N, K = len(stat), len(counts)
    sols = []
    labels = [k for k in range(K) for _ in range(counts[k])]
    for perm in set(itertools.permutations(labels)):
        ok = True
        for a in range(N):
            for b in range(N):
                # group index larger = smaller budget = must rank lower
                if perm[a] > perm[b] and not ((stat[a], a) < (stat[b], b)):
                    ok = False
                    break
            if not ok:
                break
        if ok:
            sols.append(list(perm))
    return sols


@pytest.mark.parametrize("seed", range(12))
def test_partition_brute_force(seed):
    g = torch.Generator().manual_seed(seed)
    N = int(torch.randint(1, 8, (1,), generator=g))
    # few distinct values so that ties and -0/+0 occur
    pool = torch.tensor([-0.0, 0.0, 1.5, -2.0, 3.0])
    stat = pool[torch.randint(0, 5, (N,), generator=g)]
    K = int(torch.randint(1, 4, (1,), generator=g))
    cut = sorted(int(v) for v in torch.randint(0, N + 1, (K - 1,), generator=g))
    bounds = [0] + cut + [N]
    counts = [bounds[k + 1] - bounds[k] for k in range(K)]
    budgets = [12, 6, 3][:K]
    got = oracle.partition(stat, 12, budgets, counts).tolist()
    sols = _brute_force_partition([float(v) if v != 0 else 0.0 for v in stat.tolist()], counts)
    assert len(sols) == 1
    assert got == sols[0]


def test_partition_distinct_values_threshold_property():
    """With distinct statistics, max(stat over G_{k+1}) < min(stat over G_k)."""
    w = synth.WORKLOADS["ltx"]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    for k in range(len(counts)):
        assert int((g == k).sum()) == counts[k]
    for k in range(len(counts) - 1):
        assert stat[g == k + 1].max() < stat[g == k].min()


def test_partition_box_workload_puts_boxes_in_baseline():
    w = synth.WORKLOADS["wan14b_boxes"]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    assert counts[0] >= w.N // 4
    assert torch.equal(g == 0, stat >= 1e3)


def test_partition_rejects_bad_budgets():
    stat = torch.rand(10)
    with pytest.raises(oracle.OracleError) as e:
        oracle.partition(stat, 40, [40, 15], [5, 5])     # 15 does not divide 40
    assert e.value.status == oracle.ENOTDIV
    with pytest.raises(oracle.OracleError) as e:
        oracle.partition(stat, 40, [20, 10], [5, 5])     # s_1 != T
    assert e.value.status == oracle.EINVAL
    with pytest.raises(oracle.OracleError) as e:
        oracle.partition(stat, 40, [10, 20], [5, 5])     # not non-increasing
    assert e.value.status == oracle.EINVAL
    with pytest.raises(oracle.OracleError) as e:
        oracle.partition(stat, 40, [40, 10], [5, 4])     # sizes do not cover S
    assert e.value.status == oracle.ECOUNTS
    bad = stat.clone()
    bad[3] = float("nan")
    with pytest.raises(oracle.OracleError) as e:
        oracle.partition(bad, 40, [40, 10], [5, 5])
    assert e.value.status == oracle.ENONFINITE
    bad[3] = float("inf")
    with pytest.raises(oracle.OracleError) as e:
        oracle.partition(bad, 40, [40, 10], [5, 5])
    assert e.value.status == oracle.ENONFINITE


def test_partition_empty_and_single_group():
    assert oracle.partition(torch.empty(0), 8, [8], [0]).numel() == 0
    g = oracle.partition(torch.rand(17), 8, [8], [17])
    assert torch.all(g == 0)


# ------------------------------------------------------------ gather/scatter

def test_gather_scatter_round_trip_and_canaries():
    """Sec. 2.3 step 2: cached entries of skipped tokens remain unchanged;
    the written rows are the fresh ones, readable back by a gather."""
    N, H, D = 50, 3, 8
    kc = torch.full((N, H, D), 7.0)
    vc = torch.full((N, H, D), -7.0)
    idx = synth.uniform_subset(N, 13, 5)
    kf, vf = synth.normal((13, H, D), 1), synth.normal((13, H, D), 2)
    oracle.kv_scatter(kc, vc, kf, vf, idx)
    assert torch.equal(oracle.gather(kc, idx), kf)
    assert torch.equal(oracle.gather(vc, idx), vf)
    skipped = torch.ones(N, dtype=torch.bool)
    skipped[idx.long()] = False
    assert torch.all(kc[skipped] == 7.0) and torch.all(vc[skipped] == -7.0)
    # identity gather is a copy; torch's index_select agrees on bytes
    src = synth.normal((N, 24), 3, "bf16")
    assert torch.equal(oracle.gather(src, torch.arange(N, dtype=torch.int32)), src)
    assert torch.equal(oracle.gather(src, idx), src.index_select(0, idx.long()))


def test_scatter_rejects_duplicates_and_range():
    kc = torch.zeros(5, 4)
    with pytest.raises(oracle.OracleError):
        oracle.kv_scatter(kc, kc.clone(), torch.ones(2, 4), torch.ones(2, 4),
                          torch.tensor([1, 1], dtype=torch.int32))
    with pytest.raises(oracle.OracleError):
        oracle.kv_scatter(kc, kc.clone(), torch.ones(1, 4), torch.ones(1, 4),
                          torch.tensor([5], dtype=torch.int32))
    with pytest.raises(oracle.OracleError):
        oracle.gather(kc, torch.tensor([-1], dtype=torch.int32))


# ----------------------------------------------------------------- attention

def _torch_attention(q, k, v, scale):
    """softmax(Q K^T * scale) V per head with torch's fp64 CPU routines."""
    q, k, v = (t.to(torch.float64).transpose(0, 1) for t in (q, k, v))   # [H, *, D]
    p = torch.softmax(torch.matmul(q, k.transpose(1, 2)) * scale, dim=-1)
    return torch.matmul(p, v).transpose(0, 1)


@pytest.mark.parametrize("dtype,N,H,D", [("f32", 64, 2, 64), ("bf16", 97, 3, 128),
                                         ("bf16", 1, 1, 64), ("f32", 130, 1, 16)])
def test_attention_matches_library_softmax(dtype, N, H, D):
    q = synth.normal((N, H, D), 11, dtype)
    k = synth.normal((N, H, D), 12, dtype)
    v = synth.normal((N, H, D), 13, dtype)
    idx = synth.uniform_subset(N, max(1, N // 3), 14)
    got = oracle.attention(q, k, v, q_idx=idx)
    ref = _torch_attention(q[idx.long()], k, v, 1.0 / math.sqrt(D))
    assert torch.allclose(got, ref, rtol=1e-12, atol=1e-12)
    # compact queries give the same rows
    assert torch.equal(oracle.attention(q[idx.long()].contiguous(), k, v), got)


def test_attention_closed_forms():
    N, H, D = 33, 2, 16
    q = synth.normal((5, H, D), 21)
    v = synth.normal((N, H, D), 22)
    # identical keys: uniform weights, output is the mean of V
    k = synth.normal((1, H, D), 23).expand(N, H, D).contiguous()
    assert torch.allclose(oracle.attention(q, k, v), v.double().mean(0).expand(5, H, D),
                          atol=1e-12)
    # constant values: output is that constant whatever the keys
    kk = synth.normal((N, H, D), 24)
    vc = torch.full((N, H, D), 0.375)
    assert torch.allclose(oracle.attention(q, kk, vc), torch.full((5, H, D), 0.375,
                                                                  dtype=torch.float64),
                          atol=1e-14)
    # one key: its value
    assert torch.allclose(oracle.attention(q, kk[:1], v[:1]),
                          v[:1].double().expand(5, H, D), atol=0)
    # a key aligned with the query with a huge margin takes all the weight
    k3 = torch.zeros((N, 1, D))
    q3 = torch.zeros((1, 1, D))
    q3[0, 0, 0] = 100.0
    k3[7, 0, 0] = 100.0
    out = oracle.attention(q3, k3, v[:, :1].contiguous())
    assert torch.allclose(out[0, 0], v[7, 0].double(), atol=1e-12)


def test_attention_key_permutation_invariance():
    N, H, D = 40, 2, 32
    q, k, v = (synth.normal((N, H, D), s) for s in (31, 32, 33))
    perm = torch.randperm(N, generator=torch.Generator().manual_seed(3))
    a = oracle.attention(q, k, v)
    b = oracle.attention(q, k[perm].contiguous(), v[perm].contiguous())
    assert torch.allclose(a, b, atol=1e-13)


def test_dense_equivalence_when_all_active():
    """With every token active (i = 0, or all budgets T), scatter + attention
    equals dense attention of the fresh Q, K, V (stated aim of Sec. 2.3)."""
    N, H, D, T = 48, 2, 16, 8
    stat = torch.rand(N, generator=torch.Generator().manual_seed(4))
    g = oracle.partition(stat, T, [8, 4, 2], [10, 14, 24])
    idx, _ = oracle.active_set(g, T, [8, 4, 2], 0)
    assert idx.numel() == N
    kc, vc = torch.zeros(N, H, D), torch.zeros(N, H, D)
    q, kf, vf = (synth.normal((N, H, D), s) for s in (41, 42, 43))
    oracle.kv_scatter(kc, vc, kf, vf, idx)
    assert torch.allclose(oracle.attention(q, kc, vc, q_idx=idx),
                          _torch_attention(q, kf, vf, 1 / math.sqrt(D)), atol=1e-12)


# --------------------------------------------------------------- schedules

def test_sigma_schedules():
    s = oracle.sigmas(40)
    assert s[0] == 1.0 and s[-1] == 0.0
    assert torch.allclose(s[:-1] - s[1:], torch.full((40,), 1 / 40, dtype=torch.float64),
                          atol=1e-15)
    sh = oracle.sigmas(40, 3.0)
    assert sh[0] == 1.0 and sh[-1] == 0.0 and torch.all(sh[1:] < sh[:-1])
    assert abs(float(sh[20]) - 0.75) < 1e-15          # t = 1/2: 3*0.5/(1+2*0.5)
    assert torch.equal(oracle.sigmas(40, 1.0), s)


# ------------------------------------------------------------ cached Euler

def _hsa_latent_loop(x0, v_of_step, group_of, budgets, T, sig, window=100, f32=False):
    """Run T iterations of active-set -> refresh -> cached Euler on the oracle."""
    x = x0.clone()
    vhat = torch.zeros_like(x)
    for i in range(T):
        idx, pos = oracle.active_set(group_of, T, budgets, i, window)
        vf = v_of_step(i)[idx.long()].contiguous()
        ds = float(sig[i + 1] - sig[i])
        if f32:
            oracle.cached_euler_f32(x, vhat, vf.float(), pos, ds)
        else:
            oracle.cached_euler_f64(x, vhat, vf.double(), pos, ds)
    return x


def test_euler_exact_on_flow_matching_path():
    """Eq. 1 / Eq. 2: on the linear path x_sigma = x0 + sigma*eps the velocity
    is eps for every sigma, so any mix of fresh and cached velocities (Eq. 6)
    lands exactly on x0 at sigma_T = 0, on either schedule."""
    N, C, T = 64, 16, 40
    x0 = synth.normal((N, C), 51).double()
    eps = synth.normal((N, C), 52).double()
    stat = torch.rand(N, generator=torch.Generator().manual_seed(5))
    g = oracle.partition(stat, T, [40, 20, 10, 5], [16, 16, 16, 16])
    for shift in (1.0, 3.0):
        sig = oracle.sigmas(T, shift)
        x = _hsa_latent_loop(x0 + sig[0] * eps, lambda i: eps, g, [40, 20, 10, 5], T, sig)
        assert torch.allclose(x, x0, atol=1e-13)


def test_euler_telescopes_over_skipped_steps():
    """Sec. 2.4: k cached steps with a held velocity equal one Euler step
    from sigma_i to sigma_{i+k}."""
    N, C = 1024, 16
    sig = oracle.sigmas(40)
    x = synth.normal((N, C), 61).double()
    v = synth.normal((N, C), 62).double()
    for i0, k in ((0, 4), (5, 4), (36, 4), (3, 1)):
        xs, vh = x.clone(), torch.zeros_like(x)
        all_pos = torch.arange(N, dtype=torch.int32)
        oracle.cached_euler_f64(xs, vh, v, all_pos, float(sig[i0 + 1] - sig[i0]))
        for i in range(i0 + 1, i0 + k):
            oracle.cached_euler_f64(xs, vh, None, None, float(sig[i + 1] - sig[i]))
        one = x + v * float(sig[i0 + k] - sig[i0])
        assert torch.allclose(xs, one, rtol=1e-12, atol=1e-13)


def test_euler_constant_velocity_full_linear_schedule():
    """Constant v over sigma 1 -> 0: x_T = x_0 - v."""
    N, C = 100, 8
    sig = oracle.sigmas(40)
    x0, v = synth.normal((N, C), 71).double(), synth.normal((N, C), 72).double()
    g = oracle.partition(torch.rand(N, generator=torch.Generator().manual_seed(6)), 40,
                         [40, 10], [30, 70])
    x = _hsa_latent_loop(x0, lambda i: v, g, [40, 10], 40, sig)
    assert torch.allclose(x, x0 - v, atol=1e-13)


def test_velocity_cache_refresh_semantics():
    """Sec. 2.4: v^ holds the last velocity of each token; active tokens take
    the fresh one, skipped tokens keep theirs, and every token moves."""
    N, C = 20, 4
    x = torch.zeros(N, C, dtype=torch.float64)
    vh = torch.arange(N * C, dtype=torch.float64).reshape(N, C)
    pos = torch.full((N,), -1, dtype=torch.int32)
    act = torch.tensor([2, 3, 11], dtype=torch.int32)
    pos[act.long()] = torch.arange(3, dtype=torch.int32)
    vf = -torch.ones(3, C, dtype=torch.float64)
    before = vh.clone()
    oracle.cached_euler_f64(x, vh, vf, pos, 0.5)
    assert torch.equal(vh[act.long()], vf)
    keep = pos < 0
    assert torch.equal(vh[keep], before[keep])
    assert torch.equal(x, 0.5 * vh)


def test_euler_f32_mirror_within_rounding_bound():
    """The fp32 mirror (one FMA per element and step, dsigma rounded once)
    stays within the forward error bound of T roundings of the fp64 result:
    |x32 - x64| <= 2*T*u*(|x0| + sum |v dsigma|), u = 2^-24."""
    N, C, T = 256, 16, 40
    sig = oracle.sigmas(T, 3.0)
    x0 = synth.normal((N, C), 81)
    vs = [synth.normal((N, C), 100 + i) for i in range(T)]
    g = oracle.partition(torch.rand(N, generator=torch.Generator().manual_seed(7)), T,
                         [40, 20, 10, 5], [64, 64, 64, 64])
    x32 = _hsa_latent_loop(x0, lambda i: vs[i], g, [40, 20, 10, 5], T, sig, f32=True)
    # fp64 run with the fp32-rounded step sizes, so only the update roundings differ
    sig32 = [0.0]
    for i in range(T):
        sig32.append(sig32[-1] + float(torch.tensor(float(sig[i + 1] - sig[i]),
                                                    dtype=torch.float32)))
    x64 = _hsa_latent_loop(x0.double(), lambda i: vs[i].double(), g, [40, 20, 10, 5], T,
                           torch.tensor(sig32, dtype=torch.float64))
    bound = 2 * T * 2.0 ** -24 * (x0.double().abs() + sum(v.double().abs() for v in vs) * 0.1)
    assert torch.all((x32.double() - x64).abs() <= bound)
    assert not torch.equal(x32.double(), x64)     # the mirror really is fp32


# ------------------------------------------------- velocity statistic (D)

def test_l1rel_closed_forms():
    """App. B Eq. 7 on cases with known values: a velocity that doubles has
    relative change 1/2, one that flips sign 2, one that stays 0; the measure
    is scale invariant; skipped tokens are not touched."""
    N, C = 6, 16
    vo = synth.normal((N, C), 1).double()
    vf = torch.stack([2 * vo[0], -vo[1], vo[2], 3.0 * vo[3], 7.5 * vo[4], vo[5]])
    pos = torch.tensor([0, 1, 2, 3, 4, -1], dtype=torch.int32)
    stat = torch.zeros(N, dtype=torch.float64)
    oracle.l1rel_accumulate(vo, vf[:5].contiguous(), pos, 1.0, stat)
    assert abs(stat[0] - 0.5) < 1e-15 and abs(stat[1] - 2.0) < 1e-15 and stat[2] == 0.0
    assert abs(stat[3] - 2.0 / 3.0) < 1e-15 and abs(stat[4] - 6.5 / 7.5) < 1e-15
    assert stat[5] == 0.0
    s2 = torch.zeros(N, dtype=torch.float64)
    oracle.l1rel_accumulate(4.0 * vo, 4.0 * vf[:5].contiguous(), pos, 1.0, s2)
    assert torch.allclose(s2, stat, rtol=1e-14, atol=0)


def test_l1rel_running_mean_and_zero_denominator():
    N, C, steps = 40, 8, 9
    g = torch.Generator().manual_seed(3)
    vs = [torch.randn(N, C, generator=g, dtype=torch.float64) for _ in range(steps + 1)]
    pos = torch.arange(N, dtype=torch.int32)
    stat = torch.zeros(N, dtype=torch.float64)
    for i in range(1, steps + 1):
        oracle.l1rel_accumulate(vs[i - 1], vs[i], pos, 1.0 / steps, stat)
    # the mean of the per-step relative changes, token by token
    direct = sum(((vs[i] - vs[i - 1]).abs().sum(1) / vs[i].abs().sum(1))
                 for i in range(1, steps + 1)) / steps
    assert torch.allclose(stat, direct, rtol=1e-13)
    z = torch.zeros(2, C, dtype=torch.float64)
    s0 = torch.zeros(2, dtype=torch.float64)
    one = torch.zeros(2, C, dtype=torch.float64)
    one[1, 0] = 1.0
    oracle.l1rel_accumulate(one, z, torch.tensor([0, 1], dtype=torch.int32), 1.0, s0)
    assert s0[0] == 0.0 and s0[1] == 3.4028234663852886e38


# ---------------------------------------------------- allocation strategies

@pytest.mark.parametrize("name", ["wan13b", "ltx", "wan14b_720p"])
def test_uniform_allocation_three_gaps(name):
    """U: each group's members are spaced by at most three distinct gaps
    (three-distance theorem) whose mean is N/|G_k|, and every group reaches
    both ends of the sequence."""
    w = synth.WORKLOADS[name]
    stat = oracle.uniform_stat(w.N)
    # the statistic is a permutation-free set of distinct values here
    assert torch.unique(stat).numel() == w.N
    g = oracle.partition(stat, w.T, w.budgets, w.counts)
    for k, c in enumerate(w.counts):
        members = torch.nonzero(g == k).flatten()
        assert members.numel() == c
        gaps = torch.unique(members[1:] - members[:-1])
        assert gaps.numel() <= 3, gaps
        assert members[0] < 2 * w.N / c and members[-1] > w.N - 2 * w.N / c
        assert abs(float((members[1:] - members[:-1]).double().mean()) - w.N / c) < 0.01 * w.N / c + 1


def test_uniform_stat_closed_form():
    s = oracle.uniform_stat(5)
    phi = (5 ** 0.5 - 1) / 2
    for n in range(5):
        assert s[n] == math.floor(((n + 1) * phi % 1.0) * 2 ** 24) or \
            abs(float(s[n]) - ((n + 1) * phi % 1.0) * 2 ** 24) <= 1.0


def test_first_frame_reservation():
    """F: with |G_1| >= frame size, every token of frame 0 is in the baseline
    group; the rest are ranked by the (random) statistic."""
    w = synth.WORKLOADS["wan13b"]
    frame = w.grid[1] * w.grid[2]
    stat = torch.rand(w.N, generator=torch.Generator().manual_seed(9))
    g = oracle.partition(oracle.reserve_frame(stat, frame), w.T, w.budgets, w.counts)
    assert torch.all(g[:frame] == 0)
    rest = oracle.partition(stat[frame:].contiguous(), w.T, w.budgets,
                            (w.counts[0] - frame,) + tuple(w.counts[1:]))
    assert torch.equal(g[frame:], rest)


# --------------------------------------------------------- token reordering

def test_reorder_is_stable_partition_with_inverse():
    w = synth.WORKLOADS["ltx"]
    stat, counts = synth.stat_for(w)
    g = oracle.partition(stat, w.T, w.budgets, counts)
    order, where, gn, M = oracle.reorder(g)
    N = w.N
    assert M == N - counts[0]
    assert torch.equal(torch.sort(order).values, torch.arange(N, dtype=torch.int32))
    assert torch.equal(where[order.long()], torch.arange(N, dtype=torch.int32))
    assert torch.all(gn[:M] != 0) and torch.all(gn[M:] == 0)
    assert torch.equal(gn, g[order.long()])
    assert torch.all(order[1:M] > order[:M - 1]) and torch.all(order[M + 1:] > order[M:-1])


def test_reordered_cache_gives_the_same_attention():
    """Sec. 2.5: the baseline group is active at every iteration, so a cache
    over the non-baseline prefix plus the fresh baseline K/V holds exactly the
    keys of the full cache.  Over a T = 8 schedule, attention outputs with the
    reordered, prefix-only cache equal (permuted back) those with the full
    cache."""
    N, H, D, T = 90, 2, 16, 8
    budgets, counts = (8, 4, 2), (20, 30, 40)
    g = oracle.partition(torch.rand(N, generator=torch.Generator().manual_seed(3)), T,
                         budgets, counts)
    order, where, gn, M = oracle.reorder(g)
    kc_full = synth.normal((N, H, D), 1)
    vc_full = synth.normal((N, H, D), 2)
    kc_pre = kc_full[order[:M].long()].contiguous()
    vc_pre = vc_full[order[:M].long()].contiguous()
    for it in range(T):
        kf = synth.normal((N, H, D), 100 + it)        # fresh K/V of every token
        vf = synth.normal((N, H, D), 200 + it)
        q = synth.normal((N, H, D), 300 + it)
        idx, _ = oracle.active_set(g, T, budgets, it)
        oracle.kv_scatter(kc_full, vc_full, kf[idx.long()].contiguous(),
                          vf[idx.long()].contiguous(), idx)
        ref = oracle.attention(q, kc_full, vc_full, q_idx=idx)
        idx_new, _ = oracle.active_set(gn, T, budgets, it)
        nb = int((idx_new < M).sum())
        assert torch.equal(idx_new[nb:], torch.arange(M, N, dtype=torch.int32))
        old_of_new = order[idx_new.long()].long()
        oracle.kv_scatter(kc_pre, vc_pre, kf[old_of_new[:nb]].contiguous(),
                          vf[old_of_new[:nb]].contiguous(), idx_new[:nb].contiguous())
        kb, vb = kf[order[M:].long()], vf[order[M:].long()]   # fresh baseline K/V
        got = oracle.attention(q[old_of_new].contiguous(), torch.cat([kc_pre, kb]).contiguous(),
                               torch.cat([vc_pre, vb]).contiguous())
        # rows of A_i in new order vs old order: same tokens
        assert torch.equal(torch.sort(old_of_new).values.to(torch.int32), idx)
        perm = torch.argsort(old_of_new)
        assert torch.allclose(got[perm], ref, atol=1e-12)


# ------------------------------------------------------------------- RoPE

def test_rope_table_bands_and_standard_frequencies():
    """Each band is standard RoPE along its axis: the first pair of every band
    turns by the axis position in radians, pair i by pos * theta^(-i/p); a
    token at the origin is not rotated."""
    grid, D = (3, 4, 5), 128
    tab = oracle.rope_table(grid, D).double()
    P, ph = D // 2, D // 6
    pt = P - 2 * ph
    assert (pt, ph) == (22, 21)
    assert torch.all(tab[0, :, 0] == 1.0) and torch.all(tab[0, :, 1] == 0.0)
    n = (2 * 4 + 3) * 5 + 1                     # f = 2, h = 3, w = 1
    for i, pos, p, bi in ((0, 2, pt, 0), (pt, 3, ph, 0), (pt + ph, 1, ph, 0),
                          (5, 2, pt, 5), (pt + 7, 3, ph, 7), (P - 1, 1, ph, ph - 1)):
        ang = pos * 10000.0 ** (-bi / p)
        assert abs(tab[n, i, 0] - math.cos(ang)) < 1e-7
        assert abs(tab[n, i, 1] - math.sin(ang)) < 1e-7


def test_rope_rotation_invariants():
    """Rotation keeps each pair's norm, and the dot product of two rotated
    vectors depends only on their position difference (relative encoding)."""
    grid, D = (4, 4, 4), 64
    tab = oracle.rope_table(grid, D)
    x = synth.normal((2, 1, D), 3, "bf16")
    pos = lambda f, h, w: (f * 4 + h) * 4 + w  # noqa: E731
    rot = lambda v, n: oracle.rope_rows(v, torch.tensor([n], dtype=torch.int32), tab)  # noqa: E731
    a, b = x[:1], x[1:]
    ra = rot(a, pos(1, 2, 0)).double()
    assert torch.allclose(ra.view(-1, 2).norm(dim=1), a.double().view(-1, 2).norm(dim=1),
                          rtol=1e-2)
    d1 = (rot(a, pos(1, 2, 0)).double() * rot(b, pos(2, 3, 1)).double()).sum()
    d2 = (rot(a, pos(2, 0, 2)).double() * rot(b, pos(3, 1, 3)).double()).sum()
    assert abs(float(d1 - d2)) < 0.15
    # the identity row leaves the vector unchanged
    assert torch.equal(rot(a, 0), a)


def test_rope_rotation_direction_is_complex_multiplication():
    """Fixes the rotation convention, which the invariants above leave open
    (norms and relative dot products hold for either sign): pair (x0, x1) of
    token n becomes (x0 + i x1) * exp(i * angle), the angle written out here
    from the band layout, in complex128 (torch), then rounded to bf16."""
    grid, D, H = (3, 5, 7), 64, 2
    N = grid[0] * grid[1] * grid[2]
    tab = oracle.rope_table(grid, D)
    P, ph = D // 2, D // 6
    pt = P - 2 * ph
    x = synth.normal((N, H, D), 21, "bf16")
    idx = torch.arange(N, dtype=torch.int32)
    got = oracle.rope_rows(x, idx, tab).double().view(N, H, P, 2)
    n = torch.arange(N, dtype=torch.float64)
    f = torch.div(n, grid[1] * grid[2], rounding_mode="floor")
    hh = torch.div(n, grid[2], rounding_mode="floor") % grid[1]
    ww = n % grid[2]
    ang = torch.empty((N, P), dtype=torch.float64)
    for i in range(P):
        if i < pt:
            ang[:, i] = f * 10000.0 ** (-i / pt)
        elif i < pt + ph:
            ang[:, i] = hh * 10000.0 ** (-(i - pt) / ph)
        else:
            ang[:, i] = ww * 10000.0 ** (-(i - pt - ph) / ph)
    xc = x.double().view(N, H, P, 2)
    z = torch.complex(xc[..., 0], xc[..., 1]) * torch.exp(1j * ang)[:, None, :]
    exp = torch.stack([z.real, z.imag], dim=-1)
    # bf16 rounding of each output (half an ulp, 2^-9 relative) plus the fp32
    # table and arithmetic; the opposite rotation misses by 2|x| |sin(angle)|
    tol = 2.0 ** -8 * exp.abs() + 1e-6
    assert torch.all((got - exp).abs() <= tol)
    wrong = torch.complex(xc[..., 0], xc[..., 1]) * torch.exp(-1j * ang)[:, None, :]
    wrong = torch.stack([wrong.real, wrong.imag], dim=-1)
    assert ((got - wrong).abs() > tol).float().mean() > 0.5
