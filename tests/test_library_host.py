"""CPU-only checks of libhsa: the shared library loads, exports every entry
point include/hsa.h declares, and its host-side helpers (budget checks, window
margin, |A_i|, noise schedule) agree with the oracle.  No kernel is launched."""
import ctypes
import os
import re

import pytest
import torch

import oracle
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def hsa():
    from paper_2605_06892_gb300 import build as b
    b.build()
    import paper_2605_06892_gb300 as m
    m.lib()
    return m


def _declared_functions():
    names = []
    for h in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not h.endswith(".h"):
            continue
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_\s\*]*?\b(hsa_[a-z0-9_]+)\s*\(",
                            src, flags=re.M)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(hsa):
    names = _declared_functions()
    assert len(names) >= 14, names
    lib = ctypes.CDLL(hsa.library_path)
    for n in names:
        assert hasattr(lib, n), n
    # the binding offers each entry point under the same name
    for n in names:
        assert hasattr(hsa, n), n


def test_status_strings(hsa):
    assert hsa.hsa_status_string(0) == "ok"
    for code in range(-9, 0):
        assert hsa.hsa_status_string(code) != "unknown status"
    assert hsa.hsa_version() == 1


def test_budget_checks_match_oracle(hsa):
    cases = [(40, (40, 20, 10), (1, 2, 3), 6), (40, (40, 15), (1, 1), 2),
             (40, (20, 10), (1, 1), 2), (40, (10, 20), (1, 1), 2), (40, (40, 10), (1, 1), 3),
             (40, (40, 10), (-1, 3), 2), (40, (40, 0), (1, 1), 2), (1, (1,), (5,), 5),
             (40, (40, 40, 5), (1, 1, 1), 3)]
    for T, b, c, N in cases:
        assert hsa.hsa_check_budgets(T, b, c, N) == oracle.check_budgets(T, b, c, N)


def test_window_margin_and_active_count_match_oracle(hsa):
    for T in (1, 8, 20, 40, 50):
        for k in range(0, 101, 5):
            assert hsa.hsa_window_margin(T, k) == oracle.margin(T, k)
    for w in synth.WORKLOADS.values():
        counts = w.counts or synth.stat_for(w)[1]
        for k in (100, 80, 50):
            for i in range(w.T):
                assert (hsa.hsa_active_count(w.budgets, counts, w.T, i, k)
                        == oracle.active_count(w.budgets, counts, w.T, i, k))


def test_sigma_schedule_matches_oracle(hsa):
    for T in (1, 10, 40):
        for shift in (1.0, 3.0, 5.0):
            a = hsa.hsa_sigma_schedule(T, shift)
            b = oracle.sigmas(T, shift).tolist()
            assert all(abs(x - y) <= 1e-15 for x, y in zip(a, b))
            assert a[0] == 1.0 and a[-1] == 0.0


def test_workspace_size_is_monotone(hsa):
    assert hsa.hsa_partition_workspace_bytes(0) == 0
    sizes = [hsa.hsa_partition_workspace_bytes(n) for n in (1, 4096, 4097, 75600, 10 ** 6)]
    assert sizes == sorted(sizes) and sizes[0] > 0
    assert all(s % 256 == 0 for s in sizes)


def test_rope_table_matches_oracle(hsa):
    for grid, D in (((3, 4, 5), 128), ((2, 3, 3), 64), ((1, 1, 7), 8)):
        a = hsa.hsa_rope_table(grid, D)
        b = oracle.rope_table(grid, D)
        assert torch.allclose(a, b, rtol=0, atol=1e-7)


def test_launch_counter_needs_no_gpu(hsa):
    """The launch counter is host-side: readable without a GPU, and host-only
    calls and calls that fail their argument checks add nothing."""
    c0 = hsa.hsa_launch_count()
    assert isinstance(c0, int) and c0 >= 0
    hsa.hsa_check_budgets(40, (40, 20), (1, 1), 2)
    hsa.hsa_window_margin(40, 80)
    ints = ctypes.c_int * 2
    # 15 does not divide T = 40: rejected on the host, nothing launched
    st = hsa.lib().hsa_partition(None, 4, 40, ints(40, 15), ints(2, 2), 2, None, None, 0, None)
    assert st < 0
    assert hsa.hsa_launch_count() == c0


def test_index_check_host_side(hsa):
    """hsa_check_indices: one bit per token of workspace, in whole 256-byte
    blocks; argument and workspace errors are reported on the host before any
    launch (so no GPU is needed to see them)."""
    ws = hsa.lib().hsa_check_indices_workspace_bytes
    assert ws(0) == 0
    for N in (1, 31, 32, 2048, 2049, 75600, 10 ** 6):
        b = ws(N)
        assert b % 256 == 0 and b * 8 >= N and b - 256 < (N + 7) // 8 + 16
    c0 = hsa.hsa_launch_count()
    lib = hsa.lib()
    assert lib.hsa_check_indices(None, 0, 100, None, 0, None) == 0          # nothing to check
    assert lib.hsa_check_indices(None, -1, 100, None, 0, None) == -1        # n < 0
    assert lib.hsa_check_indices(None, 5, 100, None, 0, None) == -1        # no idx
    fake = ctypes.c_void_p(4096)                                           # never dereferenced
    assert lib.hsa_check_indices(fake, 5, 100, None, 0, None) == -9        # no workspace
    assert lib.hsa_check_indices(fake, 5, 10 ** 6, fake, 256, None) == -9  # too small
    assert lib.hsa_check_indices(fake, 5, 100, ctypes.c_void_p(4100), 256, None) == -9  # misaligned
    assert hsa.hsa_launch_count() == c0


def test_static_partition_limit_agrees(hsa):
    """The binding's copy of HSA_PARTITION_STATIC_MAX_TOKENS is the header's, and
    the limit lies above the sizes that the partition serves without scratch
    (the cluster select ends at 360448 tokens), so the fixed array is used."""
    src = open(os.path.join(ROOT, "include", "hsa.h")).read()
    m = re.search(r"#define\s+HSA_PARTITION_STATIC_MAX_TOKENS\s+(\d+)", src)
    assert m and int(m.group(1)) == hsa.HSA_PARTITION_STATIC_MAX_TOKENS
    assert hsa.HSA_PARTITION_STATIC_MAX_TOKENS > 360448
    ints = ctypes.c_int * 1
    st = hsa.lib().hsa_partition_static(None, hsa.HSA_PARTITION_STATIC_MAX_TOKENS + 1, 8,
                                        ints(8), ints(hsa.HSA_PARTITION_STATIC_MAX_TOKENS + 1),
                                        1, None, None)
    assert st == -4                                                        # before any launch
