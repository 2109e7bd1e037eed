"""Seeded synthetic inputs for the HSA hot path.

This module is shared by the CPU oracle's tests and by the CUDA path's tests and
benchmark.  It holds no arithmetic of the method itself: it only draws random
tensors (torch's seeded CPU generator), converts them to storage dtypes, and
describes the five workload shapes.  Every tensor it returns lives in host
memory; callers copy what they need to the device.

Workload recipe (the paper's Wan-2.1 / LTX-2 video DiTs and VBench prompts are
not available, so these tensors stand in for them with the paper's shapes):

* Token count N follows the patchify rule of Sec. 2.1 ("Video DiT inference"):
  N = F * (H_l/2) * (W_l/2); each workload lists its (F, H_l/2, W_l/2) grid and
  tokens are numbered row-major over (f, h, w).
* Q, K, V and the cached K/V are i.i.d. N(0, 1), rounded to the storage dtype.
* The per-token velocity statistic that drives the ranking (App. B, Eq. 7,
  dynamic selection "D") is drawn lognormal, or from seeded spatial boxes for
  the spatially clustered workload.
* Latent rows x and velocities are i.i.d. N(0, 1) fp32.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch

__all__ = [
    "Workload", "WORKLOADS", "normal", "normal_blocks", "lognormal_stat", "box_stat",
    "uniform_subset", "seed_for",
]


@dataclass(frozen=True)
class Workload:
    """One synthetic HSA layer workload.

    budgets/counts: step budget s_k and group size |G_k| per group, baseline
    group first (budgets[0] == T), as in Sec. 2.2 Eq. 3.  ``counts`` is None
    when the group sizes come out of the statistic generator (box workload).
    iters: the global iterations i at which one layer step is measured.
    """
    name: str
    cid: int
    grid: tuple
    H: int
    D: int
    dtype: str                 # "bf16" or "f32": Q/K/V storage and compute input
    T: int
    budgets: tuple
    counts: tuple | None
    stat: str                  # "lognormal", "boxes" or "random"
    stat_sigma: float
    C: int                     # latent channels per token (x, v rows)
    schedule: str              # "linear" or "shifted"
    shift: float
    window_pct: int            # central caching window k in percent (100 = none)
    iters: tuple
    n_active: int | None = None   # explicit |A| (tiny workload only)
    skip: int = 1                 # cached-Euler skip length checked by the tests
    extra: dict = field(default_factory=dict)

    @property
    def N(self) -> int:
        f, h, w = self.grid
        return f * h * w


WORKLOADS = {
    # N = 4*16*16 = 1024; fp32; |A| = 256 drawn uniformly without replacement.
    "tiny_f32": Workload(
        name="tiny_f32", cid=1, grid=(4, 16, 16), H=4, D=64, dtype="f32", T=40,
        budgets=(40, 10), counts=(256, 768), stat="random", stat_sigma=1.0, C=16,
        schedule="linear", shift=1.0, window_pct=100, iters=(0, 1), n_active=256,
        skip=4),
    # Wan-2.1-1.3B shaped layer: 21x30x52 grid, 12 heads x 128.  HSA-75A split
    # 25%@40 + 25%@20 + 50%@10 (App. C preset table) gives active fractions
    # 100% (i = 0 mod 4), 50% (i = 2 mod 4) and 25% (odd i).
    "wan13b": Workload(
        name="wan13b", cid=2, grid=(21, 30, 52), H=12, D=128, dtype="bf16", T=40,
        budgets=(40, 20, 10), counts=(8190, 8190, 16380), stat="lognormal",
        stat_sigma=1.0, C=16, schedule="linear", shift=1.0, window_pct=100,
        iters=(0, 2, 1)),
    # Wan-2.1-14B shaped layer, spatially clustered active sets: seeded boxes
    # on the (f, h, w) grid get the full budget, the rest 20 or 10 steps.
    "wan14b_boxes": Workload(
        name="wan14b_boxes", cid=3, grid=(21, 30, 52), H=40, D=128, dtype="bf16",
        T=40, budgets=(40, 20, 10), counts=None, stat="boxes", stat_sigma=1.0,
        C=16, schedule="linear", shift=1.0, window_pct=100, iters=(1, 2)),
    # LTX-style compressed latent: 16x16x24 grid, 32 heads x 64, four equal
    # groups at 40/20/10/5 steps, 128-channel latent, shift-3 schedule.
    "ltx": Workload(
        name="ltx", cid=4, grid=(16, 16, 24), H=32, D=64, dtype="bf16", T=40,
        budgets=(40, 20, 10, 5), counts=(1536, 1536, 1536, 1536),
        stat="lognormal", stat_sigma=0.5, C=128, schedule="shifted", shift=3.0,
        window_pct=100, iters=(0, 4, 2, 1)),
    # Full 40-iteration schedule on a 720p-like Wan-14B layer: 21x45x80 grid.
    "wan14b_720p": Workload(
        name="wan14b_720p", cid=5, grid=(21, 45, 80), H=40, D=128, dtype="bf16",
        T=40, budgets=(40, 20, 10, 5), counts=(18900, 18900, 18900, 18900),
        stat="lognormal", stat_sigma=1.0, C=16, schedule="linear", shift=1.0,
        window_pct=100, iters=tuple(range(40))),
}


def seed_for(cid: int, rep: int, tensor_id: int) -> int:
    """Seed of tensor ``tensor_id`` for workload ``cid``, repetition ``rep``."""
    return (cid * 1000 + rep) * 64 + tensor_id


def _gen(seed: int) -> torch.Generator:
    return torch.Generator(device="cpu").manual_seed(int(seed))


def normal(shape, seed: int, dtype: str = "f32") -> torch.Tensor:
    """i.i.d. N(0,1) host tensor, drawn in fp32 and rounded to ``dtype``
    ("f32" or "bf16", round-to-nearest-even)."""
    x = torch.randn(tuple(shape), generator=_gen(seed), dtype=torch.float32)
    if dtype == "bf16":
        return x.to(torch.bfloat16)
    if dtype == "f32":
        return x
    raise ValueError(dtype)


def normal_blocks(shape, seed: int, dtype: str = "f32", workers: int | None = None,
                  block: int = 4096) -> torch.Tensor:
    """i.i.d. N(0,1) host tensor for multi-GB shapes: the first dimension is cut
    into blocks of ``block`` rows and block b is drawn by its own seeded
    generator (seed * 1000003 + b), in fp32, rounded to ``dtype``.  The blocks
    are drawn on ``workers`` threads; the values depend only on the seed and the
    block size, not on the number of threads.  Same distribution as ``normal``
    (other values)."""
    import concurrent.futures as cf
    import os
    shape = tuple(shape)
    tdt = {"bf16": torch.bfloat16, "f32": torch.float32}[dtype]
    out = torch.empty(shape, dtype=tdt)
    n = shape[0]
    n_blocks = (n + block - 1) // block

    def fill(b):
        r0, r1 = b * block, min(n, (b + 1) * block)
        g = _gen(seed * 1000003 + b)
        out[r0:r1] = torch.randn((r1 - r0,) + shape[1:], generator=g, dtype=torch.float32)

    workers = workers or max(1, min(32, len(os.sched_getaffinity(0))))
    with cf.ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(fill, range(n_blocks)))
    return out


def lognormal_stat(N: int, sigma: float, seed: int) -> torch.Tensor:
    """Per-token statistic exp(sigma * z), z ~ N(0,1), formed in fp64 and
    rounded once to fp32 (the statistic's storage type)."""
    z = torch.randn(N, generator=_gen(seed), dtype=torch.float64)
    return torch.exp(sigma * z).to(torch.float32)


def box_stat(grid, seed: int, coverage: float = 0.25, sigma: float = 1.0):
    """Spatially clustered statistic on an (F, Hh, Ww) token grid.

    Seeded axis-aligned boxes (extent uniform in [3,8] x [5,15] x [8,26],
    clipped to the grid) are added until at least ``coverage`` of the tokens
    lie inside one.  In-box tokens get 1e3 + lognormal, the rest lognormal, so
    a ranking puts every in-box token above every other one.
    Returns (stat fp32 [N], number of in-box tokens).
    """
    F, Hh, Ww = grid
    g = _gen(seed)
    inside = torch.zeros((F, Hh, Ww), dtype=torch.bool)
    lo_hi = ((3, 8), (5, 15), (8, 26))
    while inside.float().mean().item() < coverage:
        ext = [int(torch.randint(lo, hi + 1, (1,), generator=g)) for lo, hi in lo_hi]
        ext = [min(e, d) for e, d in zip(ext, grid)]
        org = [int(torch.randint(0, d - e + 1, (1,), generator=g)) for e, d in zip(ext, grid)]
        inside[org[0]:org[0] + ext[0], org[1]:org[1] + ext[1], org[2]:org[2] + ext[2]] = True
    inside = inside.reshape(-1)
    z = torch.randn(inside.numel(), generator=g, dtype=torch.float64)
    stat = torch.exp(sigma * z) + 1e3 * inside.to(torch.float64)
    return stat.to(torch.float32), int(inside.sum().item())


def uniform_subset(N: int, n: int, seed: int) -> torch.Tensor:
    """``n`` distinct token indices drawn uniformly from [0, N), ascending, int32."""
    perm = torch.randperm(N, generator=_gen(seed))
    return perm[:n].sort().values.to(torch.int32)


def counts_for(w: Workload, n_box: int | None = None) -> tuple:
    """Group sizes of a workload; the box workload derives them from the
    number of in-box tokens: |G_1| = n_box, |G_2| = floor(N/4), |G_3| = rest."""
    if w.counts is not None:
        return tuple(w.counts)
    assert n_box is not None
    c2 = w.N // 4
    return (n_box, c2, w.N - n_box - c2)


def stat_for(w: Workload, rep: int = 0):
    """(stat fp32 [N], counts) for a workload."""
    seed = seed_for(w.cid, rep, 0)
    if w.stat == "boxes":
        stat, n_box = box_stat(w.grid, seed, 0.25, w.stat_sigma)
        return stat, counts_for(w, n_box)
    if w.stat == "random":
        # Random allocation (App. B, "R"): a uniform random statistic.
        stat = torch.rand(w.N, generator=_gen(seed), dtype=torch.float32)
        return stat, counts_for(w)
    return lognormal_stat(w.N, w.stat_sigma, seed), counts_for(w)
