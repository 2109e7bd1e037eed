"""Python front end of the CPU oracle (``hsa_oracle.c``).

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference legs may import this package.  The
product library never imports it, and it imports nothing from the product.

Arrays are host torch tensors (contiguous); results come back as new host
tensors.  Status codes are the plain ints documented in ``hsa_oracle.c``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hsa_oracle.c")
_LIB = os.path.join(_HERE, "libhsa_oracle.so")

OK, EINVAL, ENOTDIV, ECOUNTS, ENONFINITE, EINDEX = 0, -1, -2, -3, -5, -6

_DT = {torch.bfloat16: 0, torch.float32: 1, torch.float64: 2}


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain -O2, no fast-math, no FP contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call([
            "gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-ffp-contract=off",
            "-fno-fast-math", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        c_int, c_p, c_sz, c_d, c_f = (ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t,
                                      ctypes.c_double, ctypes.c_float)
        sig = {
            "orc_check_budgets": [c_int, c_p, c_p, c_int, c_int],
            "orc_partition": [c_p, c_int, c_int, c_p, c_p, c_int, c_p],
            "orc_margin": [c_int, c_int],
            "orc_is_active": [c_int, c_int, c_int, c_int],
            "orc_active_set": [c_p, c_int, c_int, c_p, c_int, c_int, c_int, c_p, c_p],
            "orc_active_count": [c_p, c_p, c_int, c_int, c_int, c_int],
            "orc_gather": [c_p, c_sz, c_int, c_p, c_int, c_p],
            "orc_kv_scatter": [c_p, c_p, c_p, c_p, c_p, c_int, c_int, c_sz],
            "orc_attention": [c_p, c_int, c_p, c_int, c_p, c_p, c_int, c_int, c_int, c_int, c_d, c_p],
            "orc_cached_euler_f64": [c_p, c_p, c_p, c_p, c_int, c_int, c_d],
            "orc_cached_euler_f32": [c_p, c_p, c_p, c_p, c_int, c_int, c_f],
            "orc_sigmas": [c_int, c_d, c_p],
            "orc_l1rel_accumulate": [c_p, c_p, c_p, c_int, c_int, c_d, c_p],
            "orc_uniform_stat": [c_int, c_p],
            "orc_reserve_frame": [c_p, c_int, c_int],
            "orc_reorder": [c_p, c_int, c_p, c_p, c_p],
            "orc_rope_table": [c_int, c_int, c_int, c_int, c_d, c_p],
            "orc_rope_rows": [c_p, c_p, c_int, c_int, c_int, c_p, c_int],
        }
        for name, args in sig.items():
            f = getattr(_lib, name)
            f.argtypes = args
            f.restype = c_int
    return _lib


def _ints(xs) -> torch.Tensor:
    return torch.tensor(list(xs), dtype=torch.int32)


def _ptr(t):
    return None if t is None else t.data_ptr()


class OracleError(RuntimeError):
    def __init__(self, status: int):
        super().__init__(f"oracle status {status}")
        self.status = status


def _check(st: int) -> int:
    if st < 0:
        raise OracleError(st)
    return st


def check_budgets(T, budgets, counts, N) -> int:
    b, c = _ints(budgets), (None if counts is None else _ints(counts))
    return lib().orc_check_budgets(T, b.data_ptr(), _ptr(c), len(budgets), N)


def partition(stat: torch.Tensor, T: int, budgets, counts) -> torch.Tensor:
    """group_of int32 [N] (group 0 = baseline); raises OracleError on bad input."""
    stat = stat.contiguous().to(torch.float32)
    N = stat.numel()
    out = torch.empty(N, dtype=torch.int32)
    b, c = _ints(budgets), _ints(counts)
    _check(lib().orc_partition(stat.data_ptr(), N, T, b.data_ptr(), c.data_ptr(),
                               len(budgets), out.data_ptr()))
    return out


def margin(T: int, window_pct: int) -> int:
    return _check(lib().orc_margin(T, window_pct))


def is_active(i: int, T: int, s: int, m: int) -> bool:
    return bool(lib().orc_is_active(i, T, s, m))


def active_set(group_of: torch.Tensor, T: int, budgets, iter_: int, window_pct: int = 100):
    """(idx int32 [|A_i|] ascending, pos int32 [N])."""
    g = group_of.contiguous().to(torch.int32)
    N = g.numel()
    idx = torch.empty(max(N, 1), dtype=torch.int32)
    pos = torch.empty(max(N, 1), dtype=torch.int32)
    b = _ints(budgets)
    n = _check(lib().orc_active_set(g.data_ptr(), N, T, b.data_ptr(), len(budgets),
                                    iter_, window_pct, idx.data_ptr(), pos.data_ptr()))
    return idx[:n].clone(), pos[:N].clone()


def active_count(budgets, counts, T: int, iter_: int, window_pct: int = 100) -> int:
    b, c = _ints(budgets), _ints(counts)
    return _check(lib().orc_active_count(b.data_ptr(), c.data_ptr(), len(budgets), T,
                                         iter_, window_pct))


def gather(src: torch.Tensor, idx: torch.Tensor) -> torch.Tensor:
    """dst = src[idx] row-wise (rows = first dimension)."""
    src = src.contiguous()
    idx = idx.contiguous().to(torch.int32)
    N = src.shape[0]
    row_bytes = src[0].numel() * src.element_size() if N else 0
    dst = torch.empty((idx.numel(),) + tuple(src.shape[1:]), dtype=src.dtype)
    _check(lib().orc_gather(src.data_ptr(), row_bytes, N, idx.data_ptr(), idx.numel(),
                            dst.data_ptr()))
    return dst


def kv_scatter(k_cache, v_cache, k_fresh, v_fresh, idx) -> None:
    """In place: k_cache[idx] = k_fresh, v_cache[idx] = v_fresh."""
    assert k_cache.is_contiguous() and v_cache.is_contiguous()
    k_fresh, v_fresh = k_fresh.contiguous(), v_fresh.contiguous()
    idx = idx.contiguous().to(torch.int32)
    N = k_cache.shape[0]
    row_bytes = k_cache[0].numel() * k_cache.element_size()
    _check(lib().orc_kv_scatter(k_cache.data_ptr(), v_cache.data_ptr(), k_fresh.data_ptr(),
                                v_fresh.data_ptr(), idx.data_ptr(), idx.numel(), N, row_bytes))


def attention(q, k_cache, v_cache, q_idx=None, scale: float = 0.0) -> torch.Tensor:
    """fp64 [n_q, H, D] attention of active queries against the full cache.

    q: [rows, H, D] (bf16/fp32/fp64); q_idx selects rows (None: all rows).
    k_cache, v_cache: [N, H, D] of one dtype.
    """
    q = q.contiguous()
    k_cache, v_cache = k_cache.contiguous(), v_cache.contiguous()
    assert k_cache.dtype == v_cache.dtype
    N, H, D = k_cache.shape
    if q_idx is not None:
        q_idx = q_idx.contiguous().to(torch.int32)
        n_q = q_idx.numel()
    else:
        n_q = q.shape[0]
    out = torch.empty((n_q, H, D), dtype=torch.float64)
    _check(lib().orc_attention(q.data_ptr(), _DT[q.dtype], _ptr(q_idx), n_q,
                               k_cache.data_ptr(), v_cache.data_ptr(), _DT[k_cache.dtype],
                               N, H, D, float(scale), out.data_ptr()))
    return out


def cached_euler_f64(x, vhat, v_fresh, pos, dsigma: float) -> None:
    """In place on fp64 x, vhat [N, C]."""
    assert x.dtype == torch.float64 and vhat.dtype == torch.float64
    assert x.is_contiguous() and vhat.is_contiguous()
    N, C = x.shape
    vf = None if v_fresh is None else v_fresh.contiguous().to(torch.float64)
    p = None if pos is None else pos.contiguous().to(torch.int32)
    _check(lib().orc_cached_euler_f64(x.data_ptr(), vhat.data_ptr(), _ptr(vf), _ptr(p),
                                      N, C, float(dsigma)))


def cached_euler_f32(x, vhat, v_fresh, pos, dsigma: float) -> None:
    """In place on fp32 x, vhat [N, C]; dsigma is rounded to fp32 by the call."""
    assert x.dtype == torch.float32 and vhat.dtype == torch.float32
    assert x.is_contiguous() and vhat.is_contiguous()
    N, C = x.shape
    vf = None if v_fresh is None else v_fresh.contiguous().to(torch.float32)
    p = None if pos is None else pos.contiguous().to(torch.int32)
    _check(lib().orc_cached_euler_f32(x.data_ptr(), vhat.data_ptr(), _ptr(vf), _ptr(p),
                                      N, C, float(dsigma)))


def sigmas(T: int, shift: float = 1.0) -> torch.Tensor:
    """fp64 [T+1] noise levels sigma_0 = 1 > ... > sigma_T = 0."""
    out = torch.empty(T + 1, dtype=torch.float64)
    _check(lib().orc_sigmas(T, float(shift), out.data_ptr()))
    return out


def l1rel_accumulate(vhat_old, v_fresh, pos, weight: float, stat) -> None:
    """In place on fp64 stat [N]: App. B Eq. 7 for the refreshed tokens."""
    assert stat.dtype == torch.float64 and stat.is_contiguous()
    vo = vhat_old.contiguous().to(torch.float64)
    vf = v_fresh.contiguous().to(torch.float64)
    p = pos.contiguous().to(torch.int32)
    N, C = vo.shape
    _check(lib().orc_l1rel_accumulate(vo.data_ptr(), vf.data_ptr(), p.data_ptr(), N, C,
                                      float(weight), stat.data_ptr()))


def uniform_stat(N: int) -> torch.Tensor:
    out = torch.empty(max(N, 1), dtype=torch.float32)
    _check(lib().orc_uniform_stat(N, out.data_ptr()))
    return out[:N].clone()


def reserve_frame(stat: torch.Tensor, frame_tokens: int) -> torch.Tensor:
    out = stat.contiguous().to(torch.float32).clone()
    _check(lib().orc_reserve_frame(out.data_ptr(), out.numel(), frame_tokens))
    return out


def reorder(group_of: torch.Tensor):
    """(order, where, group_new, M) of the Sec. 2.5 token reordering."""
    g = group_of.contiguous().to(torch.int32)
    N = g.numel()
    order, where, gn = (torch.empty(max(N, 1), dtype=torch.int32) for _ in range(3))
    M = _check(lib().orc_reorder(g.data_ptr(), N, order.data_ptr(), where.data_ptr(),
                                 gn.data_ptr()))
    return order[:N].clone(), where[:N].clone(), gn[:N].clone(), M


def rope_table(grid, D: int, theta: float = 10000.0) -> torch.Tensor:
    """fp32 [N, D/2, 2] (cos, sin) table of a (F, Hh, Ww) token grid."""
    F, Hh, Ww = grid
    out = torch.empty((F * Hh * Ww, D // 2, 2), dtype=torch.float32)
    _check(lib().orc_rope_table(F, Hh, Ww, D, float(theta), out.data_ptr()))
    return out


def rope_rows(x: torch.Tensor, idx: torch.Tensor, table: torch.Tensor) -> torch.Tensor:
    """New bf16 tensor: rows of x [n, H, D] rotated by table[idx[j]]."""
    assert x.dtype == torch.bfloat16
    out = x.contiguous().clone()
    n, H, D = out.shape
    idx = idx.contiguous().to(torch.int32)
    table = table.contiguous()
    _check(lib().orc_rope_rows(out.data_ptr(), idx.data_ptr(), n, H, D, table.data_ptr(),
                               table.shape[0]))
    return out
