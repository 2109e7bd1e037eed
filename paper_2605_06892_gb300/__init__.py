"""Python binding of libhsa, the GB300 hot path of Heterogeneous Step Allocation.

Argument marshalling only: each function below has the name of a C entry
point of include/hsa.h, turns torch tensors into raw pointers and sizes, calls
the C function through ctypes on the current torch CUDA stream (or the stream
given), and raises HsaError on a negative status.  Every step runs in the
library's CUDA kernels; there is no Python or CPU fallback, and importing this
package fails loudly when libhsa.so has not been built.

Device tensors must be contiguous and live on the current CUDA device.
"""
from __future__ import annotations

import ctypes
import os

import torch

__all__ = [
    "HsaError", "lib", "library_path", "HSA_BF16", "HSA_F32",
    "hsa_status_string", "hsa_version", "hsa_check_budgets", "hsa_window_margin",
    "hsa_active_count", "hsa_sigma_schedule", "hsa_partition_workspace_bytes",
    "hsa_partition", "hsa_partition_static", "hsa_uniform_stat", "hsa_reserve_first_frame",
    "hsa_reorder_tokens", "hsa_partition_active", "hsa_gather_active",
    "hsa_kv_sync_scatter", "hsa_check_indices", "hsa_check_indices_workspace_bytes",
    "hsa_rope_table", "hsa_rope_rows", "hsa_kv_sync_scatter_rope",
    "hsa_active_attention", "hsa_active_attention_prefix",
    "hsa_active_attention_workspace_bytes",
    "hsa_cached_euler", "hsa_cached_euler_l1rel",
    "hsa_get_device_error", "hsa_launch_count", "hsa_test_inject_attention_stall",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_HERE, "libhsa.so")

HSA_BF16, HSA_F32 = 0, 1
HSA_PARTITION_STATIC_MAX_TOKENS = 524288
STATUS = {0: "HSA_OK", -1: "HSA_ERR_INVALID_ARG", -2: "HSA_ERR_NOT_DIVISOR",
          -3: "HSA_ERR_BAD_COUNTS", -4: "HSA_ERR_UNSUPPORTED", -5: "HSA_ERR_NONFINITE",
          -6: "HSA_ERR_INDEX", -7: "HSA_ERR_TIMEOUT", -8: "HSA_ERR_CUDA",
          -9: "HSA_ERR_WORKSPACE"}


class HsaError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)} ({status})")


_c_int, _c_p, _c_sz, _c_f, _c_d = (ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t,
                                   ctypes.c_float, ctypes.c_double)
_SIGS = {
    "hsa_status_string": ([_c_int], ctypes.c_char_p),
    "hsa_version": ([], _c_int),
    "hsa_check_budgets": ([_c_int, _c_p, _c_p, _c_int, _c_int], _c_int),
    "hsa_window_margin": ([_c_int, _c_int], _c_int),
    "hsa_active_count": ([_c_p, _c_p, _c_int, _c_int, _c_int, _c_int], _c_int),
    "hsa_sigma_schedule": ([_c_int, _c_d, _c_p], _c_int),
    "hsa_partition_workspace_bytes": ([_c_int], _c_sz),
    "hsa_partition": ([_c_p, _c_int, _c_int, _c_p, _c_p, _c_int, _c_p, _c_p, _c_sz, _c_p],
                      _c_int),
    "hsa_partition_static": ([_c_p, _c_int, _c_int, _c_p, _c_p, _c_int, _c_p, _c_p], _c_int),
    "hsa_uniform_stat": ([_c_p, _c_int, _c_p], _c_int),
    "hsa_reserve_first_frame": ([_c_p, _c_int, _c_int, _c_p], _c_int),
    "hsa_partition_active": ([_c_p, _c_int, _c_int, _c_p, _c_int, _c_int, _c_int, _c_p, _c_p,
                              _c_p], _c_int),
    "hsa_gather_active": ([_c_p, _c_sz, _c_int, _c_p, _c_int, _c_p, _c_p], _c_int),
    "hsa_kv_sync_scatter": ([_c_p, _c_p, _c_p, _c_p, _c_p, _c_int, _c_int, _c_int, _c_int,
                             _c_int, _c_p], _c_int),
    "hsa_active_attention": ([_c_p, _c_p, _c_int, _c_p, _c_p, _c_int, _c_int, _c_int, _c_f,
                              _c_p, _c_int, _c_p, _c_sz, _c_p], _c_int),
    "hsa_active_attention_prefix": ([_c_p, _c_p, _c_int, _c_p, _c_p, _c_int, _c_p, _c_p, _c_int,
                                     _c_int, _c_int, _c_f, _c_p, _c_int, _c_p, _c_sz, _c_p],
                                    _c_int),
    "hsa_check_indices_workspace_bytes": ([_c_int], _c_sz),
    "hsa_check_indices": ([_c_p, _c_int, _c_int, _c_p, _c_sz, _c_p], _c_int),
    "hsa_rope_table": ([_c_int, _c_int, _c_int, _c_int, _c_d, _c_p], _c_int),
    "hsa_rope_rows": ([_c_p, _c_p, _c_int, _c_int, _c_int, _c_p, _c_int, _c_p], _c_int),
    "hsa_kv_sync_scatter_rope": ([_c_p, _c_p, _c_p, _c_p, _c_p, _c_int, _c_int, _c_int, _c_int,
                                  _c_p, _c_p], _c_int),
    "hsa_reorder_tokens": ([_c_p, _c_int, _c_int, _c_p, _c_p, _c_p, _c_p], _c_int),
    "hsa_active_attention_workspace_bytes": ([_c_int, _c_int, _c_int, _c_int, _c_int], _c_sz),
    "hsa_cached_euler": ([_c_p, _c_p, _c_p, _c_p, _c_int, _c_int, _c_int, _c_f, _c_p], _c_int),
    "hsa_cached_euler_l1rel": ([_c_p, _c_p, _c_p, _c_p, _c_int, _c_int, _c_int, _c_f, _c_p,
                                _c_f, _c_p], _c_int),
    "hsa_get_device_error": ([_c_p], _c_int),
    "hsa_launch_count": ([], ctypes.c_ulonglong),
    "hsa_test_inject_attention_stall": ([_c_int], _c_int),
}

_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libhsa.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(library_path):
            raise ImportError(
                f"libhsa.so not found at {library_path}; build it with "
                "`python -m paper_2605_06892_gb300.build` (or __graft_entry__.build())")
        handle = ctypes.CDLL(library_path)
        for name, (args, res) in _SIGS.items():
            f = getattr(handle, name)
            f.argtypes = args
            f.restype = res
        _lib = handle
    return _lib


# ------------------------------------------------------------- marshalling

def _p(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    assert t.is_contiguous(), "tensors passed to libhsa must be contiguous"
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _host_ints(xs) -> ctypes.Array:
    xs = list(xs)
    return (ctypes.c_int * max(1, len(xs)))(*xs)


def _check(st: int, where: str) -> int:
    if st < 0:
        raise HsaError(st, where)
    return st


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return HSA_BF16
    if t.dtype == torch.float32:
        return HSA_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


# ---------------------------------------------------------- host helpers

def hsa_status_string(status: int) -> str:
    return lib().hsa_status_string(status).decode()


def hsa_version() -> int:
    return lib().hsa_version()


def hsa_check_budgets(T: int, budgets, counts, N: int) -> int:
    c = None if counts is None else _host_ints(counts)
    return lib().hsa_check_budgets(T, _host_ints(budgets), c, len(budgets), N)


def hsa_window_margin(T: int, window_pct: int) -> int:
    return _check(lib().hsa_window_margin(T, window_pct), "hsa_window_margin")


def hsa_active_count(budgets, counts, T: int, iter_: int, window_pct: int = 100) -> int:
    return _check(lib().hsa_active_count(_host_ints(budgets), _host_ints(counts), len(budgets),
                                         T, iter_, window_pct), "hsa_active_count")


def hsa_sigma_schedule(T: int, shift: float = 1.0) -> list:
    buf = (ctypes.c_double * (T + 1))()
    _check(lib().hsa_sigma_schedule(T, float(shift), buf), "hsa_sigma_schedule")
    return list(buf)


# ----------------------------------------------------------- device calls

def hsa_partition_workspace_bytes(N: int) -> int:
    return lib().hsa_partition_workspace_bytes(N)


def hsa_partition(stat, T: int, budgets, counts, group_of, workspace, stream=None) -> None:
    """group_of[N] (int32, device) <- group of each token; workspace: uint8 device
    tensor of at least hsa_partition_workspace_bytes(N) bytes."""
    N = stat.numel()
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().hsa_partition(_p(stat), N, T, _host_ints(budgets), _host_ints(counts),
                               len(budgets), _p(group_of), _p(workspace), ws_bytes,
                               _stream(stream)), "hsa_partition")


def hsa_partition_static(stat, T: int, budgets, counts, group_of, stream=None) -> None:
    """hsa_partition with the library's own fixed scratch instead of a caller
    workspace (N <= HSA_PARTITION_STATIC_MAX_TOKENS); calls must not overlap
    on the GPU."""
    _check(lib().hsa_partition_static(_p(stat), stat.numel(), T, _host_ints(budgets),
                                      _host_ints(counts), len(budgets), _p(group_of),
                                      _stream(stream)), "hsa_partition_static")


def hsa_uniform_stat(stat, stream=None) -> None:
    """stat[n] <- uniform-allocation statistic (App. B, U)."""
    _check(lib().hsa_uniform_stat(_p(stat), stat.numel(), _stream(stream)), "hsa_uniform_stat")


def hsa_reserve_first_frame(stat, frame_tokens: int, stream=None) -> None:
    """stat[:frame_tokens] <- FLT_MAX (App. B, F)."""
    _check(lib().hsa_reserve_first_frame(_p(stat), stat.numel(), frame_tokens,
                                         _stream(stream)), "hsa_reserve_first_frame")


def hsa_partition_active(group_of, T: int, budgets, iter_: int, idx, pos=None,
                         window_pct: int = 100, stream=None) -> None:
    _check(lib().hsa_partition_active(_p(group_of), group_of.numel(), T, _host_ints(budgets),
                                      len(budgets), iter_, window_pct, _p(idx), _p(pos),
                                      _stream(stream)), "hsa_partition_active")


def hsa_gather_active(src, idx, n_active: int, dst, stream=None) -> None:
    """dst[:n_active] = src[idx[:n_active]] (rows = first dimension)."""
    N = src.shape[0]
    row_bytes = (src.numel() // max(N, 1)) * src.element_size()
    _check(lib().hsa_gather_active(_p(src), row_bytes, N, _p(idx), n_active, _p(dst),
                                   _stream(stream)), "hsa_gather_active")


def hsa_kv_sync_scatter(k_cache, v_cache, k_fresh, v_fresh, idx, n_active: int,
                        stream=None) -> None:
    N, H, D = k_cache.shape
    _check(lib().hsa_kv_sync_scatter(_p(k_cache), _p(v_cache), _p(k_fresh), _p(v_fresh),
                                     _p(idx), n_active, N, H, D, _dtype_code(k_cache),
                                     _stream(stream)), "hsa_kv_sync_scatter")


def hsa_check_indices_workspace_bytes(N: int) -> int:
    return lib().hsa_check_indices_workspace_bytes(N)


def hsa_check_indices(idx, n: int, N: int, workspace, stream=None) -> None:
    """Opt-in check of idx[:n]: HSA_ERR_INDEX (via hsa_get_device_error) when an
    entry is outside [0, N) or repeated; workspace: uint8 device tensor of at
    least hsa_check_indices_workspace_bytes(N) bytes."""
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().hsa_check_indices(_p(idx), n, N, _p(workspace), ws_bytes, _stream(stream)),
           "hsa_check_indices")


def hsa_rope_table(grid, D: int, theta: float = 10000.0) -> torch.Tensor:
    """Host fp32 [N, D/2, 2] (cos, sin) table of a (F, Hh, Ww) token grid."""
    F, Hh, Ww = grid
    out = torch.empty((F * Hh * Ww, D // 2, 2), dtype=torch.float32)
    _check(lib().hsa_rope_table(F, Hh, Ww, D, float(theta), out.data_ptr()), "hsa_rope_table")
    return out


def hsa_rope_rows(x, idx, n: int, table, stream=None) -> None:
    _, H, D = x.shape
    _check(lib().hsa_rope_rows(_p(x), _p(idx), n, H, D, _p(table), table.shape[0],
                               _stream(stream)), "hsa_rope_rows")


def hsa_kv_sync_scatter_rope(k_cache, v_cache, k_fresh, v_fresh, idx, n_active: int, table,
                             stream=None) -> None:
    N, H, D = k_cache.shape
    _check(lib().hsa_kv_sync_scatter_rope(_p(k_cache), _p(v_cache), _p(k_fresh), _p(v_fresh),
                                          _p(idx), n_active, N, H, D, _p(table),
                                          _stream(stream)), "hsa_kv_sync_scatter_rope")


def hsa_active_attention_prefix(q, q_idx, n_active: int, k_cache, v_cache, k_base, v_base, out,
                                scale: float = 0.0, workspace=None, stream=None) -> None:
    """Attention against the M cached rows followed by the B baseline rows."""
    M, H, D = k_cache.shape
    B = k_base.shape[0]
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().hsa_active_attention_prefix(
        _p(q), _p(q_idx), n_active, _p(k_cache) if M else None, _p(v_cache) if M else None, M,
        _p(k_base) if B else None, _p(v_base) if B else None, B, H, D, float(scale), _p(out),
        _dtype_code(k_cache if M else k_base), _p(workspace), ws_bytes, _stream(stream)),
        "hsa_active_attention_prefix")


def hsa_reorder_tokens(group_of, n_baseline: int, order, where=None, group_new=None,
                       stream=None) -> None:
    _check(lib().hsa_reorder_tokens(_p(group_of), group_of.numel(), n_baseline, _p(order),
                                    _p(where), _p(group_new), _stream(stream)),
           "hsa_reorder_tokens")


def hsa_active_attention_workspace_bytes(n_active: int, N: int, H: int, D: int,
                                         dtype: int = HSA_BF16) -> int:
    return lib().hsa_active_attention_workspace_bytes(n_active, N, H, D, dtype)


def hsa_active_attention(q, q_idx, n_active: int, k_cache, v_cache, out, scale: float = 0.0,
                         workspace=None, stream=None) -> None:
    """out[j] = attention of query row q_idx[j] (q: [N,H,D]) or j (q_idx None,
    q: [n_active,H,D]) against the full cache; `workspace` (optional uint8
    device tensor) lets the last wave of CTAs be split along the keys."""
    N, H, D = k_cache.shape
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(lib().hsa_active_attention(_p(q), _p(q_idx), n_active, _p(k_cache), _p(v_cache), N,
                                      H, D, float(scale), _p(out), _dtype_code(k_cache),
                                      _p(workspace), ws_bytes, _stream(stream)),
           "hsa_active_attention")


def hsa_cached_euler(x, v_cache, v_fresh, pos, dsigma: float, n_fresh: int | None = None,
                     stream=None) -> None:
    N, C = x.shape
    if n_fresh is None:
        n_fresh = 0 if v_fresh is None else v_fresh.shape[0]
    _check(lib().hsa_cached_euler(_p(x), _p(v_cache), _p(v_fresh), _p(pos), n_fresh, N, C,
                                  float(dsigma), _stream(stream)), "hsa_cached_euler")


def hsa_cached_euler_l1rel(x, v_cache, v_fresh, pos, dsigma: float, stat, weight: float,
                           n_fresh: int | None = None, stream=None) -> None:
    N, C = x.shape
    if n_fresh is None:
        n_fresh = v_fresh.shape[0]
    _check(lib().hsa_cached_euler_l1rel(_p(x), _p(v_cache), _p(v_fresh), _p(pos), n_fresh, N, C,
                                        float(dsigma), _p(stat), float(weight),
                                        _stream(stream)), "hsa_cached_euler_l1rel")


def hsa_get_device_error(stream=None) -> int:
    """Status of the device-side checks since the last call (synchronises)."""
    return lib().hsa_get_device_error(_stream(stream))


def hsa_launch_count() -> int:
    """Kernels this library has launched in this process (host counter)."""
    return int(lib().hsa_launch_count())


def hsa_test_inject_attention_stall(mode: int) -> int:
    """Test hook (include/hsa_test.h): mode 1 makes following bf16 attention
    launches never load their first value tile, so the bounded wait for it runs
    out and HSA_ERR_TIMEOUT is reported; mode 0 restores normal operation."""
    return _check(lib().hsa_test_inject_attention_stall(mode), "hsa_test_inject_attention_stall")
