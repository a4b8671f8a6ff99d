"""STRIDE scoring path on one GB300 (arXiv 2609.14636): Python binding.

A thin ctypes layer over ``libstride.so`` (include/stride.h).  The functions
keep the C names and argument order; they take torch CUDA tensors, check
their dtype/device/shape, pass raw device pointers and the current CUDA
stream, and raise :class:`StrideError` on a non-zero status.  Every step of
the scoring path runs in the library's CUDA kernels: there is no Python or
CPU fallback, and importing this package fails if the library is missing
and cannot be built.

Per-trajectory state and per-turn statistics are opaque byte tensors
(``[n, 80]`` and ``[n, 40]`` uint8) laid out as ``stride_scan_state`` and
``stride_turn_stats``; :func:`state_to_numpy` / :func:`turn_stats_to_numpy`
view copies of them as numpy structured arrays.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

import numpy as np

from . import _build

__all__ = [
    "StrideError", "STATE_DTYPE", "TURN_STATS_DTYPE", "DTYPE_BF16", "DTYPE_F32", "TURN_MEAN",
    "TOKEN_SUM", "DEV_TOKEN_RANGE", "DEV_BAD_LAYOUT", "DEV_TIMEOUT", "lib", "new_state",
    "new_turn_stats", "state_to_numpy", "turn_stats_to_numpy", "stride_state_init",
    "stride_score_batch_workspace_size", "stride_score_batch", "stride_score_step",
    "stride_select_restart", "stride_status_string", "stride_abi_version", "ROW_OUTPUT_KEYS",
    "stride_score_batch_noalloc", "NOALLOC_MAX_ROWS", "OK", "ERR_INVALID_ARG", "ERR_UNSUPPORTED_DTYPE",
    "ERR_WORKSPACE", "ERR_CUDA", "ERR_UNSUPPORTED_DEVICE", "ERR_TOO_LARGE", "PROFILE_BINS", "new_profile",
    "stride_score_step_compact", "stride_force_batch_kernel", "stride_force_step_shape",
    "stride_selftest_bounded_wait", "stride_buffer_record", "stride_score_batch_multi_teacher",
    "multi_teacher_workspace_size", "stride_partial_lse", "stride_combine_partials", "stride_scan_logprobs",
]

DTYPE_BF16, DTYPE_F32 = 0, 1
TURN_MEAN, TOKEN_SUM = 0, 1
DEV_TOKEN_RANGE, DEV_BAD_LAYOUT, DEV_TIMEOUT = 0x1, 0x2, 0x4
ROW_OUTPUT_KEYS = ("logp_s", "logp_t", "opd", "lse_s", "lse_t", "x_s", "x_t")
NOALLOC_MAX_ROWS = 65536  # STRIDE_NOALLOC_MAX_ROWS
MAX_VOCAB = 1 << 30  # STRIDE_MAX_VOCAB
OK, ERR_INVALID_ARG, ERR_UNSUPPORTED_DTYPE, ERR_WORKSPACE, ERR_CUDA, ERR_UNSUPPORTED_DEVICE, ERR_TOO_LARGE = range(7)

STATE_DTYPE = np.dtype([("cum", "<f8"), ("turn_sum_t", "<f8"), ("turn_sum_d", "<f8"),
                        ("turn_sum_l", "<f8"), ("loss", "<f8"), ("rows_seen", "<i8"),
                        ("loss_tokens", "<i8"), ("stop_row", "<i8"), ("stop_turn", "<i4"),
                        ("turn_tokens", "<i4"), ("turn_idx", "<i4"), ("stopped", "<i4")])
TURN_STATS_DTYPE = np.dtype([("sum_t", "<f8"), ("sum_d", "<f8"), ("sum_l", "<f8"), ("cum", "<f8"),
                             ("mean_t", "<f4"), ("n", "<i4")])
PROFILE_BINS = 10
assert STATE_DTYPE.itemsize == 80 and TURN_STATS_DTYPE.itemsize == 40


class StrideError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn}: {stride_status_string(code)} (code {code})")
        self.code = code


class _RowOutputs(ctypes.Structure):
    _fields_ = [(k, ctypes.c_void_p) for k in ROW_OUTPUT_KEYS]


_LIB = None


def lib() -> ctypes.CDLL:
    """The loaded libstride.so (built in-tree on first use if absent)."""
    global _LIB
    if _LIB is None:
        path = _build.LIB
        if not _build.up_to_date():
            _build.build()
        if not Path(path).exists():
            raise ImportError(f"libstride.so not found at {path}")
        L = ctypes.CDLL(str(path))
        P, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
        L.stride_state_init.argtypes = [P, i32, P]
        L.stride_score_batch_workspace_size.argtypes = [i64]
        L.stride_score_batch_workspace_size.restype = sz
        L.stride_score_batch.argtypes = [P, P, i32, i64, i64, P, P, P, P, i32, i32, i64, i64, i32, P, f32,
                                         P, P, P, P, P, P, sz, P]
        L.stride_score_step.argtypes = [P, P, i32, i64, i64, P, P, i32, i32, P, f32, P, P, P, P, P, P]
        L.stride_score_step_compact.argtypes = [P, P, i32, i64, i64, P, P, P, i32, i32, i32, P, f32, P, P, P, P,
                                                P, P]
        L.stride_force_batch_kernel.argtypes = [ctypes.c_char_p]
        L.stride_force_step_shape.argtypes = [i32, i32]
        L.stride_select_restart.argtypes = [P, P, P, f32, i32, i32, P, P, P]
        L.stride_buffer_record.argtypes = [P, P, i32, i32, P, P, P, P, i32, P, P]
        L.stride_partial_lse.argtypes = [P, P, i32, i64, i64, i64, P, i64, P, P, P]
        L.stride_combine_partials.argtypes = [P, i32, i64, P, P, P, P, P, P]
        L.stride_scan_logprobs.argtypes = [P, P, P, P, P, i32, i32, i64, i64, i32, P, f32, P, P, P, P, P, P, sz, P]
        for fn in ("stride_partial_lse", "stride_combine_partials", "stride_scan_logprobs"):
            getattr(L, fn).restype = ctypes.c_int
        L.stride_score_batch_multi_teacher.argtypes = [P, P, P, i32, i64, P, P, i32, i64, i64, P, P, P, P, i32,
                                                       i32, i64, i64, i32, P, f32, P, P, P, P, P, P, sz, P]
        L.stride_score_batch_multi_teacher.restype = ctypes.c_int
        L.stride_buffer_record.restype = ctypes.c_int
        L.stride_selftest_bounded_wait.argtypes = [i32, ctypes.c_uint64, P, P, sz, P]
        L.stride_selftest_bounded_wait.restype = ctypes.c_int
        L.stride_selftest_stream_read.argtypes = [P, P, ctypes.c_uint64, i32, i32, P, P]
        L.stride_selftest_stream_read.restype = ctypes.c_int
        L.stride_score_batch_noalloc.argtypes = [P, P, i32, i64, i64, P, P, P, P, i32, i32, i64, i64, i32,
                                                 P, f32, P, P, P, P, P, P]
        L.stride_status_string.argtypes = [ctypes.c_int]
        L.stride_status_string.restype = ctypes.c_char_p
        L.stride_abi_version.restype = ctypes.c_int
        for fn in ("stride_state_init", "stride_score_batch", "stride_score_step", "stride_select_restart",
                   "stride_score_batch_noalloc", "stride_score_step_compact", "stride_force_batch_kernel",
                   "stride_force_step_shape"):
            getattr(L, fn).restype = ctypes.c_int
        _LIB = L
    return _LIB


def stride_status_string(code: int) -> str:
    return lib().stride_status_string(int(code)).decode()


def stride_abi_version() -> int:
    return int(lib().stride_abi_version())


# ---------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------
def _torch():
    import torch

    return torch


def _stream(stream) -> int:
    torch = _torch()
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _dev(t, name: str, dtype=None, numel: int | None = None, optional: bool = False):
    if t is None:
        if optional:
            return None
        raise ValueError(f"{name} is required")
    torch = _torch()
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements, needs {numel}")
    return t.data_ptr()


def _logits(S, T):
    torch = _torch()
    for name, x in (("S", S), ("T", T)):
        if not isinstance(x, torch.Tensor) or not x.is_cuda or x.dim() != 2 or x.stride(1) != 1:
            raise TypeError(f"{name} must be a 2-D CUDA tensor with unit column stride")
    if S.dtype != T.dtype or S.shape != T.shape or S.stride(0) != T.stride(0):
        raise ValueError("S and T must share dtype, shape and row stride")
    if S.dtype == torch.bfloat16:
        dt = DTYPE_BF16
    elif S.dtype == torch.float32:
        dt = DTYPE_F32
    else:
        raise TypeError(f"logits must be bfloat16 or float32, got {S.dtype}")
    return dt, S.stride(0)


def _row_outputs(out: dict | None, rows: int):
    if not out:
        return None
    torch = _torch()
    ro = _RowOutputs()
    for k, v in out.items():
        if k not in ROW_OUTPUT_KEYS:
            raise KeyError(f"unknown row output {k!r}")
        setattr(ro, k, _dev(v, k, torch.float32, rows))
    return ctypes.byref(ro)


def _lambda(lam, n: int):
    torch = _torch()
    if isinstance(lam, torch.Tensor):
        return _dev(lam, "lambda", torch.float32, n), float("nan")
    return None, float(lam)


def _check(fn: str, rc: int):
    if rc != 0:
        raise StrideError(fn, rc)


# ---------------------------------------------------------------------------
# state / stats buffers
# ---------------------------------------------------------------------------
def new_state(n: int, device="cuda", stream=None):
    """Allocate n stride_scan_state on the device and initialise them."""
    torch = _torch()
    st = torch.empty((max(n, 1), STATE_DTYPE.itemsize), dtype=torch.uint8, device=device)
    stride_state_init(st, n, stream)
    return st


def new_turn_stats(n: int, device="cuda"):
    torch = _torch()
    return torch.zeros((max(n, 1), TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, device=device)


def new_profile(device="cuda"):
    """A zeroed within-turn position profile: float64 [PROFILE_BINS, 3]."""
    torch = _torch()
    return torch.zeros((PROFILE_BINS, 3), dtype=torch.float64, device=device)


def state_to_numpy(st) -> np.ndarray:
    return st.detach().cpu().numpy().reshape(-1).view(STATE_DTYPE)


def turn_stats_to_numpy(ts) -> np.ndarray:
    return ts.detach().cpu().numpy().reshape(-1).view(TURN_STATS_DTYPE)


# ---------------------------------------------------------------------------
# the C ABI, one function each
# ---------------------------------------------------------------------------
def stride_state_init(state, n: int, stream=None) -> None:
    torch = _torch()
    p = _dev(state, "state", torch.uint8, n * STATE_DTYPE.itemsize)
    _check("stride_state_init", lib().stride_state_init(p, int(n), _stream(stream)))


def stride_score_batch_workspace_size(window_rows: int) -> int:
    return int(lib().stride_score_batch_workspace_size(int(window_rows)))


def stride_score_batch(S, T, tokens, traj_row_off, turn_row_off, traj_turn_off, row_begin: int,
                       row_end: int, stop_mode: int, lam, state, out: dict | None = None,
                       turn_stats=None, dev_status=None, workspace=None, V: int | None = None,
                       stream=None, profile=None) -> None:
    """Score global rows [row_begin, row_end) of a ragged trajectory layout.

    S, T: [row_end-row_begin, ld] bf16/fp32 logits of those rows; tokens int32;
    offsets int64/int64/int32 device tensors of the whole layout; lam a float
    or a float32 [n_traj] tensor; state from :func:`new_state`; out a dict
    of float32 [rows] tensors keyed by ROW_OUTPUT_KEYS; turn_stats from
    :func:`new_turn_stats`; dev_status an int32 [1] tensor; workspace a uint8
    tensor of at least stride_score_batch_workspace_size(rows) bytes (256-byte
    aligned; torch's allocator returns such blocks); profile a float64
    [10, 3] tensor from :func:`new_profile`, added to."""
    torch = _torch()
    dt, ld = _logits(S, T)
    rows = int(row_end) - int(row_begin)
    V = S.shape[1] if V is None else int(V)
    n_traj = traj_row_off.numel() - 1
    n_turns = turn_row_off.numel() - 1
    lam_p, lam_all = _lambda(lam, n_traj)
    ws_p = _dev(workspace, "workspace", torch.uint8, optional=True)  # size checked by the library
    rc = lib().stride_score_batch(
        S.data_ptr(), T.data_ptr(), dt, ld, V, _dev(tokens, "tokens", torch.int32, rows),
        _dev(traj_row_off, "traj_row_off", torch.int64), _dev(turn_row_off, "turn_row_off", torch.int64),
        _dev(traj_turn_off, "traj_turn_off", torch.int32), n_traj, n_turns, int(row_begin),
        int(row_end), int(stop_mode), lam_p, lam_all,
        _dev(state, "state", torch.uint8, n_traj * STATE_DTYPE.itemsize), _row_outputs(out, rows),
        _dev(turn_stats, "turn_stats", torch.uint8, n_turns * TURN_STATS_DTYPE.itemsize, optional=True),
        _dev(profile, "profile", torch.float64, 3 * PROFILE_BINS, optional=True),
        _dev(dev_status, "dev_status", torch.int32, 1, optional=True), ws_p,
        0 if workspace is None else workspace.numel(), _stream(stream))
    _check("stride_score_batch", rc)


def stride_score_step(S, T, tokens, turn_end, stop_mode: int, lam, state, out: dict | None = None,
                      stopped_now=None, turn_out=None, dev_status=None, V: int | None = None,
                      stream=None) -> None:
    """One decode step over B = S.shape[0] rollouts (see include/stride.h)."""
    torch = _torch()
    dt, ld = _logits(S, T)
    B = S.shape[0]
    V = S.shape[1] if V is None else int(V)
    lam_p, lam_all = _lambda(lam, B)
    rc = lib().stride_score_step(
        S.data_ptr(), T.data_ptr(), dt, ld, V, _dev(tokens, "tokens", torch.int32, B),
        _dev(turn_end, "turn_end", torch.uint8, B), B, int(stop_mode), lam_p, lam_all,
        _dev(state, "state", torch.uint8, B * STATE_DTYPE.itemsize), _row_outputs(out, B),
        _dev(stopped_now, "stopped_now", torch.uint8, B, optional=True),
        _dev(turn_out, "turn_out", torch.uint8, B * TURN_STATS_DTYPE.itemsize, optional=True),
        _dev(dev_status, "dev_status", torch.int32, 1, optional=True), _stream(stream))
    _check("stride_score_step", rc)


def stride_score_step_compact(S, T, tokens, turn_end, rollout_idx, stop_mode: int, lam, state,
                              out: dict | None = None, stopped_now=None, turn_out=None, dev_status=None,
                              V: int | None = None, n_rows: int | None = None, stream=None) -> None:
    """One decode step over the live rollouts, their rows packed: row b of
    S, T, tokens, turn_end and the outputs is rollout rollout_idx[b] (int32
    CUDA tensor of n_rows = len(rollout_idx) entries unless given) of the
    state tensor's rollouts (see include/stride.h)."""
    torch = _torch()
    dt, ld = _logits(S, T)
    n = int(rollout_idx.shape[0]) if n_rows is None else int(n_rows)
    if n > S.shape[0]:
        raise ValueError("S and T need a row per live rollout")
    n_state = state.numel() // STATE_DTYPE.itemsize
    V = S.shape[1] if V is None else int(V)
    lam_p, lam_all = _lambda(lam, n_state)
    rc = lib().stride_score_step_compact(
        S.data_ptr(), T.data_ptr(), dt, ld, V, _dev(tokens, "tokens", torch.int32, n),
        _dev(turn_end, "turn_end", torch.uint8, n), _dev(rollout_idx, "rollout_idx", torch.int32, n), n, n_state,
        int(stop_mode), lam_p, lam_all, _dev(state, "state", torch.uint8, n_state * STATE_DTYPE.itemsize),
        _row_outputs(out, n), _dev(stopped_now, "stopped_now", torch.uint8, n, optional=True),
        _dev(turn_out, "turn_out", torch.uint8, n * TURN_STATS_DTYPE.itemsize, optional=True),
        _dev(dev_status, "dev_status", torch.int32, 1, optional=True), _stream(stream))
    _check("stride_score_step_compact", rc)


def stride_force_batch_kernel(name: str | None) -> None:
    """Fix the batch kernel for tests and diagnosis (None / "auto": automatic)."""
    _check("stride_force_batch_kernel", lib().stride_force_batch_kernel(None if name is None else name.encode()))


def stride_force_step_shape(cta_threads: int, cluster_size: int) -> None:
    """Fix the decode step's CTA size (128 or 512) and CTAs per row for tests
    and diagnosis ((0, 0): automatic)."""
    _check("stride_force_step_shape", lib().stride_force_step_shape(int(cta_threads), int(cluster_size)))


def stride_select_restart(turn_mean, n_turns, correct, alpha: float, k_star, k_max, stream=None) -> None:
    """Restart choice (Eq. 6) over N records: turn_mean float32 [N, T_max],
    n_turns int32 [N], correct uint8 [N, T_max] or None; outputs int32 [N]."""
    torch = _torch()
    if turn_mean.dim() != 2:
        raise ValueError("turn_mean must be [N, T_max]")
    N, T_max = turn_mean.shape
    rc = lib().stride_select_restart(
        _dev(turn_mean, "turn_mean", torch.float32, N * T_max), _dev(n_turns, "n_turns", torch.int32, N),
        _dev(correct, "correct", torch.uint8, N * T_max, optional=True), float(alpha), N, T_max,
        _dev(k_star, "k_star", torch.int32, N), _dev(k_max, "k_max", torch.int32, N), _stream(stream))
    _check("stride_select_restart", rc)


def multi_teacher_workspace_size(window_rows: int) -> int:
    """Workspace bytes of stride_score_batch_multi_teacher for a window."""
    return stride_score_batch_workspace_size(window_rows) + ((8 * int(window_rows) + 255) & ~255)


def stride_score_batch_multi_teacher(S, T_domains, traj_domain, traj_T_row0, tokens, traj_row_off, turn_row_off,
                                     traj_turn_off, row_begin: int, row_end: int, stop_mode: int, lam, state,
                                     out: dict | None = None, turn_stats=None, dev_status=None, workspace=None,
                                     V: int | None = None, stream=None, profile=None) -> None:
    """Batch scoring with one teacher logit buffer per domain (list of 2-D
    CUDA tensors of S's dtype and a common row stride), a per-trajectory
    domain id (uint8) and the trajectory's first row in its domain buffer
    (int64).  See include/stride.h."""
    torch = _torch()
    if not isinstance(S, torch.Tensor) or not S.is_cuda or S.dim() != 2 or S.stride(1) != 1:
        raise TypeError("S must be a 2-D CUDA tensor with unit column stride")
    if S.dtype == torch.bfloat16:
        dt = DTYPE_BF16
    elif S.dtype == torch.float32:
        dt = DTYPE_F32
    else:
        raise TypeError(f"logits must be bfloat16 or float32, got {S.dtype}")
    D = len(T_domains)
    if D < 1:
        raise ValueError("at least one teacher domain")
    ld_T = T_domains[0].stride(0)
    for t in T_domains:
        if t.dtype != S.dtype or t.dim() != 2 or t.stride(1) != 1 or t.stride(0) != ld_T or not t.is_cuda:
            raise ValueError("teacher buffers must be 2-D CUDA tensors of S's dtype with one row stride")
    ptrs = (ctypes.c_void_p * D)(*[t.data_ptr() for t in T_domains])
    nrows = (ctypes.c_int64 * D)(*[t.shape[0] for t in T_domains])
    rows = int(row_end) - int(row_begin)
    V = S.shape[1] if V is None else int(V)
    n_traj = traj_row_off.numel() - 1
    n_turns = turn_row_off.numel() - 1
    lam_p, lam_all = _lambda(lam, n_traj)
    rc = lib().stride_score_batch_multi_teacher(
        S.data_ptr(), ptrs, nrows, D, ld_T, _dev(traj_domain, "traj_domain", torch.uint8, n_traj),
        _dev(traj_T_row0, "traj_T_row0", torch.int64, n_traj), dt, S.stride(0), V,
        _dev(tokens, "tokens", torch.int32, rows), _dev(traj_row_off, "traj_row_off", torch.int64),
        _dev(turn_row_off, "turn_row_off", torch.int64), _dev(traj_turn_off, "traj_turn_off", torch.int32),
        n_traj, n_turns, int(row_begin), int(row_end), int(stop_mode), lam_p, lam_all,
        _dev(state, "state", torch.uint8, n_traj * STATE_DTYPE.itemsize), _row_outputs(out, rows),
        _dev(turn_stats, "turn_stats", torch.uint8, n_turns * TURN_STATS_DTYPE.itemsize, optional=True),
        _dev(profile, "profile", torch.float64, 3 * PROFILE_BINS, optional=True),
        _dev(dev_status, "dev_status", torch.int32, 1, optional=True),
        _dev(workspace, "workspace", torch.uint8, optional=True), 0 if workspace is None else workspace.numel(),
        _stream(stream))
    _check("stride_score_batch_multi_teacher", rc)


def stride_partial_lse(S, T, tokens, col0: int, partials, dev_status=None, V_shard: int | None = None,
                       stream=None) -> None:
    """Partial log-sum-exp of one vocabulary shard (columns col0 .. col0+V_shard-1
    held in S, T [rows, ld]); partials: float32 [rows, 6]."""
    torch = _torch()
    dt, ld = _logits(S, T)
    rows = S.shape[0]
    V_shard = S.shape[1] if V_shard is None else int(V_shard)
    rc = lib().stride_partial_lse(S.data_ptr(), T.data_ptr(), dt, ld, V_shard, int(col0),
                                  _dev(tokens, "tokens", torch.int32, rows), rows,
                                  _dev(partials, "partials", torch.float32, rows * 6),
                                  _dev(dev_status, "dev_status", torch.int32, 1, optional=True), _stream(stream))
    _check("stride_partial_lse", rc)


def stride_combine_partials(partials, logp_s=None, logp_t=None, lse_s=None, lse_t=None, dev_status=None,
                            stream=None) -> None:
    """Merge float32 [n_shards, rows, 6] partials into log-probs."""
    torch = _torch()
    if partials.dim() != 3 or partials.shape[2] != 6:
        raise ValueError("partials must be [n_shards, rows, 6]")
    n, rows = partials.shape[0], partials.shape[1]
    rc = lib().stride_combine_partials(
        _dev(partials, "partials", torch.float32), n, rows, _dev(logp_s, "logp_s", torch.float32, rows, optional=True),
        _dev(logp_t, "logp_t", torch.float32, rows, optional=True), _dev(lse_s, "lse_s", torch.float32, rows, optional=True),
        _dev(lse_t, "lse_t", torch.float32, rows, optional=True),
        _dev(dev_status, "dev_status", torch.int32, 1, optional=True), _stream(stream))
    _check("stride_combine_partials", rc)


def stride_scan_logprobs(logp_s, logp_t, traj_row_off, turn_row_off, traj_turn_off, row_begin: int, row_end: int,
                         stop_mode: int, lam, state, opd=None, turn_stats=None, dev_status=None, workspace=None,
                         stream=None, profile=None) -> None:
    """The scan of stride_score_batch on given log-probs (float32, indexed by
    row - row_begin)."""
    torch = _torch()
    rows = int(row_end) - int(row_begin)
    n_traj = traj_row_off.numel() - 1
    n_turns = turn_row_off.numel() - 1
    lam_p, lam_all = _lambda(lam, n_traj)
    rc = lib().stride_scan_logprobs(
        _dev(logp_s, "logp_s", torch.float32, rows), _dev(logp_t, "logp_t", torch.float32, rows),
        _dev(traj_row_off, "traj_row_off", torch.int64), _dev(turn_row_off, "turn_row_off", torch.int64),
        _dev(traj_turn_off, "traj_turn_off", torch.int32), n_traj, n_turns, int(row_begin), int(row_end),
        int(stop_mode), lam_p, lam_all, _dev(state, "state", torch.uint8, n_traj * STATE_DTYPE.itemsize),
        _dev(opd, "opd", torch.float32, rows, optional=True),
        _dev(turn_stats, "turn_stats", torch.uint8, n_turns * TURN_STATS_DTYPE.itemsize, optional=True),
        _dev(profile, "profile", torch.float64, 3 * PROFILE_BINS, optional=True),
        _dev(dev_status, "dev_status", torch.int32, 1, optional=True),
        _dev(workspace, "workspace", torch.uint8, optional=True), 0 if workspace is None else workspace.numel(),
        _stream(stream))
    _check("stride_scan_logprobs", rc)


def stride_buffer_record(buf_mean, buf_n_turns, task_of_traj, k0_of_traj, turn_stats, traj_turn_off,
                         dev_status=None, stream=None) -> None:
    """Record trajectories' turn means in the prefix buffer H(x) (float32
    [n_tasks, T_max] and int32 [n_tasks], updated in place): each keeps the
    first k0 stored turns of its task, then its own turns (Algorithm 1)."""
    torch = _torch()
    if buf_mean.dim() != 2:
        raise ValueError("buf_mean must be [n_tasks, T_max]")
    n_tasks, T_max = buf_mean.shape
    n_traj = traj_turn_off.numel() - 1
    rc = lib().stride_buffer_record(
        _dev(buf_mean, "buf_mean", torch.float32), _dev(buf_n_turns, "buf_n_turns", torch.int32, n_tasks),
        n_tasks, T_max, _dev(task_of_traj, "task_of_traj", torch.int32, n_traj),
        _dev(k0_of_traj, "k0_of_traj", torch.int32, n_traj, optional=True),
        _dev(turn_stats, "turn_stats", torch.uint8), _dev(traj_turn_off, "traj_turn_off", torch.int32, n_traj + 1),
        n_traj, _dev(dev_status, "dev_status", torch.int32, 1, optional=True), _stream(stream))
    _check("stride_buffer_record", rc)


SELFTEST_LOOKBACK, SELFTEST_MBARRIER = 0, 1


def stride_selftest_bounded_wait(which: int, timeout_ns: int, dev_status, workspace, stream=None) -> None:
    """Run one of the library's bounded device waits on a flag nothing sets
    (include/stride_selftest.h); the kernel ORs DEV_TIMEOUT into dev_status."""
    torch = _torch()
    rc = lib().stride_selftest_bounded_wait(int(which), int(timeout_ns), _dev(dev_status, "dev_status", torch.int32, 1),
                                            _dev(workspace, "workspace", torch.uint8), workspace.numel(), _stream(stream))
    _check("stride_selftest_bounded_wait", rc)


def stride_selftest_stream_read(a, b, bytes_each: int, grid: int, threads: int, sink, stream=None) -> None:
    """Read-only stream over bytes_each bytes of CUDA tensors a (and b, or
    None) with the scoring kernels' loads (see include/stride_selftest.h)."""
    torch = _torch()
    for name, x in (("a", a), ("b", b)):
        if x is not None and (not isinstance(x, torch.Tensor) or not x.is_cuda or not x.is_contiguous()
                              or x.numel() * x.element_size() < bytes_each):
            raise ValueError(f"{name} must be a contiguous CUDA tensor of at least {bytes_each} bytes")
    rc = lib().stride_selftest_stream_read(a.data_ptr(), None if b is None else b.data_ptr(), int(bytes_each),
                                           int(grid), int(threads), _dev(sink, "sink", torch.int32, int(grid)),
                                           _stream(stream))
    _check("stride_selftest_stream_read", rc)


def stride_score_batch_noalloc(S, T, tokens, traj_row_off, turn_row_off, traj_turn_off, row_begin: int,
                               row_end: int, stop_mode: int, lam, state, out: dict | None = None,
                               turn_stats=None, dev_status=None, V: int | None = None, stream=None,
                               profile=None) -> None:
    """stride_score_batch without a workspace argument, for callers that
    cannot allocate device memory: the library's built-in scratch (at most
    NOALLOC_MAX_ROWS rows per call) is used instead.  Calls that overlap on
    the GPU race on that scratch; order them on one stream."""
    torch = _torch()
    dt, ld = _logits(S, T)
    rows = int(row_end) - int(row_begin)
    V = S.shape[1] if V is None else int(V)
    n_traj = traj_row_off.numel() - 1
    n_turns = turn_row_off.numel() - 1
    lam_p, lam_all = _lambda(lam, n_traj)
    rc = lib().stride_score_batch_noalloc(
        S.data_ptr(), T.data_ptr(), dt, ld, V, _dev(tokens, "tokens", torch.int32, max(rows, 0)),
        _dev(traj_row_off, "traj_row_off", torch.int64), _dev(turn_row_off, "turn_row_off", torch.int64),
        _dev(traj_turn_off, "traj_turn_off", torch.int32), n_traj, n_turns, int(row_begin),
        int(row_end), int(stop_mode), lam_p, lam_all,
        _dev(state, "state", torch.uint8, n_traj * STATE_DTYPE.itemsize), _row_outputs(out, max(rows, 0)),
        _dev(turn_stats, "turn_stats", torch.uint8, n_turns * TURN_STATS_DTYPE.itemsize, optional=True),
        _dev(profile, "profile", torch.float64, 3 * PROFILE_BINS, optional=True),
        _dev(dev_status, "dev_status", torch.int32, 1, optional=True), _stream(stream))
    _check("stride_score_batch_noalloc", rc)
