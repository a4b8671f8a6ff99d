"""fp64 CPU oracle for the STRIDE scoring path (arXiv 2609.14636).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline / reference leg of ``bench.py``.  The product library
never imports, links or calls anything here, and nothing here imports the
product package.

The arithmetic lives in ``oracle.c`` (plain C, fp64, libm ``exp``/``log``,
compiled without fast-math or FMA contraction); this module only builds it and
marshals numpy arrays.  Definitions followed (see the C file for detail):

* :func:`row_logprobs`   -- log-softmax gather of Eq. 1 / Eq. 4, d = -r_t.
* :func:`scan_batch`     -- Eq. 4 turn means, Eq. 5 stop rule with the
  prefix-buffer offset (Sec. 4.1), token-level variant (Sec. 5.5).
* :func:`step_update`    -- Algorithm 1's inner loop, one token per call.
* :func:`select_restart` -- quality gate (Sec. 4.2), K_max, Eq. 6.
* :func:`buffer_record`  -- Algorithm 1's record of {l_k} in H(x), with the
  reused prefix kept (Sec. 4.2 step 3).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from pathlib import Path

import numpy as np

HERE = Path(__file__).resolve().parent
SRC = HERE / "oracle.c"
LIB = HERE / "liboracle.so"

DTYPE_BF16 = 0
DTYPE_F32 = 1
TURN_MEAN = 0
TOKEN_SUM = 1

OK, ERR_ARG, ERR_TOKEN, ERR_EMPTY_TURN = 0, 1, 2, 3


def build(force: bool = False, src: Path | str = SRC, out: Path | str = LIB) -> Path:
    """Compile an oracle C source with gcc (no fast-math, no FMA contraction)."""
    src, out = Path(src), Path(out)
    if out.exists() and not force and out.stat().st_mtime >= src.stat().st_mtime:
        return out
    tmp = out.with_name(out.name + f".tmp{os.getpid()}")
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
           "-fno-fast-math", "-pthread", str(src), "-o", str(tmp), "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


class OracleLib:
    """The oracle library loaded from one compiled copy of oracle.c."""

    def __init__(self, path: Path | str):
        lib = ctypes.CDLL(str(path))
        P = ctypes.c_void_p
        i64, i32, ci = ctypes.c_int64, ctypes.c_int32, ctypes.c_int
        lib.oracle_row_logprobs.argtypes = [P, P, ci, i64, i64, P, i64, P, P, P, P, P, P, P, ci]
        lib.oracle_row_logprobs.restype = ci
        lib.oracle_scan_batch.argtypes = [P, P, P, P, P, P, i32, ci, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P]
        lib.oracle_scan_batch.restype = ci
        lib.oracle_step_update.argtypes = [P, P, P, i32, ci, P, P, P, P, P, P, P, P, P, P, P, P]
        lib.oracle_step_update.restype = ci
        lib.oracle_select_restart.argtypes = [P, P, P, ctypes.c_float, i32, i32, P, P]
        lib.oracle_select_restart.restype = ci
        lib.oracle_rollout_size.restype = ci
        lib.oracle_buffer_record.argtypes = [P, P, i32, i32, P, P, P, P, i32]
        lib.oracle_buffer_record.restype = ci
        self.lib = lib

    # ---- Eq. 1 / Eq. 4: per-row log-probs --------------------------------
    def row_logprobs(self, S: np.ndarray, T: np.ndarray, tokens: np.ndarray, V: int | None = None,
                     nthreads: int | None = None, check: bool = True) -> dict:
        """Per-row fp64 log-probs of ``tokens`` under logits S (student), T (teacher).

        S, T: 2-D arrays [rows, ld]; ``np.uint16`` holds raw bf16 bits,
        ``np.float32`` is fp32.  S may be None (teacher only; the student
        outputs are NaN).  V defaults to ld.  Returns a dict of fp64
        arrays logp_s, logp_t, d, lse_s, lse_t, x_s, x_t and the return code.
        """
        if T.dtype == np.uint16:
            dt = DTYPE_BF16
        elif T.dtype == np.float32:
            dt = DTYPE_F32
        else:
            raise TypeError(f"unsupported logit dtype {T.dtype}")
        if T.ndim != 2 or (S is not None and (S.dtype != T.dtype or S.shape != T.shape)):
            raise ValueError("S and T must be 2-D arrays of one dtype and shape (S may be None)")
        S = None if S is None else np.ascontiguousarray(S)
        T = np.ascontiguousarray(T)
        rows, ld = T.shape
        V = ld if V is None else int(V)
        tok = np.ascontiguousarray(tokens, dtype=np.int32)
        if tok.shape != (rows,):
            raise ValueError("tokens must be [rows]")
        out = {k: np.empty(rows, np.float64)
               for k in ("logp_s", "logp_t", "d", "lse_s", "lse_t", "x_s", "x_t")}
        rc = self.lib.oracle_row_logprobs(
            _ptr(S), _ptr(T), dt, ld, V, _ptr(tok), rows, _ptr(out["logp_s"]), _ptr(out["logp_t"]),
            _ptr(out["d"]), _ptr(out["lse_s"]), _ptr(out["lse_t"]), _ptr(out["x_s"]),
            _ptr(out["x_t"]), nthreads or default_threads())
        if check and rc != OK:
            raise ValueError(f"oracle_row_logprobs returned {rc}")
        out["rc"] = rc
        return out

    # ---- Eq. 4 / Eq. 5 / Sec. 5.5: batch scan ------------------------------
    def scan_batch(self, logp_t, d, traj_row_off, turn_row_off, traj_turn_off, mode: int, lam,
                   cum_in=None, logp_s=None) -> dict:
        """Turn means, the stop rule, the OPD loss on retained tokens (needs
        logp_s) and the within-turn decile profile over ragged trajectories.

        ``lam`` is a scalar or a per-trajectory array.  Row arrays are indexed
        from ``traj_row_off[0]``."""
        logp_t = np.ascontiguousarray(logp_t, np.float64)
        d = None if d is None else np.ascontiguousarray(d, np.float64)
        ls = None if logp_s is None else np.ascontiguousarray(logp_s, np.float64)
        tro = np.ascontiguousarray(traj_row_off, np.int64)
        uro = np.ascontiguousarray(turn_row_off, np.int64)
        tto = np.ascontiguousarray(traj_turn_off, np.int32)
        n_traj = tro.shape[0] - 1
        n_turns = uro.shape[0] - 1
        lam_a = np.ascontiguousarray(np.broadcast_to(np.asarray(lam, np.float64), (n_traj,)))
        cin = None if cum_in is None else np.ascontiguousarray(cum_in, np.float64)
        out = dict(
            turn_sum_t=np.empty(n_turns), turn_sum_d=np.empty(n_turns), turn_sum_l=np.empty(n_turns),
            turn_mean=np.empty(n_turns), turn_n=np.empty(n_turns, np.int64), turn_cum=np.empty(n_turns),
            traj_cum=np.empty(n_traj), stop_turn=np.empty(n_traj, np.int32),
            stop_row=np.empty(n_traj, np.int64), traj_loss=np.empty(n_traj),
            traj_loss_tokens=np.empty(n_traj, np.int64), row_cum=np.empty(logp_t.shape[0]),
            profile=np.zeros(30))
        rc = self.lib.oracle_scan_batch(
            _ptr(logp_t), _ptr(d), _ptr(ls), _ptr(tro), _ptr(uro), _ptr(tto), n_traj, mode, _ptr(lam_a),
            _ptr(cin), _ptr(out["turn_sum_t"]), _ptr(out["turn_sum_d"]), _ptr(out["turn_sum_l"]),
            _ptr(out["turn_mean"]), _ptr(out["turn_n"]), _ptr(out["turn_cum"]), _ptr(out["traj_cum"]),
            _ptr(out["stop_turn"]), _ptr(out["stop_row"]), _ptr(out["traj_loss"]),
            _ptr(out["traj_loss_tokens"]), _ptr(out["row_cum"]), _ptr(out["profile"]))
        if rc != OK:
            raise ValueError(f"oracle_scan_batch returned {rc}")
        out["profile"] = out["profile"].reshape(10, 3)
        return out

    # ---- Algorithm 1 inner loop: one decode step ---------------------------
    def new_rollouts(self, B: int):
        assert self.lib.oracle_rollout_size() == ctypes.sizeof(Rollouts)
        arr = (Rollouts * B)()
        for s in arr:
            s.stop_row = -1
            s.stop_turn = -1
        return arr

    def step_update(self, state, logp_s, logp_t, turn_end, mode: int, lam) -> dict:
        """One decode step for len(state) rollouts."""
        B = len(state)
        ps = np.ascontiguousarray(logp_s, np.float64)
        pt = np.ascontiguousarray(logp_t, np.float64)
        te = np.ascontiguousarray(turn_end, np.uint8)
        lam_a = np.ascontiguousarray(np.broadcast_to(np.asarray(lam, np.float64), (B,)))
        out = dict(logp_s=np.empty(B), logp_t=np.empty(B), d=np.empty(B),
                   stopped_now=np.empty(B, np.uint8), turn_sum_t=np.empty(B),
                   turn_sum_d=np.empty(B), turn_sum_l=np.empty(B), turn_mean=np.empty(B),
                   turn_n=np.empty(B, np.int32), turn_cum=np.empty(B))
        rc = self.lib.oracle_step_update(
            _ptr(ps), _ptr(pt), _ptr(te), B, mode, _ptr(lam_a), ctypes.cast(state, ctypes.c_void_p),
            _ptr(out["logp_s"]), _ptr(out["logp_t"]), _ptr(out["d"]), _ptr(out["stopped_now"]),
            _ptr(out["turn_sum_t"]), _ptr(out["turn_sum_d"]), _ptr(out["turn_sum_l"]),
            _ptr(out["turn_mean"]), _ptr(out["turn_n"]), _ptr(out["turn_cum"]))
        if rc != OK:
            raise ValueError(f"oracle_step_update returned {rc}")
        return out

    # ---- Algorithm 1: record {l_k} to H(x) ----------------------------------
    def buffer_record(self, mean, n_turns, task, k0, turn_mean, traj_turn_off):
        """Update a prefix buffer in place (numpy arrays mean [n_tasks, T_max]
        float32 and n_turns [n_tasks] int32) with the trajectories' records."""
        assert mean.dtype == np.float32 and mean.flags.c_contiguous and n_turns.dtype == np.int32
        n_tasks, T_max = mean.shape
        tk = np.ascontiguousarray(task, np.int32)
        k0a = None if k0 is None else np.ascontiguousarray(k0, np.int32)
        tm = np.ascontiguousarray(turn_mean, np.float32)
        tto = np.ascontiguousarray(traj_turn_off, np.int32)
        rc = self.lib.oracle_buffer_record(_ptr(mean), _ptr(n_turns), n_tasks, T_max, _ptr(tk), _ptr(k0a),
                                           _ptr(tm), _ptr(tto), tk.shape[0])
        if rc != OK:
            raise ValueError(f"oracle_buffer_record returned {rc}")

    # ---- Sec. 4.2 / Eq. 6: restart choice -----------------------------------
    def select_restart(self, mean, n_turns, mask, alpha: float):
        """Quality gate, K_max and the weakest correct turn.  Returns
        (k_star, k_max) as int32 arrays; k_star is 0-based (= K0)."""
        mean = np.ascontiguousarray(mean, np.float32)
        if mean.ndim != 2:
            raise ValueError("mean must be [N, T_max]")
        N, T_max = mean.shape
        nt = np.ascontiguousarray(n_turns, np.int32)
        m = None if mask is None else np.ascontiguousarray(mask, np.uint8)
        ks = np.empty(N, np.int32)
        km = np.empty(N, np.int32)
        rc = self.lib.oracle_select_restart(_ptr(mean), _ptr(nt), _ptr(m), float(alpha), N, T_max,
                                            _ptr(ks), _ptr(km))
        if rc != OK:
            raise ValueError(f"oracle_select_restart returned {rc}")
        return ks, km


class Rollouts(ctypes.Structure):
    """Mirror of the oracle's own per-rollout step state."""
    _fields_ = [("cum", ctypes.c_double), ("turn_sum_t", ctypes.c_double),
                ("turn_sum_d", ctypes.c_double), ("turn_sum_l", ctypes.c_double),
                ("loss", ctypes.c_double), ("rows_seen", ctypes.c_int64),
                ("stop_row", ctypes.c_int64), ("stop_turn", ctypes.c_int32),
                ("turn_tokens", ctypes.c_int32), ("turn_idx", ctypes.c_int32),
                ("stopped", ctypes.c_int32)]


def rollouts_to_numpy(state) -> dict:
    v = rollouts_view(state)
    return {k: v[k].copy() for k in v.dtype.names}


def rollouts_view(state) -> np.ndarray:
    """A live numpy structured view of a rollout array (no copy)."""
    return np.frombuffer(state, dtype=np.dtype(Rollouts))


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def default_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


_default: OracleLib | None = None


def get() -> OracleLib:
    """The oracle built from oracle.c in this directory."""
    global _default
    if _default is None:
        _default = OracleLib(build())
    return _default


def row_logprobs(*a, **k):
    return get().row_logprobs(*a, **k)


def scan_batch(*a, **k):
    return get().scan_batch(*a, **k)


def new_rollouts(B: int):
    return get().new_rollouts(B)


def step_update(*a, **k):
    return get().step_update(*a, **k)


def select_restart(*a, **k):
    return get().select_restart(*a, **k)


def buffer_record(*a, **k):
    return get().buffer_record(*a, **k)
