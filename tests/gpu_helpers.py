"""Helpers for the GPU parity tests: feed the same seeded inputs to the CUDA
path (through the C ABI) and to the oracle, and compare.

Tolerances (stated where the path's outputs are specified):
* gathered logits x_s, x_t and integer results (n_k, stop rows and turns,
  k*, K_max): bit-exact;
* per-token log-probs logp_s, logp_t, d and LSEs: 2e-3 absolute;
* running sums (cum per turn, per trajectory): 1e-5 relative;
* per-turn sums sum_t, sum_d: |error| <= 1e-5 * sum_i (|x_i| + 1) over the
  turn's terms x_i (1e-5 relative for sum_t, whose terms are <= 0 and of
  order -5; for sum_d, whose terms can cancel, the "+1" per token bounds the
  fp32 rounding of each d_i);
* l_k (fp32): 2e-3 absolute (a mean of per-token values, each within 2e-3);
* the OPD-loss sums (per turn, per trajectory over retained tokens):
  1e-5 * sum(|logp_S * d| + |logp_S| + |d| + 1) over the summed tokens -- a
  term logp_S * d carries the error of each factor scaled by the other;
  the within-turn profile sums: like the per-turn sums; retained-token counts
  and profile counts exact;
* a stop index may differ from the oracle's only where the oracle's running
  sum lies within 1e-3 of lambda at every test position between the two;
  with equal stop indices, a token whose oracle running sum before it lies
  within 1e-3 of lambda may be retained or not (the retained count lies
  between the prefixes retained for certain and at most; the loss is the
  certain prefix's plus at most those tokens' terms).
"""
from __future__ import annotations

import numpy as np

import oracle

LOGP_ATOL = 2e-3
SUM_RTOL = 1e-5
TIE_BAND = 1e-3


def torch_mod():
    import torch

    return torch


def to_dev(a: np.ndarray, device="cuda"):
    """uint16 arrays are raw bf16 bits; float32 stays float32."""
    torch = torch_mod()
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


def run_batch(stride, S, T, tokens, lay, mode, lam, windows=None, V=None, out_keys=None,
              device="cuda", state=None):
    """Score all rows of `lay` through stride_score_batch, in the given row
    windows (default: one window).  S/T are numpy arrays [rows, ld] or torch
    CUDA tensors.  Returns numpy results."""
    torch = torch_mod()
    R = lay.rows
    St = S if isinstance(S, torch.Tensor) else to_dev(S, device)
    Tt = T if isinstance(T, torch.Tensor) else to_dev(T, device)
    tk = tokens if isinstance(tokens, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(tokens, np.int32)).to(device)
    offs = [torch.from_numpy(a).to(device) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(lay.n_traj, device) if state is None else state
    ts = stride.new_turn_stats(lay.n_turns, device)
    prof = stride.new_profile(device)
    keys = out_keys or stride.ROW_OUTPUT_KEYS
    out = {k: torch.full((R,), float("nan"), dtype=torch.float32, device=device) for k in keys}
    status = torch.zeros(1, dtype=torch.int32, device=device)
    if isinstance(lam, np.ndarray):
        lam_arg = torch.from_numpy(lam.astype(np.float32)).to(device)
    else:
        lam_arg = float(np.float32(lam))
    base = int(lay.traj_row_off[0])
    if windows is None:
        windows = [(base, base + R)]
    wmax = max(b - a for a, b in windows)
    ws = torch.empty(max(1, stride.stride_score_batch_workspace_size(wmax)), dtype=torch.uint8, device=device)
    for a, b in windows:
        o = {k: v[a - base:b - base] for k, v in out.items()}
        stride.stride_score_batch(St[a - base:b - base], Tt[a - base:b - base], tk[a - base:b - base], *offs,
                                  a, b, mode, lam_arg, st, out=o, turn_stats=ts, dev_status=status,
                                  workspace=ws, V=V, profile=prof)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["state"] = stride.state_to_numpy(st)[: lay.n_traj]
    res["turn_stats"] = stride.turn_stats_to_numpy(ts)[: lay.n_turns]
    res["status"] = int(status.item())
    res["profile"] = prof.cpu().numpy()
    return res


def oracle_batch(S, T, tokens, lay, mode, lam, V=None):
    o = oracle.row_logprobs(S, T, tokens, V=V, check=False)
    lam64 = np.asarray(lam, np.float32).astype(np.float64)
    sc = oracle.scan_batch(o["logp_t"], o["d"], lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                           mode, lam64, logp_s=o["logp_s"])
    o.update(sc)
    return o


def loss_mag(ls, d) -> float:
    """Magnitude a sum of OPD-loss terms logp_S * d is compared against."""
    ls, d = np.asarray(ls, np.float64), np.asarray(d, np.float64)
    return float(np.sum(np.abs(ls * d) + np.abs(ls) + np.abs(d) + 1.0))


def stop_matches(g_row, o_row, rc, tests, lam):
    """Stop indices agree, or every test position from the earlier of the two
    up to (not including) the later one has the oracle's running sum within
    TIE_BAND of lambda ("no stop" counts as the trajectory's length)."""
    if g_row == o_row:
        return True
    n = len(rc)
    g = n if g_row < 0 else g_row
    o = n if o_row < 0 else o_row
    lo, hi = min(g, o), max(g, o)
    between = [t for t in tests if lo <= t < hi]
    return len(between) > 0 and all(abs(rc[t] - lam) < TIE_BAND for t in between)


def compare_rows(g, o, rows=slice(None)):
    for k, ok in (("logp_s", "logp_s"), ("logp_t", "logp_t"), ("opd", "d"), ("lse_s", "lse_s"), ("lse_t", "lse_t")):
        if k in g:
            a, b = g[k][rows], o[ok][rows]
            fin = np.isfinite(b)
            assert np.array_equal(np.isfinite(a), fin), f"{k}: finiteness differs"
            err = np.max(np.abs(a[fin] - b[fin])) if fin.any() else 0.0
            assert err <= LOGP_ATOL, f"{k}: max abs error {err}"
    for k in ("x_s", "x_t"):
        if k in g:
            a, b = g[k][rows].astype(np.float64), o[k][rows]
            same = (a == b) | (np.isnan(a) & np.isnan(b))
            assert same.all(), f"{k}: gathered logits differ at {np.nonzero(~same)[0][:5]}"


def compare_scan(g, o, lay, mode, lam):
    ts = g["turn_stats"]
    assert np.array_equal(ts["n"], o["turn_n"]), "turn lengths differ"
    # per-turn sums against the sum of magnitudes of the summed terms
    lp, d = o["logp_t"], o["d"]
    base = lay.traj_row_off[0]
    for k in range(lay.n_turns):
        a, b = lay.turn_row_off[k] - base, lay.turn_row_off[k + 1] - base
        mag_t = np.sum(np.abs(lp[a:b]) + 1.0)
        mag_d = np.sum(np.abs(d[a:b]) + 1.0)
        assert abs(ts["sum_t"][k] - o["turn_sum_t"][k]) <= SUM_RTOL * mag_t, ("sum_t", k)
        assert abs(ts["sum_d"][k] - o["turn_sum_d"][k]) <= SUM_RTOL * mag_d, ("sum_d", k)
        mag_l = loss_mag(lp[a:b] + d[a:b], d[a:b])
        assert abs(ts["sum_l"][k] - o["turn_sum_l"][k]) <= SUM_RTOL * mag_l, ("sum_l", k)
        assert abs(ts["mean_t"][k] - o["turn_mean"][k]) <= LOGP_ATOL, ("mean_t", k)
        assert abs(ts["cum"][k] - o["turn_cum"][k]) <= SUM_RTOL * abs(o["turn_cum"][k]) + 1e-12, ("cum", k)
    st = g["state"]
    lam_a = np.broadcast_to(np.asarray(lam, np.float32).astype(np.float64), (lay.n_traj,))
    for i in range(lay.n_traj):
        assert abs(st["cum"][i] - o["traj_cum"][i]) <= SUM_RTOL * abs(o["traj_cum"][i]) + 1e-12, ("traj_cum", i)
        r0, r1 = lay.traj_row_off[i] - base, lay.traj_row_off[i + 1] - base
        k0, k1 = lay.traj_turn_off[i], lay.traj_turn_off[i + 1]
        if mode == oracle.TOKEN_SUM:
            rc = o["row_cum"][r0:r1]
            tests = list(range(r1 - r0))
        else:
            rc = np.full(r1 - r0, np.nan)
            ends = lay.turn_row_off[k0 + 1:k1 + 1] - 1 - lay.traj_row_off[i]
            rc[ends] = o["turn_cum"][k0:k1]
            tests = list(ends)
        gr, orr = int(st["stop_row"][i]), int(o["stop_row"][i])
        assert stop_matches(gr, orr, rc, tests, lam_a[i]), (i, gr, orr)
        if gr == orr:
            assert int(st["stop_turn"][i]) == int(o["stop_turn"][i]), (i, st["stop_turn"][i], o["stop_turn"][i])
        assert bool(st["stopped"][i]) == (gr >= 0)
        assert int(st["rows_seen"][i]) == r1 - r0
        if gr == orr:
            # OPD loss on the retained tokens (Eq. 2, Algorithm 1): a token is
            # retained while the rule has not fired before it -- the
            # trajectory's first token (token mode) or first turn (turn mode)
            # always, no test preceding it; after it, while the oracle's
            # running sum at the previous test is >= lambda.  The sum never
            # rises, so the retained tokens are a prefix.  Tokens whose sum
            # before them lies within TIE_BAND of lambda may be counted
            # either way (the tie-band rule of stop_matches): the count must
            # lie between the prefix retained for certain and the prefix
            # retained at most, the loss must be the certain prefix's plus at
            # most the tie tokens' terms.  Without a tie both are exact.
            before, first = _sum_before(o, lay, mode, i)
            with np.errstate(invalid="ignore"):
                gap = before - lam_a[i]
            # (a NaN lambda never fires: every token retained)
            sure = first | (gap >= TIE_BAND) | bool(np.isnan(lam_a[i]))
            maybe = sure | (gap > -TIE_BAND)
            term = (lp[r0:r1] + d[r0:r1]) * d[r0:r1]
            n_lo, n_hi = int(sure.sum()), int(maybe.sum())
            assert n_lo <= int(o["traj_loss_tokens"][i]) <= n_hi  # the oracle's own count
            assert n_lo <= int(st["loss_tokens"][i]) <= n_hi, ("loss_tokens", i, n_lo, n_hi)
            l_tie = float(np.abs(term[maybe & ~sure]).sum())
            mag = loss_mag(lp[r0:r1] + d[r0:r1], d[r0:r1])
            assert abs(st["loss"][i] - float(term[sure].sum())) <= SUM_RTOL * mag + l_tie, ("loss", i)
            if n_lo == n_hi:
                assert int(st["loss_tokens"][i]) == int(o["traj_loss_tokens"][i]), ("loss_tokens", i)
                assert abs(st["loss"][i] - o["traj_loss"][i]) <= SUM_RTOL * mag, ("loss", i)
    if "profile" in g:
        # within-turn decile profile (Observation 1): counts exact, sums 1e-5 of magnitudes
        gp, op = g["profile"], o["profile"]
        assert np.array_equal(gp[:, 2], op[:, 2]), (gp[:, 2], op[:, 2])
        assert np.all(np.abs(gp[:, 0] - op[:, 0]) <= SUM_RTOL * (np.sum(np.abs(d)) + len(d))), "profile d"
        assert np.all(np.abs(gp[:, 1] - op[:, 1]) <= SUM_RTOL * np.sum(np.abs(lp) + 1.0)), "profile logp_t"


def _sum_before(o, lay, mode, i):
    """The oracle's running sum at the last test before each token of
    trajectory i: the previous token's (TOKEN_SUM) or the previous turn's
    end (TURN_MEAN); and the mask of the tokens no test precedes (the first
    token, or the first turn's tokens), whose entry is 0."""
    base = lay.traj_row_off[0]
    r0, r1 = lay.traj_row_off[i] - base, lay.traj_row_off[i + 1] - base
    if r1 == r0:  # a trajectory without turns
        return np.zeros(0), np.zeros(0, bool)
    if mode == oracle.TOKEN_SUM:
        before = np.concatenate([[0.0], o["row_cum"][r0:r1 - 1]])
        first = np.zeros(r1 - r0, bool)
        first[0] = True
        return before, first
    k0, k1 = lay.traj_turn_off[i], lay.traj_turn_off[i + 1]
    n = np.diff(lay.turn_row_off[k0:k1 + 1])
    prev = np.concatenate([[0.0], o["turn_cum"][k0:k1 - 1]])
    first = np.repeat(np.arange(k1 - k0) == 0, n)
    return np.repeat(prev, n), first


def pad_cols(a: np.ndarray, ld: int, fill) -> np.ndarray:
    out = np.full((a.shape[0], ld), fill, a.dtype)
    out[:, : a.shape[1]] = a
    return out
