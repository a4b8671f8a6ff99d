"""The comparison rule the GPU parity tests apply to retained tokens
(gpu_helpers.compare_scan), checked on the CPU against the oracle's own
results: with the stop indices equal, the retained-token count and the OPD
loss must match the oracle's exactly, except for tokens whose oracle running
sum before them lies within TIE_BAND of lambda (reading 13: at a tie either
side is rounding noise).  A difference confined to tie tokens passes; the
same difference away from a tie, a token more than the tie holds, or a loss
that is not the retained prefix's, fails."""
import numpy as np
import pytest

import oracle
import synth
from gpu_helpers import compare_scan

# turn lengths and per-token log pi_T as binary fractions (every sum exact)
TURNS = [[4, 4, 2], [2, 4, 4]]


def _case(mode, lam_at):
    lay = synth.layout_from_turn_lengths(TURNS)
    R = lay.rows
    rng = np.random.default_rng(7)
    lpt = -rng.integers(1, 9, R).astype(np.float64) * 0.25
    d = rng.integers(-4, 5, R).astype(np.float64) * 0.125
    lps = lpt + d
    o0 = oracle.scan_batch(lpt, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode,
                           np.full(lay.n_traj, -1e30), logp_s=lps)
    # lambda of trajectory 0 equal to its running sum after turn 0 (a tie),
    # of trajectory 1 far below every sum (no stop, no tie)
    lam = np.array([o0["turn_cum"][0] if mode == oracle.TURN_MEAN else o0["row_cum"][lam_at], -1e6], np.float64)
    o = oracle.scan_batch(lpt, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, lam, logp_s=lps)
    o.update(logp_t=lpt, logp_s=lps, d=d)
    return lay, o, lam


def _as_gpu(o, lay):
    """The oracle's results in the layout the GPU path returns."""
    import paper_2609_14636_gb300 as stride

    ts = np.zeros(lay.n_turns, stride.TURN_STATS_DTYPE)
    ts["sum_t"], ts["sum_d"], ts["sum_l"] = o["turn_sum_t"], o["turn_sum_d"], o["turn_sum_l"]
    ts["cum"], ts["mean_t"], ts["n"] = o["turn_cum"], o["turn_mean"], o["turn_n"]
    st = np.zeros(lay.n_traj, stride.STATE_DTYPE)
    st["cum"], st["stop_row"], st["stop_turn"] = o["traj_cum"], o["stop_row"], o["stop_turn"]
    st["stopped"] = o["stop_row"] >= 0
    st["rows_seen"] = np.diff(lay.traj_row_off)
    st["loss"], st["loss_tokens"] = o["traj_loss"], o["traj_loss_tokens"]
    return {"turn_stats": ts, "state": st}


def _drop_rows(g, o, lay, i, rows):
    """Take trajectory-local rows `rows` out of trajectory i's retained set."""
    base = lay.traj_row_off[0]
    r0 = lay.traj_row_off[i] - base
    terms = o["logp_s"][r0:] * o["d"][r0:]
    g["state"]["loss_tokens"][i] -= len(rows)
    g["state"]["loss"][i] -= float(sum(terms[r] for r in rows))


@pytest.mark.parametrize("mode", [oracle.TURN_MEAN, oracle.TOKEN_SUM])
def test_identical_results_pass(mode):
    lay, o, lam = _case(mode, lam_at=3)
    compare_scan(_as_gpu(o, lay), o, lay, mode, lam)


def test_turn_mean_tie_turn_may_be_dropped():
    lay, o, lam = _case(oracle.TURN_MEAN, lam_at=0)
    assert o["stop_row"][0] < 0 or o["stop_turn"][0] > 0  # the tie itself does not stop (strict <)
    g = _as_gpu(o, lay)
    _drop_rows(g, o, lay, 0, range(4, 8))  # turn 1: its sum before is the tie value
    compare_scan(g, o, lay, oracle.TURN_MEAN, lam)


def test_turn_mean_drop_beyond_tie_fails():
    lay, o, lam = _case(oracle.TURN_MEAN, lam_at=0)
    g = _as_gpu(o, lay)
    _drop_rows(g, o, lay, 0, range(3, 8))  # the tie turn and the last token before it
    with pytest.raises(AssertionError):
        compare_scan(g, o, lay, oracle.TURN_MEAN, lam)


def test_turn_mean_loss_must_follow_the_prefix():
    """The count within bounds, but the loss of other tokens than the
    prefix: fails."""
    lay, o, lam = _case(oracle.TURN_MEAN, lam_at=0)
    g = _as_gpu(o, lay)
    terms = o["logp_s"] * o["d"]  # trajectory 0 starts at row 0
    g["state"]["loss"][0] += 10.0 * (abs(terms[:8]).sum() + 1.0)
    with pytest.raises(AssertionError):
        compare_scan(g, o, lay, oracle.TURN_MEAN, lam)


def test_token_sum_tie_token_may_be_dropped():
    lay, o, lam = _case(oracle.TOKEN_SUM, lam_at=2)
    g = _as_gpu(o, lay)
    _drop_rows(g, o, lay, 0, [3])  # token 3: the running sum before it is the tie value
    compare_scan(g, o, lay, oracle.TOKEN_SUM, lam)
    _drop_rows(g, o, lay, 0, [1])  # and one away from the tie: fails
    with pytest.raises(AssertionError):
        compare_scan(g, o, lay, oracle.TOKEN_SUM, lam)


def test_no_tie_trajectory_is_exact():
    lay, o, lam = _case(oracle.TURN_MEAN, lam_at=0)
    g = _as_gpu(o, lay)
    _drop_rows(g, o, lay, 1, [0])
    with pytest.raises(AssertionError):
        compare_scan(g, o, lay, oracle.TURN_MEAN, lam)


@pytest.mark.parametrize("mode", [oracle.TURN_MEAN, oracle.TOKEN_SUM])
def test_first_test_is_always_retained(mode):
    """lambda = +inf: the rule fires at the first test, after the first turn
    (or token), which is retained -- the comparison must demand it."""
    lay = synth.layout_from_turn_lengths(TURNS)
    rng = np.random.default_rng(7)
    R = lay.rows
    lpt = -rng.integers(1, 9, R).astype(np.float64) * 0.25
    d = rng.integers(-4, 5, R).astype(np.float64) * 0.125
    lps = lpt + d
    lam = np.array([np.inf, -np.inf])
    o = oracle.scan_batch(lpt, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, lam, logp_s=lps)
    o.update(logp_t=lpt, logp_s=lps, d=d)
    kept = TURNS[0][0] if mode == oracle.TURN_MEAN else 1
    assert o["traj_loss_tokens"][0] == kept and o["traj_loss_tokens"][1] == sum(TURNS[1])
    compare_scan(_as_gpu(o, lay), o, lay, mode, lam)
    g = _as_gpu(o, lay)
    _drop_rows(g, o, lay, 0, range(kept))
    with pytest.raises(AssertionError):
        compare_scan(g, o, lay, mode, lam)
