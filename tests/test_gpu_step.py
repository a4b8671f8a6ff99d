"""GPU parity of stride_score_step (one decode step over B rollouts) against
the oracle's step rule, over many steps with carried state and masking."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from gpu_helpers import LOGP_ATOL, SUM_RTOL, TIE_BAND, loss_mag, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


def _ring(seed, ring, B, V, ld):
    rng = np.random.default_rng(seed)
    S = synth.bf16_bits_from_f32(rng.standard_normal((ring * B, V), dtype=np.float32) * np.float32(3.0))
    T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + rng.standard_normal((ring * B, V), dtype=np.float32) * np.float32(0.5))
    tok = rng.integers(0, V, ring * B).astype(np.int32)
    Sp = np.zeros((ring * B, ld), np.uint16)
    Tp = np.zeros((ring * B, ld), np.uint16)
    Sp[:, :V], Tp[:, :V] = S, T
    return S, T, tok, Sp, Tp


def run_steps(stride, St, Tt, tk, turn_end, ring, B, mode, lam, V, check_every=None, o_rows=None):
    """Run len(turn_end) steps; step s reads slab s % ring.  Returns the GPU
    and oracle final states and the per-step checks done along the way."""
    import torch

    steps = turn_end.shape[0]
    st = stride.new_state(B)
    ost = oracle.new_rollouts(B)
    te_dev = torch.from_numpy(turn_end).cuda()
    out = {k: torch.empty(B, dtype=torch.float32, device="cuda") for k in ("logp_s", "logp_t", "opd")}
    sn = torch.empty(B, dtype=torch.uint8, device="cuda")
    tout = torch.empty((B, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, device="cuda")
    lam_arg = float(np.float32(lam))
    fired_g = np.zeros((steps, B), np.uint8)
    fired_o = np.zeros((steps, B), np.uint8)
    worst = 0.0
    loss_m = np.zeros(B)        # magnitude of each rollout's loss sum so far
    turn_m = np.zeros(B)        # ... of its open turn's loss sum
    for s in range(steps):
        j = s % ring
        stride.stride_score_step(St[j * B:(j + 1) * B], Tt[j * B:(j + 1) * B], tk[j * B:(j + 1) * B], te_dev[s],
                                 mode, lam_arg, st, out=out, stopped_now=sn, turn_out=tout, V=V)
        ps, pt = o_rows["logp_s"][j * B:(j + 1) * B], o_rows["logp_t"][j * B:(j + 1) * B]
        oo = oracle.step_update(ost, ps, pt, turn_end[s], mode, np.float32(lam))
        fired_o[s] = oo["stopped_now"]
        act_now = ~np.isnan(oo["logp_t"])
        m_now = np.where(act_now, np.abs(ps * (ps - pt)) + np.abs(ps) + np.abs(ps - pt) + 1.0, 0.0)
        loss_m += m_now
        turn_m += m_now
        closed_mag = turn_m.copy()
        turn_m[oo["turn_n"] > 0] = 0.0
        if check_every and (s % check_every == 0 or s == steps - 1):
            torch.cuda.synchronize()
            g_lp = out["logp_t"].cpu().numpy()
            act = ~np.isnan(oo["logp_t"])
            assert np.array_equal(np.isnan(g_lp), ~act)
            if act.any():
                worst = max(worst, float(np.max(np.abs(g_lp[act] - oo["logp_t"][act]))))
            fired_g[s] = sn.cpu().numpy()
            tg = stride.turn_stats_to_numpy(tout)
            closed = oo["turn_n"] > 0
            assert np.array_equal(tg["n"], oo["turn_n"])
            if closed.any():
                assert np.all(np.abs(tg["mean_t"][closed] - oo["turn_mean"][closed]) <= LOGP_ATOL)
                assert np.all(np.abs(tg["sum_l"][closed] - oo["turn_sum_l"][closed]) <= SUM_RTOL * closed_mag[closed])
    torch.cuda.synchronize()
    o = oracle.rollouts_to_numpy(ost)
    o["loss_mag"] = loss_m
    return stride.state_to_numpy(st), o, worst


def _check_final(g, o, mode, lam):
    for b in range(len(g)):
        if g["stop_row"][b] != o["stop_row"][b]:
            # only acceptable inside the tie band around lambda
            assert abs(o["cum"][b] - lam) < TIE_BAND or abs(g["cum"][b] - lam) < TIE_BAND, b
            continue
        assert g["stop_turn"][b] == o["stop_turn"][b]
        assert g["stopped"][b] == (1 if o["stopped"][b] else 0)
        assert g["rows_seen"][b] == o["rows_seen"][b]
        assert g["turn_idx"][b] == o["turn_idx"][b] and g["turn_tokens"][b] == o["turn_tokens"][b]
        assert abs(g["cum"][b] - o["cum"][b]) <= SUM_RTOL * abs(o["cum"][b]) + 1e-12
        assert g["loss_tokens"][b] == g["rows_seen"][b]
        assert abs(g["loss"][b] - o["loss"][b]) <= SUM_RTOL * o["loss_mag"][b]


@pytest.mark.parametrize("mode,lam", [(0, -30.0), (1, -400.0)])
@pytest.mark.parametrize("V,ld", [(4099, 4104), (4099, 4099), (151_936, 151_936)])
def test_steps_small(stride, mode, lam, V, ld):
    ring, B, steps = 3, 24, 160
    S, T, tok, Sp, Tp = _ring(V + ld + mode, ring, B, V, ld)
    o_rows = oracle.row_logprobs(S, T, tok)
    rng = np.random.default_rng(1)
    turn_end = (rng.random((steps, B)) < 1 / 25).astype(np.uint8)
    St, Tt = to_dev(Sp), to_dev(Tp)
    import torch

    tk = torch.from_numpy(tok).cuda()
    g, o, worst = run_steps(stride, St, Tt, tk, turn_end, ring, B, mode, lam, V, check_every=1, o_rows=o_rows)
    assert worst <= LOGP_ATOL
    assert int(o["stopped"].astype(bool).sum()) > 0, "the threshold should stop some rollouts"
    _check_final(g, o, mode, lam)


@pytest.mark.parametrize("B,V,ld", [(1, 4099, 4104), (3, 100, 104), (2, 9, 9), (5, 64, 64), (1500, 40, 40)])
def test_steps_tiny_problems(stride, B, V, ld):
    """One rollout, rows of one vector plus a tail, scalar rows, and more
    rollouts than a wave of clusters holds."""
    import torch

    ring, steps = 2, 40
    S, T, tok, Sp, Tp = _ring(B * 7 + V, ring, B, V, ld)
    o_rows = oracle.row_logprobs(S, T, tok)
    rng = np.random.default_rng(2)
    turn_end = (rng.random((steps, B)) < 1 / 6).astype(np.uint8)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    g, o, worst = run_steps(stride, St, Tt, tk, turn_end, ring, B, 0, -25.0, V, check_every=1, o_rows=o_rows)
    assert worst <= LOGP_ATOL
    _check_final(g, o, 0, -25.0)


def test_step_full_decode_workload(stride):
    """B=256 rollouts x 4,096 steps, V=151,936 bf16, a ring of 16 distinct
    step slabs (more bytes than L2), turn ends every U{96..768} steps, stopped
    rollouts masked; turn-mean and token-sum thresholds."""
    import torch

    w = synth.decode_steps()
    B, ring = w["B"], w["ring"]
    V = w["recipe"].V
    S, T, tok = synth.generate_rows(w["recipe"], 0, ring * B, device="cuda")
    torch.cuda.synchronize()
    Sh = S.view(torch.int16).cpu().numpy().view(np.uint16)
    Th = T.view(torch.int16).cpu().numpy().view(np.uint16)
    o_rows = oracle.row_logprobs(Sh, Th, tok.cpu().numpy())
    for mode, lam in ((0, w["lam_turn"]), (1, w["lam_token"])):
        g, o, worst = run_steps(stride, S, T, tok, w["turn_end"], ring, B, mode, lam, V, check_every=97,
                                o_rows=o_rows)
        assert worst <= LOGP_ATOL
        _check_final(g, o, mode, lam)
        assert int(o["stopped"].astype(bool).sum()) > 0
