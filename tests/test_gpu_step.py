"""GPU parity of the decode step (stride_score_step, and the compacted form
stride_score_step_compact) against the oracle's step rule, over many steps
with carried state, masking and first crossings.

Every output is compared at every step: the per-row log-probs and d (2e-3
absolute), the stop flag of the step (bit-exact, except where the oracle's
running sum at that test position lies within 1e-3 of lambda), and the stats
of every closed turn (n exact; l_k 2e-3; the sums 1e-5 of the summed
magnitudes; the running sum 1e-5 relative).  At the end the carried state is
compared, with the stop index under the batch path's rule: the two may
differ only where the oracle's running sum lies within 1e-3 of lambda at
every test position between them.  The running sums at positions past a stop
come from a second oracle rollout set that never stops (lambda = -inf), so
the rule can be checked on either side of a stop."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from gpu_helpers import LOGP_ATOL, SUM_RTOL, TIE_BAND, stop_matches, to_dev

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


def run_steps(stride, St, Tt, tk, turn_end, ring, B, mode, lam, V, o_rows, form="masked", cum0=None):
    """Run len(turn_end) steps; step s reads slab s % ring (rollout b's row is
    row b of the slab).  form = "masked": stride_score_step over all B rows;
    "compact": stride_score_step_compact over the rows of the rollouts that
    have not stopped, gathered from the slab as a rollout engine that
    batches only live sequences would hand them over (the live set is the
    GPU's own, from stopped_now).  lam: a scalar or a float32 array [B].
    cum0: optional starting running sums [B] (a carried offset), set in the
    GPU state and in the oracle's.  Returns a summary of the run."""
    import torch

    steps = turn_end.shape[0]
    lam32 = np.asarray(lam, np.float32)
    lam64 = np.broadcast_to(lam32.astype(np.float64), (B,))
    lam_arg = torch.from_numpy(np.array(np.broadcast_to(lam32, (B,)))).cuda() if lam32.ndim else float(lam32)
    st = stride.new_state(B)
    ost, shadow = oracle.new_rollouts(B), oracle.new_rollouts(B)
    ov, sv = oracle.rollouts_view(ost), oracle.rollouts_view(shadow)
    if cum0 is not None:
        h = stride.state_to_numpy(st)[:B].copy()
        h["cum"] = cum0
        st[:B].copy_(torch.from_numpy(h.view(np.uint8).reshape(B, -1)).cuda())
        ov["cum"][:] = cum0
        sv["cum"][:] = cum0
    out = {k: torch.empty(B, dtype=torch.float32, device="cuda") for k in ("logp_s", "logp_t", "opd")}
    sn = torch.empty(B, dtype=torch.uint8, device="cuda")
    tout = torch.empty((B, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    g_stopped = np.zeros(B, bool)
    diverged = np.zeros(B, bool)
    rc = np.empty((steps, B))             # never-stopping oracle's running sum after each step
    tests = np.ones((steps, B), bool) if mode == oracle.TOKEN_SUM else turn_end.astype(bool)
    mag_t, mag_d, mag_l, loss_m = (np.zeros(B) for _ in range(4))
    worst = 0.0
    rows_scored = 0
    for s in range(steps):
        j = s % ring
        ps, pt = o_rows["logp_s"][j * B:(j + 1) * B], o_rows["logp_t"][j * B:(j + 1) * B]
        live_o = ov["stopped"] == 0
        oo = oracle.step_update(ost, ps, pt, turn_end[s], mode, lam64)
        oracle.step_update(shadow, ps, pt, turn_end[s], mode, -np.inf)
        rc[s] = sv["cum"]

        Sj, Tj, kj = St[j * B:(j + 1) * B], Tt[j * B:(j + 1) * B], tk[j * B:(j + 1) * B]
        g_lp = {k: np.full(B, np.nan, np.float32) for k in out}
        g_fired = np.zeros(B, np.uint8)
        g_ts = np.zeros(B, stride.TURN_STATS_DTYPE)
        if form == "masked":
            te = torch.from_numpy(np.ascontiguousarray(turn_end[s])).cuda()
            stride.stride_score_step(Sj, Tj, kj, te, mode, lam_arg, st, out=out, stopped_now=sn, turn_out=tout,
                                     dev_status=status, V=V)
            for k in out:
                g_lp[k] = out[k].cpu().numpy()
            g_fired = sn.cpu().numpy()
            g_ts = stride.turn_stats_to_numpy(tout)
            # a rollout stopped on the GPU is masked: NaN, no flag, no turn
            assert np.isnan(g_lp["logp_t"][g_stopped]).all() and not g_fired[g_stopped].any()
            assert not g_ts["n"][g_stopped].any()
            rows_scored += int((~g_stopped).sum())
        else:
            idx = np.nonzero(~g_stopped)[0].astype(np.int32)
            n = idx.shape[0]
            if n:
                it = torch.from_numpy(idx).cuda()
                te = torch.from_numpy(np.ascontiguousarray(turn_end[s][idx])).cuda()
                stride.stride_score_step_compact(Sj.index_select(0, it), Tj.index_select(0, it), kj.index_select(0, it),
                                                 te, it, mode, lam_arg, st, out=out, stopped_now=sn, turn_out=tout,
                                                 dev_status=status, V=V)
                for k in out:
                    g_lp[k][idx] = out[k][:n].cpu().numpy()
                g_fired[idx] = sn[:n].cpu().numpy()
                g_ts[idx] = stride.turn_stats_to_numpy(tout)[:n]
            rows_scored += n

        cmp = live_o & ~g_stopped & ~diverged
        # per-row log-probs and d
        for k, ok in (("logp_s", "logp_s"), ("logp_t", "logp_t"), ("opd", "d")):
            a, b = g_lp[k][cmp].astype(np.float64), oo[ok][cmp]
            fin = np.isfinite(b)
            assert np.array_equal(np.isfinite(a), fin), (s, k)
            if fin.any():
                err = float(np.max(np.abs(a[fin] - b[fin])))
                assert err <= LOGP_ATOL, (s, k, err)
                worst = max(worst, err)
        # open-turn magnitudes the turn sums are compared against
        d = ps - pt
        mag_t[cmp] += np.abs(pt[cmp]) + 1.0
        mag_d[cmp] += np.abs(d[cmp]) + 1.0
        m_l = np.abs(ps * d) + np.abs(ps) + np.abs(d) + 1.0
        mag_l[cmp] += m_l[cmp]
        loss_m[cmp] += m_l[cmp]
        # the stats of every closed turn
        assert np.array_equal(g_ts["n"][cmp], oo["turn_n"][cmp]), s
        closed = cmp & (oo["turn_n"] > 0)
        if closed.any():
            assert np.all(np.abs(g_ts["mean_t"][closed] - oo["turn_mean"][closed]) <= LOGP_ATOL), s
            assert np.all(np.abs(g_ts["sum_t"][closed] - oo["turn_sum_t"][closed]) <= SUM_RTOL * mag_t[closed]), s
            assert np.all(np.abs(g_ts["sum_d"][closed] - oo["turn_sum_d"][closed]) <= SUM_RTOL * mag_d[closed]), s
            assert np.all(np.abs(g_ts["sum_l"][closed] - oo["turn_sum_l"][closed]) <= SUM_RTOL * mag_l[closed]), s
            assert np.all(np.abs(g_ts["cum"][closed] - oo["turn_cum"][closed])
                          <= SUM_RTOL * np.abs(oo["turn_cum"][closed]) + 1e-12), s
        ends = oo["turn_n"] > 0
        mag_t[ends] = mag_d[ends] = mag_l[ends] = 0.0
        # the stop flag of this step
        differ = cmp & (g_fired != oo["stopped_now"])
        for r in np.nonzero(differ)[0]:
            assert tests[s, r] and abs(rc[s, r] - lam64[r]) < TIE_BAND, ("stop flag", s, r, rc[s, r])
            diverged[r] = True
        g_stopped |= g_fired.astype(bool)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    g = stride.state_to_numpy(st)
    o = oracle.rollouts_to_numpy(ost)
    for r in range(B):
        gr, orr = int(g["stop_row"][r]), int(o["stop_row"][r])
        assert stop_matches(gr, orr, rc[:, r], list(np.nonzero(tests[:, r])[0]), lam64[r]), (r, gr, orr)
        assert bool(g["stopped"][r]) == (gr >= 0)
        if gr != orr:
            continue
        assert g["stop_turn"][r] == o["stop_turn"][r], r
        assert g["rows_seen"][r] == o["rows_seen"][r], r
        assert g["turn_idx"][r] == o["turn_idx"][r] and g["turn_tokens"][r] == o["turn_tokens"][r], r
        assert abs(g["cum"][r] - o["cum"][r]) <= SUM_RTOL * abs(o["cum"][r]) + 1e-12, r
        assert g["loss_tokens"][r] == g["rows_seen"][r]
        assert abs(g["loss"][r] - o["loss"][r]) <= SUM_RTOL * loss_m[r], r
    assert int(g["rows_seen"].sum()) == rows_scored
    return {"worst": worst, "stopped": int(o["stopped"].astype(bool).sum()), "diverged": int(diverged.sum()),
            "rows": rows_scored}


@pytest.mark.parametrize("form", ["masked", "compact"])
@pytest.mark.parametrize("mode,lam", [(0, -30.0), (1, -400.0)])
@pytest.mark.parametrize("V,ld", [(4099, 4104), (4099, 4099), (151_936, 151_936)])
def test_steps_small(stride, mode, lam, V, ld, form):
    import torch

    ring, B, steps = 3, 24, 160
    S, T, tok, Sp, Tp = _ring(V + ld + mode, ring, B, V, ld)
    o_rows = oracle.row_logprobs(S, T, tok)
    rng = np.random.default_rng(1)
    turn_end = (rng.random((steps, B)) < 1 / 25).astype(np.uint8)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    r = run_steps(stride, St, Tt, tk, turn_end, ring, B, mode, lam, V, o_rows, form=form)
    assert r["stopped"] > 0, "the threshold should stop some rollouts"


def test_steps_compact_per_rollout_lambda(stride):
    """Per-rollout thresholds in the compacted form: lambda, like the state,
    is read through the rollout index, not the row."""
    import torch

    ring, B, steps, V = 3, 40, 200, 4099
    S, T, tok, Sp, Tp = _ring(77, ring, B, V, V)
    o_rows = oracle.row_logprobs(S, T, tok)
    rng = np.random.default_rng(5)
    turn_end = (rng.random((steps, B)) < 1 / 20).astype(np.uint8)
    lam = (-30.0 + rng.uniform(-12.0, 12.0, B)).astype(np.float32)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    r = run_steps(stride, St, Tt, tk, turn_end, ring, B, 0, lam, V, o_rows, form="compact")
    assert 0 < r["stopped"] < B


@pytest.mark.parametrize("form", ["masked", "compact"])
@pytest.mark.parametrize("closes", ["every_token", "never"])
def test_steps_turn_end_extremes(stride, form, closes):
    """Every token closes its own turn (each step tests, turn means are
    single log-probs), or no turn ever closes (turn mode never tests, so
    nothing stops and every token is retained)."""
    import torch

    ring, B, steps, V = 3, 16, 120, 4099
    S, T, tok, Sp, Tp = _ring(79, ring, B, V, V)
    o_rows = oracle.row_logprobs(S, T, tok)
    turn_end = np.full((steps, B), 1 if closes == "every_token" else 0, np.uint8)
    # even rollouts: half their final never-stopping sum (they stop midway
    # when tests happen); odd rollouts: out of reach
    pre = oracle.new_rollouts(B)
    for s in range(steps):
        j = s % ring
        oracle.step_update(pre, o_rows["logp_s"][j * B:(j + 1) * B], o_rows["logp_t"][j * B:(j + 1) * B],
                           np.ones(B, np.uint8), 0, np.full(B, -np.inf))
    lam = np.where(np.arange(B) % 2 == 0, 0.5 * oracle.rollouts_view(pre)["cum"], -1e6).astype(np.float32)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    r = run_steps(stride, St, Tt, tk, turn_end, ring, B, 0, lam, V, o_rows, form=form)
    if closes == "never":
        assert r["stopped"] == 0 and r["rows"] == steps * B
    else:
        assert r["stopped"] == B // 2


@pytest.mark.parametrize("form", ["masked", "compact"])
@pytest.mark.parametrize("seed", list(range(6)))
def test_steps_mixed_degenerate(stride, form, seed):
    """Seeded decode runs mixing per-rollout lambda finite, +inf, -inf and
    NaN, carried starting sums (some already below lambda: those stop at
    their first test), random turn ends, both modes."""
    import torch

    rng = np.random.default_rng(300 + seed)
    ring, B, steps = 3, int(rng.integers(5, 40)), int(rng.integers(40, 160))
    V = int(rng.choice([257, 4099]))
    mode = int(rng.integers(0, 2))
    S, T, tok, Sp, Tp = _ring(400 + seed, ring, B, V, V)
    o_rows = oracle.row_logprobs(S, T, tok)
    turn_end = (rng.random((steps, B)) < rng.uniform(0.02, 0.3)).astype(np.uint8)
    scale = -4.0 * steps if mode == oracle.TOKEN_SUM else -4.0 * max(1.0, turn_end.sum(0).mean())
    lam = (scale * rng.uniform(0.2, 1.0, B)).astype(np.float32)
    u = rng.random(B)
    lam[u < 0.15] = np.float32(np.inf)
    lam[(u >= 0.15) & (u < 0.3)] = np.float32(-np.inf)
    lam[(u >= 0.3) & (u < 0.45)] = np.float32(np.nan)
    cum0 = np.where(rng.random(B) < 0.3, rng.uniform(1.5, 3.0, B) * np.where(np.isfinite(lam), lam, -10.0), 0.0)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    run_steps(stride, St, Tt, tk, turn_end, ring, B, mode, lam, V, o_rows, form=form, cum0=cum0)


@pytest.mark.parametrize("form", ["masked", "compact"])
def test_steps_nan_thresholds_never_fire(stride, form):
    """A NaN entry of the per-rollout lambda never fires (the test is
    strict): that rollout never stops and every token it scores is
    retained, beside rollouts with finite thresholds that stop as usual."""
    import torch

    ring, B, steps, V = 3, 24, 160, 4099
    S, T, tok, Sp, Tp = _ring(78, ring, B, V, V)
    o_rows = oracle.row_logprobs(S, T, tok)
    rng = np.random.default_rng(6)
    turn_end = (rng.random((steps, B)) < 1 / 16).astype(np.uint8)
    lam = (-24.0 + rng.uniform(-8.0, 8.0, B)).astype(np.float32)
    lam[::3] = np.float32(np.nan)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    r = run_steps(stride, St, Tt, tk, turn_end, ring, B, 0, lam, V, o_rows, form=form)
    assert 0 < r["stopped"] <= B - len(lam[::3])


@pytest.mark.parametrize("threads,C", [(128, 1), (128, 2), (128, 3), (128, 5), (128, 8), (128, 12), (128, 16),
                                       (512, 1), (512, 3), (512, 8), (512, 16)])
def test_steps_every_launch_shape(stride, threads, C):
    """The same step rule whatever CTA size and number of CTAs a row is split
    over (stride_force_step_shape), ragged slices and a tail included."""
    import torch

    ring, B, steps, V = 2, 12, 60, 4099
    S, T, tok, Sp, Tp = _ring(C + threads, ring, B, V, V)
    o_rows = oracle.row_logprobs(S, T, tok)
    rng = np.random.default_rng(C + threads)
    turn_end = (rng.random((steps, B)) < 1 / 8).astype(np.uint8)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    stride.stride_force_step_shape(threads, C)
    try:
        for form in ("masked", "compact"):
            run_steps(stride, St, Tt, tk, turn_end, ring, B, 0, -20.0, V, o_rows, form=form)
    finally:
        stride.stride_force_step_shape(0, 0)


@pytest.mark.parametrize("B,V,ld", [(1, 4099, 4104), (3, 100, 104), (2, 9, 9), (5, 64, 64), (1500, 40, 40)])
@pytest.mark.parametrize("form", ["masked", "compact"])
def test_steps_tiny_problems(stride, B, V, ld, form):
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
    run_steps(stride, St, Tt, tk, turn_end, ring, B, 0, -25.0, V, o_rows, form=form)


def test_compact_edge_cases(stride):
    """No rows; a rollout index out of range; a row of a rollout that has
    already stopped; a missing index array."""
    import torch

    B, V = 6, 4099
    S, T, tok, Sp, Tp = _ring(3, 1, B, V, V)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    st = stride.new_state(B)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = {k: torch.zeros(B, dtype=torch.float32, device="cuda") for k in ("logp_s", "logp_t", "opd")}
    sn = torch.full((B,), 7, dtype=torch.uint8, device="cuda")
    te1 = torch.ones(B, dtype=torch.uint8, device="cuda")
    before = stride.state_to_numpy(st)
    # no rows: nothing launched, nothing changed
    stride.stride_score_step_compact(St, Tt, tk, te1, torch.empty(0, dtype=torch.int32, device="cuda"), 0, -1.0, st,
                                     out=out, stopped_now=sn, dev_status=status)
    torch.cuda.synchronize()
    assert np.array_equal(stride.state_to_numpy(st), before) and int(status.item()) == 0
    assert (sn.cpu().numpy() == 7).all()
    # rollout 1 stops at once (lambda above any running sum); an index of 9 is out of range
    idx = torch.tensor([1, 9, 4], dtype=torch.int32, device="cuda")
    stride.stride_score_step_compact(St, Tt, tk, te1, idx, 0, float("inf"), st, out=out, stopped_now=sn,
                                     dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 2  # STRIDE_DEV_BAD_LAYOUT
    lp = out["logp_t"].cpu().numpy()
    o = oracle.row_logprobs(S, T, tok)
    assert abs(lp[0] - o["logp_t"][0]) <= LOGP_ATOL and np.isnan(lp[1]) and abs(lp[2] - o["logp_t"][2]) <= LOGP_ATOL
    assert list(sn.cpu().numpy()[:3]) == [1, 0, 1]
    g = stride.state_to_numpy(st)
    assert list(g["rows_seen"]) == [0, 1, 0, 0, 1, 0] and list(g["stopped"]) == [0, 1, 0, 0, 1, 0]
    # rollout 1 again: read, not scored; its state stays as it was
    stride.stride_score_step_compact(St, Tt, tk, te1, torch.tensor([1], dtype=torch.int32, device="cuda"), 0,
                                     float("inf"), st, out=out, stopped_now=sn)
    torch.cuda.synchronize()
    assert np.isnan(out["logp_t"][0].item()) and int(sn[0].item()) == 0
    assert np.array_equal(stride.state_to_numpy(st), g)
    # a missing index array with rows to score is an argument error
    rc = stride.lib().stride_score_step_compact(St.data_ptr(), Tt.data_ptr(), 0, V, V, tk.data_ptr(), te1.data_ptr(),
                                                None, 2, B, 0, None, -1.0, st.data_ptr(), None, None, None, None, None)
    assert rc == 1


@pytest.mark.parametrize("form", ["masked", "compact"])
def test_step_full_decode_workload(stride, form):
    """B=256 rollouts x 4,096 steps, V=151,936 bf16, a ring of 16 distinct
    step slabs (more bytes than L2), turn ends every U{96..768} steps;
    stopped rollouts masked, or left out of the compacted steps; every step
    checked, turn-mean and token-sum thresholds."""
    import torch

    w = synth.decode_steps()
    B, ring = w["B"], w["ring"]
    V = w["recipe"].V
    S, T, tok = synth.generate_rows(w["recipe"], 0, ring * B, device="cuda")
    torch.cuda.synchronize()
    Sh = S.view(torch.int16).cpu().numpy().view(np.uint16)
    Th = T.view(torch.int16).cpu().numpy().view(np.uint16)
    o_rows = oracle.row_logprobs(Sh, Th, tok.cpu().numpy())
    del Sh, Th
    for mode, lam in ((0, w["lam_turn"]), (1, w["lam_token"])):
        r = run_steps(stride, S, T, tok, w["turn_end"], ring, B, mode, lam, V, o_rows, form=form)
        assert r["stopped"] > 0
        assert r["rows"] < B * w["turn_end"].shape[0]


@pytest.mark.parametrize("threads,C", [(128, 4), (128, 12), (512, 8)])
def test_compact_equals_masked_bitwise(stride, threads, C):
    """With the launch shape fixed, the compacted form computes each live
    row exactly as the masked form does (same slices, same merge order, same
    state arithmetic): outputs and carried state bit-identical over a run in
    which rollouts stop."""
    import torch

    ring, B, steps, V = 3, 48, 120, 8192
    S, T, tok, Sp, Tp = _ring(31 + C, ring, B, V, V)
    rng = np.random.default_rng(C)
    turn_end = (rng.random((steps, B)) < 1 / 10).astype(np.uint8)
    St, Tt = to_dev(Sp), to_dev(Tp)
    tk = torch.from_numpy(tok).cuda()
    st_m, st_c = stride.new_state(B), stride.new_state(B)
    keys = ("logp_s", "logp_t", "opd", "lse_s", "lse_t")
    om = {k: torch.empty(B, dtype=torch.float32, device="cuda") for k in keys}
    oc = {k: torch.empty(B, dtype=torch.float32, device="cuda") for k in keys}
    sn_m = torch.empty(B, dtype=torch.uint8, device="cuda")
    sn_c = torch.empty(B, dtype=torch.uint8, device="cuda")
    tm = torch.empty((B, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, device="cuda")
    tc = torch.empty((B, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, device="cuda")
    stopped = np.zeros(B, bool)
    n_stops = 0
    stride.stride_force_step_shape(threads, C)
    try:
        for s in range(steps):
            j = s % ring
            Sj, Tj, kj = St[j * B:(j + 1) * B], Tt[j * B:(j + 1) * B], tk[j * B:(j + 1) * B]
            te = torch.from_numpy(np.ascontiguousarray(turn_end[s])).cuda()
            stride.stride_score_step(Sj, Tj, kj, te, 0, -25.0, st_m, out=om, stopped_now=sn_m, turn_out=tm)
            idx = np.nonzero(~stopped)[0].astype(np.int32)
            n = idx.shape[0]
            if n == 0:
                break
            it = torch.from_numpy(idx).cuda()
            stride.stride_score_step_compact(Sj.index_select(0, it), Tj.index_select(0, it), kj.index_select(0, it),
                                             te.index_select(0, it.long()), it, 0, -25.0, st_c, out=oc,
                                             stopped_now=sn_c, turn_out=tc)
            torch.cuda.synchronize()
            for k in keys:
                a = om[k].cpu().numpy()[idx].view(np.uint32)
                b = oc[k][:n].cpu().numpy().view(np.uint32)
                assert np.array_equal(a, b), (s, k)
            assert np.array_equal(sn_m.cpu().numpy()[idx], sn_c[:n].cpu().numpy()), s
            assert np.array_equal(tm.cpu().numpy()[idx], tc[:n].cpu().numpy()), s
            fired = sn_m.cpu().numpy().astype(bool)
            n_stops += int(fired.sum())
            stopped |= fired
    finally:
        stride.stride_force_step_shape(0, 0)
    assert np.array_equal(stride.state_to_numpy(st_m).view(np.uint8), stride.state_to_numpy(st_c).view(np.uint8))
    assert n_stops > 0


@pytest.mark.parametrize("form", ["masked", "compact"])
def test_step_non_finite_logits(stride, form):
    """One step over rows with a NaN logit, a +inf logit (off and at the
    token) and a row of -inf: log-probs NaN exactly where the oracle's are,
    the clean rows untouched, no trap."""
    import torch

    rng = np.random.default_rng(91)
    B, V = 6, 999
    S32 = rng.standard_normal((B, V), dtype=np.float32) * np.float32(2.0)
    T32 = S32 + rng.standard_normal((B, V), dtype=np.float32)
    tok = rng.integers(0, V, B).astype(np.int32)
    S32[0, 3 if tok[0] != 3 else 4] = np.nan
    T32[1, 9 if tok[1] != 9 else 10] = np.inf
    T32[2, tok[2]] = np.inf
    S32[3, :] = -np.inf
    S, T = synth.bf16_bits_from_f32(S32), synth.bf16_bits_from_f32(T32)
    o = oracle.row_logprobs(S, T, tok)
    St, Tt = to_dev(S), to_dev(T)
    tk = torch.from_numpy(tok).cuda()
    st = stride.new_state(B)
    out = {k: torch.full((B,), 7.0, dtype=torch.float32, device="cuda") for k in ("logp_s", "logp_t", "opd")}
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    te = torch.zeros(B, dtype=torch.uint8, device="cuda")
    if form == "masked":
        stride.stride_score_step(St, Tt, tk, te, 1, -1e30, st, out=out, dev_status=status)
    else:
        idx = torch.arange(B, dtype=torch.int32, device="cuda")
        stride.stride_score_step_compact(St, Tt, tk, te, idx, 1, -1e30, st, out=out, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    for k, ok in (("logp_s", "logp_s"), ("logp_t", "logp_t"), ("opd", "d")):
        a, b = out[k].cpu().numpy().astype(np.float64), o[ok]
        fin = np.isfinite(b)
        assert np.array_equal(np.isfinite(a), fin), (k, a, b)
        assert np.all(np.abs(a[fin] - b[fin]) <= LOGP_ATOL), k
    assert np.isfinite(o["logp_t"][4:]).all() and np.isfinite(o["logp_s"][4:]).all()
