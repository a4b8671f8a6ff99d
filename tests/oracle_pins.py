"""Pins for the fp64 oracle: checks against what the paper and the mathematics
fix, independent of the oracle's own code.

Each ``check_*`` takes an ``oracle.OracleLib`` and raises AssertionError on a
mismatch.  tests/test_oracle_pins.py runs them against the oracle;
tests/test_oracle_mutants.py runs them against copies of oracle.c with a
planted mistake and requires that some check fails for each.

Kinds of pin used here:
* closed forms: uniform logits give log pi = -ln V; one hot logit a among V
  gives a - ln(e^a + V - 1) and -ln(e^a + V - 1);
* arbitrary-precision brute force (mpmath, 60 digits, no max-shift) on tiny V;
* a library routine for a special case (torch.log_softmax in float64);
* invariants: sum_y exp(log pi(y)) = 1, shift invariance, logp <= 0,
  monotone running sums, turn-stat totals;
* hand-worked cases of Eq. 5 / Sec. 5.5 / Eq. 6 stored in tests/golden/ with
  their citation and derivation;
* brute-force enumeration of Eq. 6 over all 2^12 masks;
* two independent formulations of one definition: the online step rule
  (Algorithm 1 inner loop) against the batch scan.
"""
from __future__ import annotations

import json
import math
from pathlib import Path

import numpy as np

import oracle
from synth import bf16_bits_from_f32, f32_from_bf16_bits, layout_from_turn_lengths, ragged_layout

GOLD = Path(__file__).resolve().parent / "golden"


def _f(x) -> float:
    if isinstance(x, str):
        return {"-inf": -math.inf, "inf": math.inf, "nan": math.nan}[x]
    return float(x)


# ---------------------------------------------------------------------------
# log-softmax gather (Eq. 1, Eq. 4)
# ---------------------------------------------------------------------------
def check_uniform_closed_form(orc):
    """Uniform logits (any constant c): log pi(y) = -ln V for every y."""
    for V in (1, 7, 8, 33, 32_000, 151_936):
        for c in (0.0, 3.5, -7.25):
            x = np.full((1, V), c, np.float32)
            for S in (x, bf16_bits_from_f32(x)):
                for y in {0, V - 1, V // 2}:
                    o = orc.row_logprobs(S, S, np.array([y], np.int32))
                    want = -math.log(V)
                    assert abs(o["logp_s"][0] - want) <= 1e-12 * max(1.0, abs(want)), (V, c, y, o["logp_s"][0])
                    assert abs(o["lse_s"][0] - (c + math.log(V))) <= 1e-12 * max(1.0, abs(c) + math.log(V))


def check_one_hot_closed_form(orc):
    """One logit a at index h, zeros elsewhere."""
    V, h = 1000, 17
    for a in (5.0, -3.0, 20.0, 0.5):
        x = np.zeros((2, V), np.float32)
        x[:, h] = a
        o = orc.row_logprobs(x, x, np.array([h, 3], np.int32))
        lz = math.log(math.exp(a) + V - 1)
        assert abs(o["logp_s"][0] - (a - lz)) <= 1e-12, (a, o["logp_s"][0], a - lz)
        assert abs(o["logp_s"][1] - (-lz)) <= 1e-12
        assert o["x_s"][0] == a and o["x_s"][1] == 0.0


def check_d_sign_and_operands(orc):
    """d = log pi_S - log pi_T (= -r_t of Eq. 1), with S and T not swapped.

    Student: one-hot a at h; teacher: uniform.  logp_S(h) = a - ln(e^a+V-1),
    logp_T(h) = -ln V."""
    V, h, a = 64, 5, 4.0
    S = np.zeros((1, V), np.float32)
    S[0, h] = a
    T = np.full((1, V), 2.0, np.float32)
    o = orc.row_logprobs(S, T, np.array([h], np.int32))
    ps = a - math.log(math.exp(a) + V - 1)
    pt = -math.log(V)
    assert abs(o["logp_s"][0] - ps) <= 1e-12
    assert abs(o["logp_t"][0] - pt) <= 1e-12
    assert abs(o["d"][0] - (ps - pt)) <= 1e-12
    assert o["x_t"][0] == 2.0 and abs(o["lse_t"][0] - (2.0 + math.log(V))) <= 1e-12


def check_bruteforce_mpmath(orc):
    """Tiny V: log pi(y) = x_y - ln sum_j exp(x_j), evaluated in 60-digit
    arithmetic with no max-shift, including logits far beyond exp's fp64
    range."""
    import mpmath

    mpmath.mp.dps = 60
    rng = np.random.default_rng(11)
    for V in (1, 2, 3, 5, 8, 13, 16):
        for scale in (1.0, 30.0, 800.0):
            x = (rng.standard_normal((1, V)) * scale).astype(np.float32)
            z = mpmath.log(mpmath.fsum(mpmath.e ** mpmath.mpf(float(v)) for v in x[0]))
            for y in range(V):
                o = orc.row_logprobs(x, x, np.array([y], np.int32))
                want = float(mpmath.mpf(float(x[0, y])) - z)
                assert abs(o["logp_s"][0] - want) <= 1e-12 * max(1.0, abs(want)), (V, scale, y)


def check_normalisation(orc):
    """sum_y exp(log pi(y)) = 1, and logp <= 0."""
    rng = np.random.default_rng(12)
    V = 33
    x = (rng.standard_normal((V, V)) * 4).astype(np.float32)
    x[:] = x[0]
    o = orc.row_logprobs(x, x, np.arange(V, dtype=np.int32))
    assert abs(math.fsum(np.exp(o["logp_s"])) - 1.0) <= 1e-12
    assert (o["logp_s"] <= 0).all()


def check_shift_invariance(orc):
    """Adding a bf16-exact constant to every logit leaves log pi unchanged."""
    rng = np.random.default_rng(13)
    V = 300
    # quarter-step grid in [-4, 4]: shifted values keep <= 8 significant bits
    xf = (rng.integers(-16, 17, size=(4, V)) / 4.0).astype(np.float32)
    x = bf16_bits_from_f32(xf)
    assert np.array_equal(f32_from_bf16_bits(x), xf)
    y = rng.integers(0, V, 4).astype(np.int32)
    o0 = orc.row_logprobs(x, x, y)
    for c in (1.0, -8.0):
        xs = bf16_bits_from_f32(xf + np.float32(c))
        assert np.array_equal(f32_from_bf16_bits(xs), xf + np.float32(c)), "shift must be exact"
        o1 = orc.row_logprobs(xs, xs, y)
        assert np.max(np.abs(o1["logp_s"] - o0["logp_s"])) <= 1e-12


def check_torch_log_softmax(orc):
    """Library special case: torch.log_softmax in float64 on the CPU."""
    import torch

    rng = np.random.default_rng(14)
    R, V = 16, 4096
    S = (rng.standard_normal((R, V)) * 5).astype(np.float32)
    T = (S + rng.standard_normal((R, V)) * 0.7).astype(np.float32)
    y = rng.integers(0, V, R).astype(np.int32)
    o = orc.row_logprobs(S, T, y)
    ls = torch.log_softmax(torch.from_numpy(S).double(), dim=1)[torch.arange(R), torch.from_numpy(y).long()]
    lt = torch.log_softmax(torch.from_numpy(T).double(), dim=1)[torch.arange(R), torch.from_numpy(y).long()]
    assert np.max(np.abs(o["logp_s"] - ls.numpy())) <= 1e-12
    assert np.max(np.abs(o["logp_t"] - lt.numpy())) <= 1e-12


def check_teacher_only(orc):
    """S = None scores the teacher alone with the same results."""
    rng = np.random.default_rng(16)
    V = 500
    S = (rng.standard_normal((5, V)) * 3).astype(np.float32)
    T = (rng.standard_normal((5, V)) * 3).astype(np.float32)
    y = rng.integers(0, V, 5).astype(np.int32)
    a = orc.row_logprobs(S, T, y)
    b = orc.row_logprobs(None, T, y)
    assert np.array_equal(a["logp_t"], b["logp_t"]) and np.isnan(b["logp_s"]).all()
    lt = np.array([math.log(math.fsum(math.exp(float(v)) for v in row)) for row in T])
    assert np.max(np.abs(b["logp_t"] - (T[np.arange(5), y] - lt))) <= 1e-12


def check_bf16_decode(orc):
    """bf16 bit patterns decode to the values IEEE-754 fixes."""
    cases = {0x3F80: 1.0, 0xC0A0: -5.0, 0x4049: 3.140625, 0x0001: 2.0 ** -133,
             0x8000: -0.0, 0x7F7F: 3.3895313892515355e38}
    bits = np.array(list(cases), np.uint16)
    vals = np.array(list(cases.values()))
    V = bits.shape[0]
    row = np.tile(bits, (V, 1))
    o = orc.row_logprobs(row, row, np.arange(V, dtype=np.int32))
    assert np.array_equal(o["x_s"], vals), o["x_s"]


def check_special_values(orc):
    """-inf entries carry no mass; an all -inf row has LSE -inf and NaN
    log-probs; NaN logits give NaN; an out-of-range token gives NaN for its
    row and an error code."""
    x = np.full((1, 10), -np.inf, np.float32)
    x[0, [1, 4, 6, 9]] = 0.0
    o = orc.row_logprobs(x, x, np.array([4], np.int32))
    assert abs(o["logp_s"][0] + math.log(4)) <= 1e-12
    o = orc.row_logprobs(x, x, np.array([0], np.int32))
    assert o["logp_s"][0] == -math.inf
    z = np.full((1, 10), -np.inf, np.float32)
    o = orc.row_logprobs(z, z, np.array([2], np.int32))
    assert o["lse_s"][0] == -math.inf and math.isnan(o["logp_s"][0])
    n = np.zeros((1, 10), np.float32)
    n[0, 3] = np.nan
    o = orc.row_logprobs(n, n, np.array([1], np.int32))
    assert math.isnan(o["logp_s"][0])
    g = np.zeros((2, 10), np.float32)
    o = orc.row_logprobs(g, g, np.array([10, 1], np.int32), check=False)
    assert o["rc"] == oracle.ERR_TOKEN and math.isnan(o["logp_s"][0]) and not math.isnan(o["logp_s"][1])
    o = orc.row_logprobs(g, g, np.array([-1, 1], np.int32), check=False)
    assert o["rc"] == oracle.ERR_TOKEN and math.isnan(o["logp_t"][0])


def check_strided_rows(orc):
    """ld > V: padding columns are never read."""
    rng = np.random.default_rng(15)
    V, ld = 100, 128
    x = (rng.standard_normal((3, ld)) * 3).astype(np.float32)
    y = np.array([0, 50, 99], np.int32)
    o0 = orc.row_logprobs(np.ascontiguousarray(x[:, :V]), np.ascontiguousarray(x[:, :V]), y)
    x[:, V:] = 1e30
    o1 = orc.row_logprobs(x, x, y, V=V)
    assert np.array_equal(o0["logp_s"], o1["logp_s"])


# ---------------------------------------------------------------------------
# turn means and stop rule (Eq. 4, Eq. 5, Sec. 4.1 offset, Sec. 5.5)
# ---------------------------------------------------------------------------
def _golden_stop_cases():
    return json.loads((GOLD / "stop_rule_cases.json").read_text())["cases"]


def _case_turns(c):
    if "turns_repeat" in c:
        return [[c["turns_repeat"]["value"]] * c["turns_repeat"]["count"]]
    return c["turns"]


def check_stop_rule_golden(orc):
    for c in _golden_stop_cases():
        turns = _case_turns(c)
        lay = layout_from_turn_lengths([[len(t) for t in turns]])
        lp = np.array([v for t in turns for v in t], np.float64)
        mode = oracle.TURN_MEAN if c["mode"] == "turn_mean" else oracle.TOKEN_SUM
        cin = None if "cum_in" not in c else np.array([c["cum_in"]])
        o = orc.scan_batch(lp, np.zeros_like(lp), lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                           mode, float(c["lambda"]), cum_in=cin)  # "nan" / "inf" stored as strings
        assert list(o["turn_mean"]) == c["turn_mean"], (c["name"], o["turn_mean"])
        assert list(o["turn_cum"]) == c["turn_cum"], (c["name"], o["turn_cum"])
        assert int(o["stop_turn"][0]) == c["stop_turn"], (c["name"], o["stop_turn"])
        assert int(o["stop_row"][0]) == c["stop_row"], (c["name"], o["stop_row"])


def _loss_cases():
    return json.loads((GOLD / "opd_loss_cases.json").read_text())


def check_opd_loss_golden(orc):
    """Retained-token OPD loss (Eq. 2, Algorithm 1) on hand-worked cases."""
    for c in _loss_cases()["cases"]:
        lay = layout_from_turn_lengths([[len(t) for t in c["turns"]]])
        rows = np.array([r for t in c["turns"] for r in t], np.float64)
        ls, lt = rows[:, 0], rows[:, 1]
        mode = oracle.TURN_MEAN if c["mode"] == "turn_mean" else oracle.TOKEN_SUM
        cin = None if "cum_in" not in c else np.array([c["cum_in"]])
        o = orc.scan_batch(lt, ls - lt, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode,
                           float(c["lambda"]), cum_in=cin, logp_s=ls)
        assert list(o["turn_sum_l"]) == c["turn_sum_l"], (c["name"], o["turn_sum_l"])
        assert o["traj_loss"][0] == c["loss"], (c["name"], o["traj_loss"])
        assert int(o["traj_loss_tokens"][0]) == c["loss_tokens"], c["name"]
        assert int(o["stop_turn"][0]) == c["stop_turn"], c["name"]


def check_turn_profile_golden(orc):
    """Within-turn decile profile (Observation 1) on a hand-worked case."""
    pc = _loss_cases()["profile_case"]
    lay = layout_from_turn_lengths([pc["turn_lengths"]])
    d = np.concatenate([np.arange(20.0), [100.0, 200.0, 300.0]])
    lt = np.concatenate([np.full(20, -1.0), np.full(3, -4.0)])
    o = orc.scan_batch(lt, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, oracle.TURN_MEAN, -1e300)
    assert np.array_equal(o["profile"], np.array(pc["profile"])), o["profile"]


def check_loss_invariants(orc):
    """Loss over all tokens when the rule never fires; in turn mode the
    retained loss is the sum of turn sums up to the stopping turn; in token
    mode the sum of terms up to the stopping token; profile counts sum to the
    rows and its d column to the sum of d."""
    for seed in range(4):
        lay, lp, d = _random_scan_data(400 + seed)
        ls = lp + d
        terms = ls * d
        for mode, lam in ((oracle.TURN_MEAN, -4.0), (oracle.TOKEN_SUM, -30.0)):
            never = orc.scan_batch(lp, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, -1e300,
                                   logp_s=ls)
            o = orc.scan_batch(lp, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, lam, logp_s=ls)
            assert int(o["profile"][:, 2].sum()) == lay.rows
            assert abs(o["profile"][:, 0].sum() - math.fsum(d)) <= 1e-9 * math.fsum(np.abs(d))
            for i in range(lay.n_traj):
                r0, r1 = lay.traj_row_off[i], lay.traj_row_off[i + 1]
                k0, k1 = lay.traj_turn_off[i], lay.traj_turn_off[i + 1]
                assert abs(never["traj_loss"][i] - math.fsum(terms[r0:r1])) <= 1e-9 * (1 + math.fsum(np.abs(terms[r0:r1])))
                assert never["traj_loss_tokens"][i] == r1 - r0
                if o["stop_row"][i] < 0:
                    assert o["traj_loss_tokens"][i] == r1 - r0
                    continue
                if mode == oracle.TURN_MEAN:
                    kk = k0 + int(o["stop_turn"][i])
                    want = math.fsum(o["turn_sum_l"][k0:kk + 1])
                    n = int(lay.turn_row_off[kk + 1] - r0)
                else:
                    n = int(o["stop_row"][i]) + 1
                    want = math.fsum(terms[r0:r0 + n])
                assert o["traj_loss_tokens"][i] == n
                assert abs(o["traj_loss"][i] - want) <= 1e-9 * (1 + abs(want))


def check_prefix_buffer_offset(orc):
    """Scanning only the new turns after K0 reused turns (Sec. 4.1) differs
    from scanning the whole record, as the golden derivation states."""
    c = next(c for c in _golden_stop_cases() if c["name"] == "prefix_buffer_new_turns_only")
    rec = c["record_means"]
    lay = layout_from_turn_lengths([[1] * len(rec)])
    o = orc.scan_batch(np.array(rec), None, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                       oracle.TURN_MEAN, c["lambda"])
    assert int(o["stop_turn"][0]) == 3
    new = rec[c["K0"]:]
    lay2 = layout_from_turn_lengths([[1] * len(new)])
    o2 = orc.scan_batch(np.array(new), None, lay2.traj_row_off, lay2.turn_row_off, lay2.traj_turn_off,
                        oracle.TURN_MEAN, c["lambda"])
    assert int(o2["stop_turn"][0]) == c["stop_turn"] and c["K0"] + int(o2["stop_turn"][0]) == 4


def _random_scan_data(seed, n_traj=7, turns=(1, 9), lo=1, hi=40):
    rng = np.random.default_rng(seed)
    lay = ragged_layout(rng, n_traj, turns, lo, hi)
    lp = -rng.exponential(1.5, lay.rows)
    d = rng.standard_normal(lay.rows)
    return lay, lp, d


def check_scan_invariants(orc):
    """Turn totals, means, monotone running sums, first crossing = count of
    non-crossed test positions (brute-force linear scan)."""
    for seed in range(5):
        lay, lp, d = _random_scan_data(100 + seed)
        for mode, lam in ((oracle.TURN_MEAN, -4.0), (oracle.TOKEN_SUM, -30.0)):
            o = orc.scan_batch(lp, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, lam)
            assert int(o["turn_n"].sum()) == lay.rows
            assert abs(math.fsum(o["turn_sum_t"]) - math.fsum(lp)) <= 1e-9 * math.fsum(np.abs(lp))
            assert abs(math.fsum(o["turn_sum_d"]) - math.fsum(d)) <= 1e-9 * math.fsum(np.abs(d))
            assert np.allclose(o["turn_mean"] * o["turn_n"], o["turn_sum_t"], rtol=1e-12, atol=0)
            for i in range(lay.n_traj):
                a, b = lay.traj_turn_off[i], lay.traj_turn_off[i + 1]
                tc = o["turn_cum"][a:b]
                assert (np.diff(tc) <= 0).all()
                if mode == oracle.TURN_MEAN:
                    # brute force: walk the turns, adding each turn's mean
                    s, first = 0.0, -1
                    for j, k in enumerate(range(a, b)):
                        r0, r1 = lay.turn_row_off[k], lay.turn_row_off[k + 1]
                        s += math.fsum(lp[r0:r1]) / (r1 - r0)
                        if first < 0 and s < lam:
                            first = j
                    assert int(o["stop_turn"][i]) == first
                    if first >= 0:
                        assert int(o["stop_row"][i]) == lay.turn_row_off[a + first + 1] - 1 - lay.traj_row_off[i]
                else:
                    r0, r1 = lay.traj_row_off[i], lay.traj_row_off[i + 1]
                    rc = o["row_cum"][r0:r1]
                    assert (np.diff(rc) <= 0).all()
                    nonx = int((rc >= lam).sum())  # monotone: non-crossed rows form a prefix
                    want = nonx if nonx < (r1 - r0) else -1
                    assert int(o["stop_row"][i]) == want


def check_traj_independence(orc):
    """Each trajectory's result depends only on its own rows."""
    lay, lp, d = _random_scan_data(200, n_traj=5)
    for mode, lam in ((oracle.TURN_MEAN, -3.0), (oracle.TOKEN_SUM, -25.0)):
        o = orc.scan_batch(lp, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, lam)
        for i in range(lay.n_traj):
            r0, r1 = lay.traj_row_off[i], lay.traj_row_off[i + 1]
            k0, k1 = lay.traj_turn_off[i], lay.traj_turn_off[i + 1]
            sub = layout_from_turn_lengths([list(np.diff(lay.turn_row_off[k0:k1 + 1]))])
            oi = orc.scan_batch(lp[r0:r1], d[r0:r1], sub.traj_row_off, sub.turn_row_off, sub.traj_turn_off,
                                mode, lam)
            assert oi["stop_turn"][0] == o["stop_turn"][i] and oi["stop_row"][0] == o["stop_row"][i]
            assert np.array_equal(oi["turn_cum"], o["turn_cum"][k0:k1])


def check_per_trajectory_lambda(orc):
    lay = layout_from_turn_lengths([[1, 1], [1, 1]])
    lp = np.array([-1.0, -1.0, -1.0, -1.0])
    o = orc.scan_batch(lp, None, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, oracle.TURN_MEAN,
                       np.array([-1.5, -2.5]))
    assert list(o["stop_turn"]) == [1, -1]


def check_empty_turn_rejected(orc):
    lay = layout_from_turn_lengths([[2, 0, 1]])
    try:
        orc.scan_batch(np.zeros(3), None, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                       oracle.TURN_MEAN, -1.0)
    except ValueError:
        return
    raise AssertionError("an empty turn must be rejected")


# ---------------------------------------------------------------------------
# online step rule (Algorithm 1 inner loop) against the batch scan
# ---------------------------------------------------------------------------
def _run_steps(orc, lay, lp, d, mode, lam):
    B = lay.n_traj
    lens = np.diff(lay.traj_row_off)
    st = orc.new_rollouts(B)
    row_turn = lay.row_turn()
    turn_last = np.zeros(lay.rows, np.uint8)
    turn_last[lay.turn_row_off[1:] - 1] = 1
    outs = []
    for s in range(int(lens.max())):
        ps = np.zeros(B)
        pt = np.zeros(B)
        te = np.zeros(B, np.uint8)
        for b in range(B):
            if s < lens[b]:
                r = lay.traj_row_off[b] + s
                ps[b], pt[b], te[b] = lp[r] + d[r], lp[r], turn_last[r]
        # rollouts past their end are marked stopped-by-length for the oracle
        for b in range(B):
            if s == lens[b]:
                st[b].stopped = max(st[b].stopped, 2)
        outs.append(orc.step_update(st, ps, pt, te, mode, lam))
    return st, outs, row_turn


def check_step_matches_batch(orc):
    for seed in range(3):
        lay, lp, d = _random_scan_data(300 + seed, n_traj=6)
        for mode, lam in ((oracle.TURN_MEAN, -4.0), (oracle.TOKEN_SUM, -30.0)):
            ob = orc.scan_batch(lp, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, lam)
            obl = orc.scan_batch(lp, d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode, lam,
                                 logp_s=lp + d)
            st, outs, _ = _run_steps(orc, lay, lp, d, mode, lam)
            for b in range(lay.n_traj):
                # every token a rollout scores is retained: its loss is the batch retained loss
                assert abs(st[b].loss - obl["traj_loss"][b]) <= 1e-9 * (1 + abs(obl["traj_loss"][b])), (seed, mode, b)
                assert st[b].rows_seen == obl["traj_loss_tokens"][b] or st[b].stop_row < 0
                assert st[b].stop_turn == ob["stop_turn"][b], (seed, mode, b)
                assert st[b].stop_row == ob["stop_row"][b], (seed, mode, b)
                if st[b].stop_row >= 0:
                    # nothing is scored after the stop
                    assert st[b].rows_seen == st[b].stop_row + 1
                    k0 = lay.traj_turn_off[b]
                    if mode == oracle.TURN_MEAN:
                        assert abs(st[b].cum - ob["turn_cum"][k0 + st[b].stop_turn]) <= 1e-12 * abs(st[b].cum)
                else:
                    assert abs(st[b].cum - ob["traj_cum"][b]) <= 1e-12 * max(1.0, abs(st[b].cum))
            # closed-turn stats reported at turn ends equal the batch turn stats
            for s, o in enumerate(outs):
                for b in range(lay.n_traj):
                    if o["turn_n"][b] > 0:
                        k = lay.row_turn()[lay.traj_row_off[b] + s]
                        assert o["turn_n"][b] == ob["turn_n"][k]
                        assert abs(o["turn_mean"][b] - ob["turn_mean"][k]) <= 1e-12 * abs(ob["turn_mean"][k]) + 1e-300


def check_step_golden(orc):
    for c in _golden_stop_cases():
        turns = _case_turns(c)
        if "cum_in" in c:
            continue
        lay = layout_from_turn_lengths([[len(t) for t in turns]])
        lp = np.array([v for t in turns for v in t], np.float64)
        mode = oracle.TURN_MEAN if c["mode"] == "turn_mean" else oracle.TOKEN_SUM
        st, _, _ = _run_steps(orc, lay, lp, np.zeros_like(lp), mode, float(c["lambda"]))
        assert st[0].stop_turn == c["stop_turn"] and st[0].stop_row == c["stop_row"], c["name"]


# ---------------------------------------------------------------------------
# restart choice (Sec. 4.2, Eq. 6, Algorithm 1)
# ---------------------------------------------------------------------------
def check_select_golden(orc):
    cases = json.loads((GOLD / "select_cases.json").read_text())["cases"]
    for c in cases:
        means = np.array([[_f(v) for v in c["means"]]], np.float32)
        T_max = means.shape[1]
        nt = np.array([c.get("n_turns", T_max)], np.int32)
        mask = None if c["mask"] is None else np.array([c["mask"]], np.uint8)
        ks, km = orc.select_restart(means, nt, mask, _f(c["alpha"]))
        assert int(km[0]) == c["k_max"] and int(ks[0]) == c["k_star"], (c["name"], ks, km)


def check_select_bruteforce(orc):
    """All 2^12 masks, values from a small set (forcing ties), several alphas:
    K_max = max{K : every turn before K is correct}, k* = lowest index of the
    minimum over the first K_max turns, both by enumeration."""
    rng = np.random.default_rng(21)
    T = 12
    masks = ((np.arange(1 << T)[:, None] >> np.arange(T)[None, :]) & 1).astype(np.uint8)
    vals = np.array([-0.5, -0.75, -1.0, -0.25], np.float32)
    means = vals[rng.integers(0, 4, size=(masks.shape[0], T))]
    nt = rng.integers(0, T + 1, size=masks.shape[0]).astype(np.int32)
    for alpha in (-math.inf, -0.8, -0.6):
        ks, km = orc.select_restart(means, nt, masks, alpha)
        for i in range(masks.shape[0]):
            corr = [bool(masks[i, k]) and bool(means[i, k] > np.float32(alpha)) for k in range(nt[i])]
            K = max([K for K in range(nt[i] + 1) if all(corr[:K])])
            kstar = min(range(K), key=lambda k: (means[i, k], k)) if K > 0 else 0
            assert km[i] == K and ks[i] == kstar, (i, alpha)


def check_prefix_buffer_golden(orc):
    """Algorithm 1's record of {l_k} in H(x) with the reused prefix kept, and
    the restart choice before and after (hand-worked cases)."""
    cases = json.loads((GOLD / "prefix_buffer_cases.json").read_text())["cases"]
    for c in cases:
        T_max = c["T_max"]
        mean = np.full((1, T_max), np.float32(123.0), np.float32)
        n = np.array([len(c["stored"])], np.int32)
        mean[0, :len(c["stored"])] = c["stored"]
        ks, km = orc.select_restart(mean, n, None, _f(c["alpha"]))
        assert (int(km[0]), int(ks[0])) == (c["select_before"]["k_max"], c["select_before"]["k_star"]), c["name"]
        new = np.array(c["new_turn_means"], np.float32)
        orc.buffer_record(mean, n, [0], ks, new, [0, len(new)])
        assert int(n[0]) == len(c["record_after"]), c["name"]
        assert list(mean[0, :n[0]]) == c["record_after"], (c["name"], mean[0, :n[0]])
        ks, km = orc.select_restart(mean, n, None, _f(c["alpha"]))
        assert (int(km[0]), int(ks[0])) == (c["select_after"]["k_max"], c["select_after"]["k_star"]), c["name"]


def check_prefix_buffer_properties(orc):
    """Random records: the kept prefix is unchanged, the new means follow it,
    k0 beyond the stored length is clamped, other tasks are untouched."""
    rng = np.random.default_rng(31)
    n_tasks, T_max = 40, 9
    mean = rng.standard_normal((n_tasks, T_max)).astype(np.float32)
    n = rng.integers(0, T_max + 1, n_tasks).astype(np.int32)
    before_m, before_n = mean.copy(), n.copy()
    tasks = rng.permutation(n_tasks)[:25].astype(np.int32)
    k0 = rng.integers(0, T_max + 3, 25).astype(np.int32)
    lens = rng.integers(0, 7, 25)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    tm = rng.standard_normal(int(off[-1])).astype(np.float32)
    orc.buffer_record(mean, n, tasks, k0, tm, off)
    for j, x in enumerate(tasks):
        keep = min(int(k0[j]), int(before_n[x]))
        want = np.concatenate([before_m[x, :keep], tm[off[j]:off[j + 1]]])[:T_max]
        assert int(n[x]) == len(want)
        assert np.array_equal(mean[x, :n[x]], want)
    others = np.setdiff1d(np.arange(n_tasks), tasks)
    assert np.array_equal(mean[others], before_m[others]) and np.array_equal(n[others], before_n[others])


ALL_CHECKS = [
    check_uniform_closed_form, check_one_hot_closed_form, check_d_sign_and_operands,
    check_bruteforce_mpmath, check_normalisation, check_shift_invariance, check_torch_log_softmax,
    check_teacher_only, check_bf16_decode, check_special_values, check_strided_rows,
    check_stop_rule_golden, check_prefix_buffer_offset, check_scan_invariants,
    check_traj_independence, check_per_trajectory_lambda, check_empty_turn_rejected,
    check_opd_loss_golden, check_turn_profile_golden, check_loss_invariants,
    check_step_matches_batch, check_step_golden,
    check_select_golden, check_select_bruteforce,
    check_prefix_buffer_golden, check_prefix_buffer_properties,
]
