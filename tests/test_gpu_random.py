"""Randomised GPU parity of the batch path: seeded random ragged layouts
(one-row turns and trajectories included), vocabulary sizes, logit dtypes,
row strides (aligned or not), stop modes, per-trajectory thresholds placed
between the oracle's running sums, and row windows cut at random places,
through the automatic kernel choice and each forced batch kernel; every row,
turn and trajectory against the oracle under the tolerances of
gpu_helpers.  And the scan alone (stride_scan_logprobs) on random layouts of
thousands of rows -- many 256-row tiles, lookbacks across them, seeded rows
inside tiles -- fed the same fp32 log-probs as the oracle's scan."""
from __future__ import annotations

import numpy as np
import pytest

import synth
from gpu_helpers import compare_rows, compare_scan, oracle_batch, pad_cols, run_batch

pytestmark = pytest.mark.gpu

SEEDS = list(range(40))
VOCABS = (257, 1000, 4099, 8192, 32_000)


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


def _case(seed):
    rng = np.random.default_rng(1000 + seed)
    n_traj = int(rng.integers(1, 7))
    lens = []
    for _ in range(n_traj):
        nt = int(rng.integers(1, 6))
        lens.append([1 if rng.random() < 0.25 else int(rng.integers(2, 121)) for _ in range(nt)])
    lay = synth.layout_from_turn_lengths(lens)
    R = lay.rows
    V = int(rng.choice(VOCABS))
    while R * V > 12_000_000 and V > VOCABS[0]:
        V = max(v for v in VOCABS if v < V)
    f32 = bool(rng.random() < 0.4)
    ld = V + (int(rng.integers(1, 10)) if rng.random() < 0.4 else 0)
    mode = int(rng.integers(0, 2))
    sigma = float(rng.uniform(1.0, 5.0))
    S32 = rng.standard_normal((R, V), dtype=np.float32) * np.float32(sigma)
    T32 = S32 + rng.standard_normal((R, V), dtype=np.float32) * np.float32(rng.uniform(0.2, 2.0))
    if f32:
        S, T = S32, T32.astype(np.float32)
        fill = np.float32(np.nan)
    else:
        S = synth.bf16_bits_from_f32(S32)
        T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + (T32 - S32))
        fill = 0x7FC0  # NaN padding: never read
    tok = rng.integers(0, V, R).astype(np.int32)
    n_cuts = int(rng.integers(0, 4))
    cuts = sorted(set([0, R] + [int(x) for x in rng.integers(1, R, size=n_cuts)] if R > 1 else [0, R]))
    windows = list(zip(cuts[:-1], cuts[1:]))
    return lay, S, T, tok, V, ld, mode, windows, fill, rng


def _lambda(o, lay, mode, rng):
    """Per-trajectory thresholds halfway between two of the oracle's
    consecutive test values (or below all of them), so that about half the
    trajectories stop, none inside the tie band."""
    lam = np.empty(lay.n_traj, np.float32)
    for i in range(lay.n_traj):
        if mode == 1:
            r0, r1 = lay.traj_row_off[i], lay.traj_row_off[i + 1]
            vals = o["row_cum"][r0:r1]
        else:
            vals = o["turn_cum"][lay.traj_turn_off[i]:lay.traj_turn_off[i + 1]]
        if len(vals) == 0:  # a trajectory without turns: nothing to test
            lam[i] = np.float32(-1e6)
            continue
        if rng.random() < 0.5 or len(vals) == 1:
            lam[i] = np.float32(vals[-1] - 1.0)  # never crosses
        else:
            t = int(rng.integers(1, len(vals)))
            lam[i] = np.float32(0.5 * (vals[t - 1] + vals[t]))
    return lam


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("seed", SEEDS)
def test_random_layouts(stride, seed, kernel):
    lay, S, T, tok, V, ld, mode, windows, fill, rng = _case(seed)
    o0 = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
    lam = _lambda(o0, lay, mode, rng)
    o = oracle_batch(S, T, tok, lay, mode, lam)
    Sp, Tp = (S, T) if ld == V else (pad_cols(S, ld, fill), pad_cols(T, ld, fill))
    stride.stride_force_batch_kernel(kernel)
    try:
        g = run_batch(stride, Sp, Tp, tok, lay, mode, lam, windows=windows, V=V)
    finally:
        stride.stride_force_batch_kernel("auto")
    assert g["status"] == 0
    compare_rows(g, o)
    compare_scan(g, o, lay, mode, lam)


@pytest.mark.parametrize("seed", list(range(12)))
def test_random_scan_on_logprobs(stride, seed):
    import torch

    import oracle

    rng = np.random.default_rng(5000 + seed)
    n_traj = int(rng.integers(1, 40))
    lens = []
    for _ in range(n_traj):
        nt = int(rng.integers(1, 12))
        lens.append([1 if rng.random() < 0.2 else int(rng.integers(2, 700)) for _ in range(nt)])
    lay = synth.layout_from_turn_lengths(lens)
    R = lay.rows
    mode = int(rng.integers(0, 2))
    # log-probs as the scan receives them (fp32, <= 0)
    lpt = (-np.abs(rng.standard_normal(R)) * rng.uniform(1.0, 8.0)).astype(np.float32)
    lps = (lpt + rng.standard_normal(R).astype(np.float32) * np.float32(0.7)).astype(np.float32)
    lps = np.minimum(lps, np.float32(0.0))
    d = (lps.astype(np.float64) - lpt.astype(np.float64))
    o0 = oracle.scan_batch(lpt.astype(np.float64), d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                           mode, np.float64(-1e30), logp_s=lps.astype(np.float64))
    o0.update(logp_t=lpt.astype(np.float64), d=d)
    lam = _lambda(o0, lay, mode, rng)
    o = oracle.scan_batch(lpt.astype(np.float64), d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                          mode, lam.astype(np.float64), logp_s=lps.astype(np.float64))
    o.update(logp_t=lpt.astype(np.float64), logp_s=lps.astype(np.float64), d=d)
    dev = "cuda"
    offs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(lay.n_traj)
    ts = stride.new_turn_stats(lay.n_turns)
    prof = stride.new_profile(dev)
    opd = torch.empty(R, dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    n_cuts = int(rng.integers(0, 4))
    cuts = sorted(set([0, R] + [int(x) for x in rng.integers(1, R, size=n_cuts)]))
    ws = torch.empty(stride.stride_score_batch_workspace_size(R), dtype=torch.uint8, device=dev)
    lps_d, lpt_d = torch.from_numpy(lps).to(dev), torch.from_numpy(lpt).to(dev)
    for a, b in zip(cuts[:-1], cuts[1:]):
        stride.stride_scan_logprobs(lps_d[a:b], lpt_d[a:b], *offs, a, b, mode, torch.from_numpy(lam).to(dev), st,
                                    opd=opd[a:b], turn_stats=ts, dev_status=status, workspace=ws, profile=prof)
    torch.cuda.synchronize()
    g = {"opd": opd.cpu().numpy(), "state": stride.state_to_numpy(st)[: lay.n_traj],
         "turn_stats": stride.turn_stats_to_numpy(ts)[: lay.n_turns], "profile": prof.cpu().numpy()}
    assert int(status.item()) == 0
    assert np.max(np.abs(g["opd"] - d)) <= 2e-3
    compare_scan(g, o, lay, mode, lam)


def _window_layout(rng, total, first):
    """Turn lengths summing to `total` rows: a first trajectory of about
    `first` rows (several turns), then trajectories of 1-5 turns of 1-200
    rows (one-row turns among them)."""
    lens, used = [], 0
    while used < total:
        goal = first if not lens else int(rng.integers(1, 600))
        traj, n = [], 0
        while n < goal and used + n < total and len(traj) < (40 if not lens else 5):
            t = 1 if rng.random() < 0.2 else int(rng.integers(2, 201))
            t = min(t, goal - n, total - used - n)
            traj.append(max(t, 1))
            n += traj[-1]
        lens.append(traj)
        used += n
    return synth.layout_from_turn_lengths(lens)


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("rows", [1, 128, 129, 1024, 1025, 1152, 2047, 2048, 2049])
def test_small_window_scan_every_cluster_size(stride, rows, mode):
    """The scan after the small-window kernel at each size class of its
    launch: windows of 1-16 tiles of 128 rows (one cluster, sizes above 8
    non-portable) and of 17 tiles (the lookback form); a first trajectory
    that runs through the whole first window into the second (its state
    carried into the second window's first tiles, every tile folding all
    its predecessors' aggregates), short trajectories and one-row turns
    after it; two windows of `rows` rows, every row, turn and trajectory
    against the oracle."""
    rng = np.random.default_rng(9000 + 2 * rows + mode)
    lay = _window_layout(rng, 2 * rows, first=max(1, (13 * rows) // 10))
    R = lay.rows
    assert R == 2 * rows
    V = 257
    S = rng.standard_normal((R, V), dtype=np.float32) * np.float32(3.0)
    T = S + rng.standard_normal((R, V), dtype=np.float32)
    tok = rng.integers(0, V, R).astype(np.int32)
    o0 = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
    lam = _lambda(o0, lay, mode, rng)
    o = oracle_batch(S, T, tok, lay, mode, lam)
    stride.stride_force_batch_kernel("split")
    try:
        g = run_batch(stride, S, T, tok, lay, mode, lam, windows=[(0, rows), (rows, R)], V=V)
    finally:
        stride.stride_force_batch_kernel("auto")
    assert g["status"] == 0
    compare_rows(g, o)
    compare_scan(g, o, lay, mode, lam)


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("lam", [float("inf"), float("-inf")])
def test_infinite_thresholds(stride, kernel, mode, lam):
    """lambda = +inf: every trajectory stops at its first test (its first
    turn's end, or its first token) and keeps exactly that turn or token;
    lambda = -inf: none stops and every token is retained -- in one window
    and in three windows with the carried state."""
    rng = np.random.default_rng(777 + mode)
    lens = [[1 if rng.random() < 0.2 else int(rng.integers(2, 90)) for _ in range(int(rng.integers(1, 5)))]
            for _ in range(6)]
    lay = synth.layout_from_turn_lengths(lens)
    R, V = lay.rows, 1000
    S = rng.standard_normal((R, V), dtype=np.float32) * np.float32(2.0)
    T = S + rng.standard_normal((R, V), dtype=np.float32)
    tok = rng.integers(0, V, R).astype(np.int32)
    o = oracle_batch(S, T, tok, lay, mode, np.float32(lam))
    # the definitions' answer, independent of the oracle
    first = np.diff(lay.turn_row_off)[lay.traj_turn_off[:-1]]
    if lam > 0:
        want_row = np.zeros(lay.n_traj, np.int64) if mode == 1 else first - 1
        assert np.array_equal(o["stop_row"], want_row) and np.all(o["stop_turn"] == 0)
        assert np.array_equal(o["traj_loss_tokens"], want_row + 1)
    else:
        assert np.all(o["stop_row"] == -1)
        assert np.array_equal(o["traj_loss_tokens"], np.diff(lay.traj_row_off))
    cuts = [0, R // 3, (2 * R) // 3, R]
    stride.stride_force_batch_kernel(kernel)
    try:
        for windows in (None, list(zip(cuts[:-1], cuts[1:]))):
            g = run_batch(stride, S, T, tok, lay, mode, np.float32(lam), windows=windows, V=V)
            assert g["status"] == 0
            compare_rows(g, o)
            compare_scan(g, o, lay, mode, np.float32(lam))
            assert np.array_equal(g["state"]["stop_row"], o["stop_row"])
            assert np.array_equal(g["state"]["loss_tokens"], o["traj_loss_tokens"])
    finally:
        stride.stride_force_batch_kernel("auto")


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("mode", [0, 1])
def test_nan_thresholds_never_fire(stride, kernel, mode):
    """A NaN entry of the per-trajectory lambda array never fires (the test
    is strict, sum < lambda): its trajectory never stops and keeps every
    token, while the finite entries beside it stop as usual."""
    rng = np.random.default_rng(991 + mode)
    lens = [[int(rng.integers(2, 60)) for _ in range(int(rng.integers(2, 6)))] for _ in range(8)]
    lay = synth.layout_from_turn_lengths(lens)
    R, V = lay.rows, 1000
    S = rng.standard_normal((R, V), dtype=np.float32) * np.float32(2.0)
    T = S + rng.standard_normal((R, V), dtype=np.float32)
    tok = rng.integers(0, V, R).astype(np.int32)
    o0 = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
    lam = _lambda(o0, lay, mode, rng)
    lam[::2] = np.float32(np.nan)
    o = oracle_batch(S, T, tok, lay, mode, lam)
    assert np.all(o["stop_row"][::2] == -1)
    assert np.array_equal(o["traj_loss_tokens"][::2], np.diff(lay.traj_row_off)[::2])
    stride.stride_force_batch_kernel(kernel)
    try:
        for windows in (None, [(0, R // 2), (R // 2, R)]):
            g = run_batch(stride, S, T, tok, lay, mode, lam, windows=windows, V=V)
            assert g["status"] == 0
            compare_rows(g, o)
            compare_scan(g, o, lay, mode, lam)
            assert np.array_equal(g["state"]["loss_tokens"][::2], np.diff(lay.traj_row_off)[::2])
    finally:
        stride.stride_force_batch_kernel("auto")


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("mode", [0, 1])
def test_starting_sums_below_and_above_lambda(stride, kernel, mode):
    """Running sums that start from a carried offset (the prefix-buffer
    restart, Sec. 4.1, expressed through the state's cum): where the offset
    is already below lambda the first test fires and the first turn (or
    token) is retained; elsewhere the rule runs as usual -- against the
    oracle given the same starting sums."""
    import torch

    import oracle

    rng = np.random.default_rng(515 + mode)
    lens = [[int(rng.integers(2, 50)) for _ in range(int(rng.integers(2, 6)))] for _ in range(8)]
    lay = synth.layout_from_turn_lengths(lens)
    R, V = lay.rows, 1000
    S = rng.standard_normal((R, V), dtype=np.float32) * np.float32(2.0)
    T = S + rng.standard_normal((R, V), dtype=np.float32)
    tok = rng.integers(0, V, R).astype(np.int32)
    lam = np.float32(-40.0 if mode == 0 else -300.0)
    cum0 = np.where(np.arange(lay.n_traj) % 2 == 0, float(lam) - 5.0, 0.0)  # even: below lambda already
    o = oracle_batch(S, T, tok, lay, mode, lam)
    sc = oracle.scan_batch(o["logp_t"], o["d"], lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode,
                           np.float64(lam), cum_in=cum0, logp_s=o["logp_s"])
    o.update(sc)
    first = np.diff(lay.turn_row_off)[lay.traj_turn_off[:-1]]
    want_row = np.zeros(lay.n_traj, np.int64) if mode == 1 else first - 1
    assert np.array_equal(o["stop_row"][::2], want_row[::2])
    assert np.array_equal(o["traj_loss_tokens"][::2], want_row[::2] + 1)

    def seeded():
        st = stride.new_state(lay.n_traj)
        h = stride.state_to_numpy(st)[: lay.n_traj].copy()
        h["cum"] = cum0
        st[: lay.n_traj].copy_(torch.from_numpy(h.view(np.uint8).reshape(lay.n_traj, -1)).cuda())
        return st

    stride.stride_force_batch_kernel(kernel)
    try:
        for windows in (None, [(0, R // 2), (R // 2, R)]):
            g = run_batch(stride, S, T, tok, lay, mode, lam, windows=windows, V=V, state=seeded())
            assert g["status"] == 0
            compare_scan(g, o, lay, mode, lam)
            assert np.array_equal(g["state"]["stop_row"][::2], want_row[::2])
            assert np.array_equal(g["state"]["loss_tokens"][::2], want_row[::2] + 1)
    finally:
        stride.stride_force_batch_kernel("auto")


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("mode", [0, 1])
def test_trajectories_without_turns(stride, kernel, mode):
    """Trajectories with no turns (no rows) among the others -- at the start,
    between, at the end, and a run of 300 of them (more than one tile of the
    tiled scan stages) -- are left as initialised, and the rows around them
    are scored as if they were not there."""
    rng = np.random.default_rng(808 + mode)
    lens = [[], []]
    for k in range(10):
        lens.append([1 if rng.random() < 0.2 else int(rng.integers(2, 70)) for _ in range(int(rng.integers(1, 5)))])
        lens.extend([[]] * (300 if k == 4 else int(rng.integers(0, 3))))
    lens.extend([[], []])
    lay = synth.layout_from_turn_lengths(lens)
    R, V = lay.rows, 1000
    S = rng.standard_normal((R, V), dtype=np.float32) * np.float32(2.0)
    T = S + rng.standard_normal((R, V), dtype=np.float32)
    tok = rng.integers(0, V, R).astype(np.int32)
    o0 = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
    lam = _lambda(o0, lay, mode, np.random.default_rng(9))
    o = oracle_batch(S, T, tok, lay, mode, lam)
    empty = np.diff(lay.traj_row_off) == 0
    stride.stride_force_batch_kernel(kernel)
    try:
        for windows in (None, [(0, R // 3), (R // 3, R)]):
            g = run_batch(stride, S, T, tok, lay, mode, lam, windows=windows, V=V)
            assert g["status"] == 0
            compare_rows(g, o)
            compare_scan(g, o, lay, mode, lam)
            st = g["state"]
            assert np.all(st["stop_row"][empty] == -1) and np.all(st["rows_seen"][empty] == 0)
            assert np.all(st["cum"][empty] == 0.0) and np.all(st["loss_tokens"][empty] == 0)
    finally:
        stride.stride_force_batch_kernel("auto")


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("width", [1, 2, 3])
def test_tiny_windows(stride, kernel, width):
    """Windows of 1-3 rows: nearly every turn, and every trajectory but the
    shortest, crosses window edges, so the running sum and the open turn's
    sums go through the carried state at almost every row."""
    rng = np.random.default_rng(31 + width)
    lens = [[1 if rng.random() < 0.25 else int(rng.integers(2, 9)) for _ in range(int(rng.integers(1, 4)))]
            for _ in range(5)]
    lay = synth.layout_from_turn_lengths(lens)
    R, V = lay.rows, 300
    S = rng.standard_normal((R, V), dtype=np.float32) * np.float32(2.0)
    T = S + rng.standard_normal((R, V), dtype=np.float32)
    tok = rng.integers(0, V, R).astype(np.int32)
    for mode in (0, 1):
        o0 = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
        lam = _lambda(o0, lay, mode, np.random.default_rng(3))
        o = oracle_batch(S, T, tok, lay, mode, lam)
        windows = [(a, min(R, a + width)) for a in range(0, R, width)]
        stride.stride_force_batch_kernel(kernel)
        try:
            g = run_batch(stride, S, T, tok, lay, mode, lam, windows=windows, V=V)
        finally:
            stride.stride_force_batch_kernel("auto")
        assert g["status"] == 0
        compare_rows(g, o)
        compare_scan(g, o, lay, mode, lam)


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("f32", [False, True])
def test_non_finite_logits(stride, kernel, f32):
    """A NaN logit, a +inf logit (off the token, and at the token), and a row
    of -inf logits: the row's log-probs are NaN (LSE NaN, or -inf with a -inf
    gathered logit) exactly where the oracle's are, on both sides of the
    pair; the other rows are untouched.  Kernels never trap on them."""
    rng = np.random.default_rng(606 + f32)
    lay = synth.layout_from_turn_lengths([[6, 5], [7], [4, 4, 4]])
    R, V = lay.rows, 1000
    S32 = rng.standard_normal((R, V), dtype=np.float32) * np.float32(2.0)
    T32 = S32 + rng.standard_normal((R, V), dtype=np.float32)
    tok = rng.integers(0, V, R).astype(np.int32)
    S32[1, 5 if tok[1] != 5 else 6] = np.nan       # NaN in S, off the token
    T32[3, 7 if tok[3] != 7 else 8] = np.inf       # +inf in T, off the token
    T32[9, tok[9]] = np.inf                        # +inf at the token
    S32[12, :] = -np.inf                           # a fully masked row
    S32[20, 0] = np.nan
    T32[20, 1] = np.inf                            # both sides
    if f32:
        S, T = S32, T32
    else:
        S, T = synth.bf16_bits_from_f32(S32), synth.bf16_bits_from_f32(T32)
    o = oracle_batch(S, T, tok, lay, 1, np.float32(-1e30))
    bad = [1, 3, 9, 12, 20]
    for r in bad:
        assert not (np.isfinite(o["logp_s"][r]) and np.isfinite(o["logp_t"][r])), r
    good = np.setdiff1d(np.arange(R), bad)
    assert np.isfinite(o["logp_s"][good]).all() and np.isfinite(o["logp_t"][good]).all()
    stride.stride_force_batch_kernel(kernel)
    try:
        g = run_batch(stride, S, T, tok, lay, 1, np.float32(-1e30), V=V)
    finally:
        stride.stride_force_batch_kernel("auto")
    assert g["status"] == 0
    compare_rows(g, o)


def _mixed_case(seed):
    """A layout mixing the degenerate cases: empty trajectories, one-row
    turns and long turns; per-trajectory lambda finite, +inf, -inf or NaN;
    starting sums 0 or carried (some below lambda); random window cuts;
    both dtypes, padded or exact strides."""
    rng = np.random.default_rng(20_000 + seed)
    lens = []
    for _ in range(int(rng.integers(3, 12))):
        u = rng.random()
        if u < 0.15:
            lens.append([])
        else:
            lens.append([1 if rng.random() < 0.25 else int(rng.integers(2, 400 if u < 0.3 else 60))
                         for _ in range(int(rng.integers(1, 6)))])
    if all(len(t) == 0 for t in lens):
        lens.append([int(rng.integers(1, 30))])
    lay = synth.layout_from_turn_lengths(lens)
    R = lay.rows
    V = int(rng.choice([129, 1000, 4099]))
    f32 = bool(rng.random() < 0.5)
    ld = V + (int(rng.integers(1, 9)) if rng.random() < 0.4 else 0)
    mode = int(rng.integers(0, 2))
    S32 = rng.standard_normal((R, V), dtype=np.float32) * np.float32(rng.uniform(1.0, 4.0))
    T32 = S32 + rng.standard_normal((R, V), dtype=np.float32) * np.float32(rng.uniform(0.2, 1.5))
    if f32:
        S, T, fill = S32, T32, np.float32(np.nan)
    else:
        S = synth.bf16_bits_from_f32(S32)
        T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + (T32 - S32))
        fill = 0x7FC0
    tok = rng.integers(0, V, R).astype(np.int32)
    cuts = sorted(set([0, R] + [int(x) for x in rng.integers(1, R, size=int(rng.integers(0, 5)))])) if R > 1 else [0, R]
    return rng, lay, S, T, tok, V, ld, mode, list(zip(cuts[:-1], cuts[1:])), fill


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
@pytest.mark.parametrize("seed", list(range(24)))
def test_mixed_degenerate_layouts(stride, seed, kernel):
    import torch

    import oracle

    rng, lay, S, T, tok, V, ld, mode, windows, fill = _mixed_case(seed)
    o0 = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
    lam = _lambda(o0, lay, mode, rng)
    special = rng.random(lay.n_traj)
    lam[special < 0.1] = np.float32(np.inf)
    lam[(special >= 0.1) & (special < 0.2)] = np.float32(-np.inf)
    lam[(special >= 0.2) & (special < 0.3)] = np.float32(np.nan)
    cum0 = np.where(rng.random(lay.n_traj) < 0.3, rng.uniform(-80.0, 0.0, lay.n_traj), 0.0)
    o = oracle_batch(S, T, tok, lay, mode, lam)
    o.update(oracle.scan_batch(o["logp_t"], o["d"], lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode,
                               lam.astype(np.float64), cum_in=cum0, logp_s=o["logp_s"]))
    st = stride.new_state(lay.n_traj)
    h = stride.state_to_numpy(st)[: lay.n_traj].copy()
    h["cum"] = cum0
    st[: lay.n_traj].copy_(torch.from_numpy(h.view(np.uint8).reshape(lay.n_traj, -1)).cuda())
    Sp, Tp = (S, T) if ld == V else (pad_cols(S, ld, fill), pad_cols(T, ld, fill))
    stride.stride_force_batch_kernel(kernel)
    try:
        g = run_batch(stride, Sp, Tp, tok, lay, mode, lam, windows=windows, V=V, state=st)
    finally:
        stride.stride_force_batch_kernel("auto")
    assert g["status"] == 0
    compare_rows(g, o)
    compare_scan(g, o, lay, mode, lam)


@pytest.mark.parametrize("seed", list(range(24)))
def test_mixed_degenerate_scan_on_logprobs(stride, seed):
    """The mixed layouts through stride_scan_logprobs (the tiled scan on its
    own: 256-row tiles by ticket, one lookback per tile), fed the oracle's
    log-probs rounded to fp32, with the same thresholds and starting sums."""
    import torch

    import oracle

    rng, lay, S, T, tok, V, ld, mode, windows, fill = _mixed_case(seed)
    o_rows = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
    lps = o_rows["logp_s"].astype(np.float32)
    lpt = o_rows["logp_t"].astype(np.float32)
    d = lps.astype(np.float64) - lpt.astype(np.float64)
    o0 = oracle.scan_batch(lpt.astype(np.float64), d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode,
                           np.float64(-1e30), logp_s=lps.astype(np.float64))
    lam = _lambda(o0, lay, mode, rng)
    special = rng.random(lay.n_traj)
    lam[special < 0.1] = np.float32(np.inf)
    lam[(special >= 0.1) & (special < 0.2)] = np.float32(-np.inf)
    lam[(special >= 0.2) & (special < 0.3)] = np.float32(np.nan)
    cum0 = np.where(rng.random(lay.n_traj) < 0.3, rng.uniform(-80.0, 0.0, lay.n_traj), 0.0)
    o = oracle.scan_batch(lpt.astype(np.float64), d, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, mode,
                          lam.astype(np.float64), cum_in=cum0, logp_s=lps.astype(np.float64))
    o.update(logp_t=lpt.astype(np.float64), logp_s=lps.astype(np.float64), d=d)
    dev = "cuda"
    R = lay.rows
    offs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(lay.n_traj)
    h = stride.state_to_numpy(st)[: lay.n_traj].copy()
    h["cum"] = cum0
    st[: lay.n_traj].copy_(torch.from_numpy(h.view(np.uint8).reshape(lay.n_traj, -1)).cuda())
    ts = stride.new_turn_stats(lay.n_turns)
    prof = stride.new_profile(dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    ws = torch.empty(stride.stride_score_batch_workspace_size(max(1, R)), dtype=torch.uint8, device=dev)
    lps_d, lpt_d, lam_d = (torch.from_numpy(a).to(dev) for a in (lps, lpt, lam))
    for a, b in windows:
        stride.stride_scan_logprobs(lps_d[a:b], lpt_d[a:b], *offs, a, b, mode, lam_d, st, turn_stats=ts,
                                    dev_status=status, workspace=ws, profile=prof)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    g = {"state": stride.state_to_numpy(st)[: lay.n_traj], "turn_stats": stride.turn_stats_to_numpy(ts)[: lay.n_turns],
         "profile": prof.cpu().numpy()}
    compare_scan(g, o, lay, mode, lam)
