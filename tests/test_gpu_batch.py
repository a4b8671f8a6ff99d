"""GPU parity of stride_score_batch against the oracle (CUDA path through the
C ABI, same seeded inputs on both sides)."""
from __future__ import annotations

import math

import numpy as np
import pytest

import oracle
import synth
from gpu_helpers import (LOGP_ATOL, compare_rows, compare_scan, oracle_batch, pad_cols, run_batch,
                         to_dev)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


@pytest.fixture(params=["auto", "stream", "split", "split1", "split8", "rows"])
def kernel(request, stride):
    """Runs a test under each of the batch kernels, and the split kernel at
    its automatic, smallest (one CTA per row) and largest (8-CTA) cluster
    size (stride_force_batch_kernel; automatic again afterwards)."""
    stride.stride_force_batch_kernel(request.param)
    yield request.param
    stride.stride_force_batch_kernel("auto")


def _bf16_rows(seed, R, V, sigma=4.0, noise=0.5):
    rng = np.random.default_rng(seed)
    S32 = (rng.standard_normal((R, V), dtype=np.float32) * np.float32(sigma))
    S = synth.bf16_bits_from_f32(S32)
    T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + rng.standard_normal((R, V), dtype=np.float32) * np.float32(noise))
    tok = rng.integers(0, V, R).astype(np.int32)
    return S, T, tok


def _lam_between_turns(o, lay, targets):
    """Per-trajectory lambda (fp32) halfway between the oracle's running sums
    at turn target-1 and target, so that trajectory i stops at turn
    targets[i] (-1: never, lambda below every sum)."""
    lam = np.empty(lay.n_traj, np.float32)
    for i, t in enumerate(targets):
        k0, k1 = lay.traj_turn_off[i], lay.traj_turn_off[i + 1]
        cums = o["turn_cum"][k0:k1]
        if t < 0:
            lam[i] = np.float32(cums[-1] - 1.0)  # below every running sum
        elif t == 0:
            lam[i] = np.float32(0.5 * cums[0])  # sums are < 0: the first one already crosses
        else:
            lam[i] = np.float32(0.5 * (cums[t - 1] + cums[t]))
    return lam


# ---------------------------------------------------------------------------
# tiny reference workload: 1 x 4 turns x 128 tokens, V = 32,000, fp32
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("mode,lam_key", [(1, "lam_token"), (0, "lam_turn")])
def test_tiny_reference(stride, kernel, mode, lam_key):
    w = synth.tiny_reference(0)
    g = run_batch(stride, w["S"], w["T"], w["tokens"], w["layout"], mode, w[lam_key])
    o = oracle_batch(w["S"], w["T"], w["tokens"], w["layout"], mode, w[lam_key])
    assert g["status"] == 0
    compare_rows(g, o)
    compare_scan(g, o, w["layout"], mode, w[lam_key])
    assert g["state"]["stop_row"][0] >= 0  # both thresholds fire on this workload


# ---------------------------------------------------------------------------
# ragged bf16 rows: vector body, ragged tail, scalar path, tiny V
# ---------------------------------------------------------------------------
LENS = [[1, 5, 17, 3], [9, 1], [33, 2, 1, 1, 4], [2]]


@pytest.mark.parametrize("V,ld", [(151_936, 151_936), (151_933, 151_936), (151_933, 151_933),
                                  (262_147, 262_152), (4099, 4099), (8, 8), (7, 8), (1, 1), (1, 8)])
@pytest.mark.parametrize("mode", [0, 1])
def test_bf16_ragged(stride, kernel, V, ld, mode):
    lay = synth.layout_from_turn_lengths(LENS)
    S, T, tok = _bf16_rows(V + ld, lay.rows, V)
    Sp, Tp = pad_cols(S, ld, 0x7FC0), pad_cols(T, ld, 0x7FC0)  # NaN padding must never be read
    lam0 = np.float32(-1e30)
    o0 = oracle_batch(S, T, tok, lay, mode, lam0)
    if mode == 0:
        lam = _lam_between_turns(o0, lay, [2, 0, 4, -1])
    else:
        lam = np.array([np.float32(0.5 * (o0["row_cum"][3] + o0["row_cum"][4])), lam0, lam0, lam0], np.float32)
    g = run_batch(stride, Sp, Tp, tok, lay, mode, lam, V=V)
    o = oracle_batch(S, T, tok, lay, mode, lam)
    assert g["status"] == 0
    compare_rows(g, o)
    compare_scan(g, o, lay, mode, lam)


def test_f32_vector_and_scalar_paths(stride, kernel):
    rng = np.random.default_rng(5)
    lay = synth.layout_from_turn_lengths([[7, 3], [11]])
    V = 32_000
    S = (rng.standard_normal((lay.rows, V)) * 3).astype(np.float32)
    T = (S + rng.standard_normal((lay.rows, V)) * 0.5).astype(np.float32)
    tok = rng.integers(0, V, lay.rows).astype(np.int32)
    o = oracle_batch(S, T, tok, lay, 1, -40.0)
    for ld in (32_000, 32_001, 32_004):
        g = run_batch(stride, pad_cols(S, ld, np.float32(np.nan)), pad_cols(T, ld, np.float32(np.nan)),
                      tok, lay, 1, -40.0, V=V)
        compare_rows(g, o)
        compare_scan(g, o, lay, 1, -40.0)


# ---------------------------------------------------------------------------
# chunked windows: same results as one call and as the oracle
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("mode", [0, 1])
def test_chunked_windows(stride, kernel, mode):
    rng = np.random.default_rng(9)
    lay = synth.ragged_layout(rng, 6, (1, 7), 1, 60)
    V = 3000
    S, T, tok = _bf16_rows(10, lay.rows, V)
    o0 = oracle_batch(S, T, tok, lay, mode, -1e30)
    if mode == 0:
        lam = _lam_between_turns(o0, lay, [min(2, lay.traj_turn_off[i + 1] - lay.traj_turn_off[i] - 1) for i in range(lay.n_traj)])
    else:
        lam = np.float32(-60.0)
    o = oracle_batch(S, T, tok, lay, mode, lam)
    one = run_batch(stride, S, T, tok, lay, mode, lam)
    compare_rows(one, o)
    compare_scan(one, o, lay, mode, lam)
    R = lay.rows
    for cuts in ([1], [37, 38, 100], list(range(5, R, 23)), [R - 1]):
        edges = [0] + [c for c in cuts if 0 < c < R] + [R]
        windows = list(zip(edges[:-1], edges[1:]))
        g = run_batch(stride, S, T, tok, lay, mode, lam, windows=windows)
        compare_rows(g, o)
        compare_scan(g, o, lay, mode, lam)
        assert np.array_equal(g["state"]["stop_row"], one["state"]["stop_row"])
        assert np.array_equal(g["turn_stats"]["n"], one["turn_stats"]["n"])


def test_many_tiles(stride, kernel):
    """Thousands of tiles, hundreds of trajectories, single-row turns: the
    lookback chain crosses many trajectory and turn boundaries."""
    rng = np.random.default_rng(21)
    lay = synth.ragged_layout(rng, 300, (1, 12), 1, 12)
    V = 257
    S, T, tok = _bf16_rows(22, lay.rows, V, sigma=2.0)
    for mode, lam in ((0, np.float32(-9.0)), (1, np.float32(-30.0))):
        g = run_batch(stride, S, T, tok, lay, mode, lam)
        o = oracle_batch(S, T, tok, lay, mode, lam)
        compare_rows(g, o)
        compare_scan(g, o, lay, mode, lam)
        assert 0 < int((g["state"]["stop_row"] >= 0).sum()) < lay.n_traj


def test_long_token_sum_trajectory(stride, kernel):
    """One 40,000-token trajectory in token mode (the math setting): the
    running sum over many tiles stays within 1e-5 relative (under the split
    kernels the tiled scan chains 157 tiles of one segment)."""
    rng = np.random.default_rng(23)
    lay = synth.layout_from_turn_lengths([[40_000]])
    V = 64
    S, T, tok = _bf16_rows(24, lay.rows, V, sigma=1.0, noise=0.3)
    o0 = oracle_batch(S, T, tok, lay, 1, -1e30)
    lam = np.float32(0.5 * (o0["row_cum"][29_999] + o0["row_cum"][30_000]))
    g = run_batch(stride, S, T, tok, lay, 1, lam)
    o = oracle_batch(S, T, tok, lay, 1, lam)
    compare_rows(g, o)
    compare_scan(g, o, lay, 1, lam)


# ---------------------------------------------------------------------------
# closed forms and special values on the GPU
# ---------------------------------------------------------------------------
def test_uniform_rows_closed_form(stride):
    for V in (1, 7, 8, 4099, 151_936):
        lay = synth.layout_from_turn_lengths([[3]])
        S = np.full((3, V), 0x4060, np.uint16)  # 3.5 in bf16
        tok = np.array([0, V - 1, V // 2], np.int32)
        g = run_batch(stride, S, S, tok, lay, 1, -1e30)
        assert np.max(np.abs(g["logp_s"] + math.log(V))) <= LOGP_ATOL
        assert np.array_equal(g["opd"], np.zeros(3, np.float32))


def test_identical_rows_zero_opd(stride):
    lay = synth.layout_from_turn_lengths([[40, 9]])
    S, _, tok = _bf16_rows(31, lay.rows, 151_936)
    g = run_batch(stride, S, S, tok, lay, 0, -1e30)
    assert np.array_equal(g["logp_s"], g["logp_t"])
    assert np.array_equal(g["opd"], np.zeros(lay.rows, np.float32))
    assert np.array_equal(g["turn_stats"]["sum_d"], np.zeros(2))


def test_masked_vocab_entries(stride, kernel):
    """-inf logits carry no probability mass."""
    lay = synth.layout_from_turn_lengths([[6]])
    V = 5000
    S, T, tok = _bf16_rows(41, lay.rows, V)
    S[:, 1000:3000] = 0xFF80
    T[:, 2000:4500] = 0xFF80
    tok[:3] = [5, 10, 4999]
    tok[3] = 1500  # masked in S: logp_s = -inf
    g = run_batch(stride, S, T, tok, lay, 1, -1e30)
    o = oracle_batch(S, T, tok, lay, 1, -1e30)
    compare_rows(g, o, rows=slice(0, 3))
    assert g["logp_s"][3] == -np.inf


@pytest.mark.parametrize("mode", [0, 1])
def test_masked_teacher_token_stops_at_minus_inf(stride, kernel, mode):
    """A sampled token whose teacher logit is -inf: log pi_T = -inf, so the
    running sum is -inf from that row (token mode) or that turn's end (turn
    mode) on, and the trajectory stops there, as in the fp64 oracle."""
    lay = synth.layout_from_turn_lengths([[6, 6, 4], [5, 7]])
    V = 5000
    S, T, tok = _bf16_rows(43, lay.rows, V)
    T[8, 2000:2500] = 0xFF80  # trajectory 0, turn 1, its third row
    tok[8] = 2100
    g = run_batch(stride, S, T, tok, lay, mode, -1e30)
    o = oracle_batch(S, T, tok, lay, mode, -1e30)
    assert g["logp_t"][8] == -np.inf and o["logp_t"][8] == -np.inf
    st = g["state"]
    assert int(st["stop_turn"][0]) == 1
    assert int(st["stop_row"][0]) == (8 if mode == 1 else 11)
    assert int(st["stop_row"][1]) == -1 and int(st["stop_turn"][1]) == -1
    ts = g["turn_stats"]
    assert ts["sum_t"][1] == -np.inf and o["turn_sum_t"][1] == -np.inf
    assert ts["sum_t"][3] == pytest.approx(o["turn_sum_t"][3], rel=1e-5)


def test_token_out_of_range_sets_status(stride, kernel):
    lay = synth.layout_from_turn_lengths([[4], [3]])
    S, T, tok = _bf16_rows(51, lay.rows, 1000)
    tok[1] = 1000
    tok[5] = -3
    g = run_batch(stride, S, T, tok, lay, 0, -1e30)
    assert g["status"] & stride.DEV_TOKEN_RANGE
    assert np.isnan(g["logp_t"][1]) and np.isnan(g["logp_s"][5])
    o = oracle_batch(S, T, tok, lay, 0, -1e30)
    ok = [0, 2, 3, 4, 6]
    compare_rows({k: g[k][ok] for k in ("logp_s", "logp_t", "opd")}, {k: o[k][ok] for k in ("logp_s", "logp_t", "d")})


def test_empty_turn_sets_status(stride):
    lay = synth.layout_from_turn_lengths([[3, 0, 2]])
    S, T, tok = _bf16_rows(61, lay.rows, 100)
    g = run_batch(stride, S, T, tok, lay, 0, -1e30)
    assert g["status"] & stride.DEV_BAD_LAYOUT


def test_prefix_buffer_restart_scores_new_turns(stride):
    """A restarted rollout is scored over its newly generated turns only
    (Sec. 4.1): the caller passes the new turns as the trajectory, and a
    fresh state gives the running sum that starts at K0."""
    rng = np.random.default_rng(71)
    lens = [int(x) for x in rng.integers(20, 60, 6)]
    V = 2048
    lay_full = synth.layout_from_turn_lengths([lens])
    S, T, tok = _bf16_rows(72, lay_full.rows, V)
    K0 = 2
    r0 = int(lay_full.turn_row_off[K0])
    lay_new = synth.layout_from_turn_lengths([lens[K0:]])
    o_full = oracle_batch(S, T, tok, lay_full, 0, -1e30)
    o_new = oracle_batch(S[r0:], T[r0:], tok[r0:], lay_new, 0, -1e30)
    lam = _lam_between_turns(o_new, lay_new, [2])
    g = run_batch(stride, S[r0:], T[r0:], tok[r0:], lay_new, 0, lam)
    o = oracle_batch(S[r0:], T[r0:], tok[r0:], lay_new, 0, lam)
    compare_scan(g, o, lay_new, 0, lam)
    assert int(g["state"]["stop_turn"][0]) == 2
    # the same lambda over the whole record would have fired at another turn
    assert not np.allclose(o_full["turn_cum"][K0:], o_new["turn_cum"])


def test_invalid_arguments(stride):
    import torch

    lay = synth.layout_from_turn_lengths([[4]])
    S, T, tok = _bf16_rows(81, 4, 64)
    St, Tt = to_dev(S), to_dev(T)
    tk = torch.from_numpy(tok).cuda()
    offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(1)
    ws = torch.empty(stride.stride_score_batch_workspace_size(4), dtype=torch.uint8, device="cuda")
    with pytest.raises(stride.StrideError) as e:
        stride.stride_score_batch(St, Tt, tk, *offs, 0, 4, 0, -1.0, st, workspace=ws, V=65)
    assert e.value.code == 1
    with pytest.raises(stride.StrideError) as e:
        stride.stride_score_batch(St, Tt, tk, *offs, 0, 4, 0, -1.0, st, workspace=ws[:64])
    assert e.value.code == 3
    with pytest.raises(stride.StrideError) as e:
        stride.stride_score_batch(St, Tt, tk, *offs, 0, 4, 7, -1.0, st, workspace=ws)
    assert e.value.code == 1
    stride.stride_score_batch(St, Tt, tk, *offs, 2, 2, 0, -1.0, st, workspace=ws)  # empty window: no-op
