"""GPU parity of the vocabulary-sharded path (stride_partial_lse ->
stride_combine_partials -> stride_scan_logprobs): tensor-parallel shards of
a row combine to the full row's log-probs, and the scan on log-probs gives
the results of the fused call and of the oracle."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from gpu_helpers import LOGP_ATOL, compare_rows, compare_scan, oracle_batch, run_batch, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


def _case(seed, V):
    rng = np.random.default_rng(seed)
    lay = synth.ragged_layout(rng, 5, (2, 6), 16, 160)
    S = synth.bf16_bits_from_f32(rng.standard_normal((lay.rows, V), dtype=np.float32) * np.float32(4.0))
    T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + rng.standard_normal((lay.rows, V), dtype=np.float32)
                                 * np.float32(0.5))
    tok = rng.integers(0, V, lay.rows).astype(np.int32)
    return lay, S, T, tok


def _sharded_logprobs(stride, St, Tt, tk, bounds):
    import torch

    R = St.shape[0]
    parts = torch.empty((len(bounds) - 1, R, 6), dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for k, (c0, c1) in enumerate(zip(bounds[:-1], bounds[1:])):
        stride.stride_partial_lse(St[:, c0:c1], Tt[:, c0:c1], tk, c0, parts[k], status, V_shard=c1 - c0)
    ls = torch.empty(R, dtype=torch.float32, device="cuda")
    lt = torch.empty(R, dtype=torch.float32, device="cuda")
    stride.stride_combine_partials(parts, ls, lt, dev_status=status)
    torch.cuda.synchronize()
    return ls, lt, int(status.item())


def _scan(stride, ls, lt, lay, mode, lam, windows=None):
    import torch

    R = lay.rows
    offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(lay.n_traj)
    ts = stride.new_turn_stats(lay.n_turns)
    prof = stride.new_profile()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    opd = torch.empty(R, dtype=torch.float32, device="cuda")
    windows = windows or [(0, R)]
    ws = torch.empty(stride.stride_score_batch_workspace_size(max(b - a for a, b in windows)), dtype=torch.uint8,
                     device="cuda")
    for a, b in windows:
        stride.stride_scan_logprobs(ls[a:b], lt[a:b], *offs, a, b, mode, float(np.float32(lam)), st, opd=opd[a:b],
                                    turn_stats=ts, dev_status=status, workspace=ws, profile=prof)
    torch.cuda.synchronize()
    return dict(logp_s=ls.cpu().numpy(), logp_t=lt.cpu().numpy(), opd=opd.cpu().numpy(),
                state=stride.state_to_numpy(st)[: lay.n_traj], turn_stats=stride.turn_stats_to_numpy(ts)[: lay.n_turns],
                status=int(status.item()), profile=prof.cpu().numpy())


@pytest.mark.parametrize("bounds_kind", ["4_equal", "3_ragged", "aligned_with_tail"])
def test_shards_combine_to_full_rows(stride, bounds_kind):
    """4_equal: 16-byte-aligned shards of whole vectors; 3_ragged: shards
    starting off the 16-byte grid; aligned_with_tail: an aligned shard whose
    width leaves 3 logits past its last whole vector, then an unaligned
    one."""
    import torch

    V = 151_936
    lay, S, T, tok = _case(61, V)
    bounds = {"4_equal": [0, 37_984, 75_968, 113_952, V], "3_ragged": [0, 50_001, 100_003, V],
              "aligned_with_tail": [0, 40_000, 80_003, V]}[bounds_kind]
    St, Tt = to_dev(S), to_dev(T)
    tk = torch.from_numpy(tok).cuda()
    ls, lt, status = _sharded_logprobs(stride, St, Tt, tk, bounds)
    assert status == 0
    full = run_batch(stride, St, Tt, tk, lay, stride.TURN_MEAN, -1e30)
    assert np.max(np.abs(ls.cpu().numpy() - full["logp_s"])) <= 1e-4
    assert np.max(np.abs(lt.cpu().numpy() - full["logp_t"])) <= 1e-4
    o = oracle_batch(S, T, tok, lay, oracle.TURN_MEAN, -1e30)
    assert np.max(np.abs(ls.cpu().numpy() - o["logp_s"])) <= LOGP_ATOL
    assert np.max(np.abs(lt.cpu().numpy() - o["logp_t"])) <= LOGP_ATOL


@pytest.mark.parametrize("V,n_shards", [(37, 37), (4099, 64)])
def test_many_and_single_column_shards(stride, V, n_shards):
    """Many shards: one column each (every shard but one misses the token),
    or 64 shards of random widths (most of them starting off the 16-byte
    grid); their partials merge to the oracle's log-probs."""
    import torch

    lay, S, T, tok = _case(64, V)
    rng = np.random.default_rng(65)
    cuts = np.sort(rng.choice(np.arange(1, V), size=n_shards - 1, replace=False)) if n_shards < V else np.arange(1, V)
    bounds = [0] + [int(c) for c in cuts] + [V]
    St, Tt = to_dev(S), to_dev(T)
    tk = torch.from_numpy(tok).cuda()
    ls, lt, status = _sharded_logprobs(stride, St, Tt, tk, bounds)
    assert status == 0
    o = oracle_batch(S, T, tok, lay, oracle.TURN_MEAN, -1e30)
    assert np.max(np.abs(ls.cpu().numpy() - o["logp_s"])) <= LOGP_ATOL
    assert np.max(np.abs(lt.cpu().numpy() - o["logp_t"])) <= LOGP_ATOL


@pytest.mark.parametrize("mode", [0, 1])
def test_scan_on_sharded_logprobs(stride, mode):
    import torch

    V = 8192
    lay, S, T, tok = _case(62, V)
    St, Tt = to_dev(S), to_dev(T)
    tk = torch.from_numpy(tok).cuda()
    ls, lt, status = _sharded_logprobs(stride, St, Tt, tk, [0, 2048, 4096, 6144, V])
    assert status == 0
    o0 = oracle_batch(S, T, tok, lay, mode, -1e30)
    lam = np.float32(np.median(o0["turn_cum"]) if mode == 0 else np.median(o0["row_cum"]))
    o = oracle_batch(S, T, tok, lay, mode, lam)
    R = lay.rows
    for windows in (None, [(0, 100), (100, R // 2), (R // 2, R)]):
        g = _scan(stride, ls, lt, lay, mode, lam, windows)
        assert g["status"] == 0
        compare_rows(g, o)
        compare_scan(g, o, lay, mode, lam)
    # the scan alone, on the oracle's own log-probs
    g = _scan(stride, torch.from_numpy(o["logp_s"].astype(np.float32)).cuda(),
              torch.from_numpy(o["logp_t"].astype(np.float32)).cuda(), lay, mode, lam)
    compare_scan(g, o, lay, mode, lam)


def _tile_layout(kind, rng):
    if kind == "one_row_turns":  # hundreds of turns inside one 256-row tile
        turns = [[int(x) for x in rng.choice([1, 1, 1, 2, 5, 40], size=180)] for _ in range(3)]
    else:  # trajectories spanning dozens of tiles
        turns = [[int(x) for x in rng.integers(64, 513, size=30)] for _ in range(3)]
    return synth.layout_from_turn_lengths(turns)


@pytest.mark.parametrize("kind", ["one_row_turns", "long_trajectories"])
@pytest.mark.parametrize("mode", [0, 1])
def test_scan_tiles_on_logprobs(stride, kind, mode):
    """stride_scan_logprobs on given log-probs against the oracle's scan of
    the same values: many one-row turns per tile, trajectories across many
    tiles, and windows that cut tiles, trajectories and turns."""
    import torch

    rng = np.random.default_rng(63 + mode)
    lay = _tile_layout(kind, rng)
    R = lay.rows
    lt = (-np.abs(rng.standard_normal(R) * 2.0) - 0.5).astype(np.float32)
    ls = (lt + rng.standard_normal(R).astype(np.float32) * np.float32(0.3)).astype(np.float32)
    d = (ls - lt).astype(np.float32)  # as the kernel forms it
    o0 = oracle.scan_batch(lt.astype(np.float64), d.astype(np.float64), lay.traj_row_off, lay.turn_row_off,
                           lay.traj_turn_off, mode, np.float64(-1e30), logp_s=ls.astype(np.float64))
    lam = np.float32(np.median(o0["turn_cum"]) if mode == 0 else np.median(o0["row_cum"]))
    o = oracle.scan_batch(lt.astype(np.float64), d.astype(np.float64), lay.traj_row_off, lay.turn_row_off,
                          lay.traj_turn_off, mode, np.float64(lam), logp_s=ls.astype(np.float64))
    o.update(logp_t=lt.astype(np.float64), d=d.astype(np.float64), logp_s=ls.astype(np.float64))
    ls_d, lt_d = torch.from_numpy(ls).cuda(), torch.from_numpy(lt).cuda()
    for windows in (None, [(0, 777), (777, R // 2 + 13), (R // 2 + 13, R)]):
        g = _scan(stride, ls_d, lt_d, lay, mode, lam, windows)
        assert g["status"] == 0
        assert np.array_equal(g["opd"], d)
        compare_scan(g, o, lay, mode, lam)
    assert int(np.sum(o["stop_row"] >= 0)) > 0


def test_token_owned_by_no_shard(stride):
    import torch

    V = 1024
    lay, S, T, tok = _case(63, V)
    tok[3] = V + 5
    St, Tt = to_dev(S), to_dev(T)
    ls, lt, status = _sharded_logprobs(stride, St, Tt, torch.from_numpy(tok).cuda(), [0, 512, V])
    assert status & stride.DEV_TOKEN_RANGE
    assert np.isnan(ls.cpu().numpy()[3]) and np.isfinite(ls.cpu().numpy()[4])
