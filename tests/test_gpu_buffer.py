"""GPU parity of the device-resident prefix buffer H(x) (stride_buffer_record)
and of Algorithm 1's loop on the device: score -> record -> select -> restart."""
from __future__ import annotations

import json
import math
from pathlib import Path

import numpy as np
import pytest

import oracle
import synth
from gpu_helpers import LOGP_ATOL, run_batch

pytestmark = pytest.mark.gpu
GOLD = Path(__file__).resolve().parent / "golden"


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


def _stats_tensor(stride, means):
    """Device turn stats whose mean_t are `means` (other fields zero)."""
    import torch

    a = np.zeros(max(1, len(means)), stride.TURN_STATS_DTYPE)
    a["mean_t"][: len(means)] = means
    return torch.from_numpy(a.view(np.uint8).reshape(len(a), -1).copy()).cuda()


def _record(stride, mean, n, task, k0, means, off):
    import torch

    m, nt = torch.from_numpy(mean).cuda(), torch.from_numpy(n).cuda()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    stride.stride_buffer_record(m, nt, torch.from_numpy(np.asarray(task, np.int32)).cuda(),
                                None if k0 is None else torch.from_numpy(np.asarray(k0, np.int32)).cuda(),
                                _stats_tensor(stride, np.asarray(means, np.float32)),
                                torch.from_numpy(np.asarray(off, np.int32)).cuda(), status)
    torch.cuda.synchronize()
    return m.cpu().numpy(), nt.cpu().numpy(), int(status.item())


def _f(x):
    return -math.inf if x == "-inf" else float(x)


def test_buffer_golden(stride):
    for c in json.loads((GOLD / "prefix_buffer_cases.json").read_text())["cases"]:
        T_max = c["T_max"]
        mean = np.full((1, T_max), np.float32(123.0), np.float32)
        mean[0, :len(c["stored"])] = c["stored"]
        n = np.array([len(c["stored"])], np.int32)
        ks, _ = oracle.select_restart(mean, n, None, _f(c["alpha"]))
        m, nt, st = _record(stride, mean, n, [0], ks, c["new_turn_means"], [0, len(c["new_turn_means"])])
        assert st == 0 and int(nt[0]) == len(c["record_after"]) and list(m[0, :nt[0]]) == c["record_after"], c["name"]


def test_buffer_random_matches_oracle(stride):
    rng = np.random.default_rng(41)
    n_tasks, T_max = 300, 12
    mean = rng.standard_normal((n_tasks, T_max)).astype(np.float32)
    n = rng.integers(0, T_max + 1, n_tasks).astype(np.int32)
    tasks = rng.permutation(n_tasks)[:200].astype(np.int32)
    k0 = rng.integers(0, T_max + 2, 200).astype(np.int32)
    lens = rng.integers(0, 15, 200)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    tm = rng.standard_normal(int(off[-1])).astype(np.float32)
    m, nt, st = _record(stride, mean, n, tasks, k0, tm, off)
    om, on = mean.copy(), n.copy()
    oracle.buffer_record(om, on, tasks, k0, tm, off)
    assert st == 0 and np.array_equal(nt, on)
    for x in range(n_tasks):
        assert np.array_equal(m[x, :nt[x]], om[x, :on[x]])
    # a bad task id is reported and skipped
    m2, nt2, st2 = _record(stride, mean, n, [n_tasks], None, [1.0], [0, 1])
    assert st2 & stride.DEV_BAD_LAYOUT and np.array_equal(nt2, n)


def test_algorithm1_loop_on_device(stride):
    """Three iterations of Algorithm 1 for 12 tasks of 6 turns each: score
    the rollouts (turn-mean stop rule), record {l_k} in H(x) keeping the
    reused prefix, choose the next restart k* (alpha gate); the device
    buffer follows the oracle's at every iteration."""
    import torch

    rng = np.random.default_rng(43)
    n_tasks, T_turns, V = 12, 6, 2048
    buf = torch.zeros((n_tasks, T_turns), dtype=torch.float32, device="cuda")
    nt = torch.zeros(n_tasks, dtype=torch.int32, device="cuda")
    obuf = np.zeros((n_tasks, T_turns), np.float32)
    ont = np.zeros(n_tasks, np.int32)
    k0 = np.zeros(n_tasks, np.int32)
    alpha = -12.3  # mid-range of this workload's turn means (uniform tokens score about -12)
    reused = 0
    for it in range(3):
        reused += int((k0 > 0).sum())
        # each task's rollout regenerates turns k0 .. T_turns-1
        lens = [[int(x) for x in rng.integers(8, 40, T_turns - k0[x])] for x in range(n_tasks)]
        lay = synth.layout_from_turn_lengths(lens)
        S = synth.bf16_bits_from_f32(rng.standard_normal((lay.rows, V), dtype=np.float32) * np.float32(3.0))
        T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + rng.standard_normal((lay.rows, V), dtype=np.float32)
                                     * np.float32(1.2 - 0.4 * it))
        tok = rng.integers(0, V, lay.rows).astype(np.int32)
        g = run_batch(stride, S, T, tok, lay, stride.TURN_MEAN, -1e30)
        o = oracle.row_logprobs(S, T, tok)
        osc = oracle.scan_batch(o["logp_t"], o["d"], lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                                oracle.TURN_MEAN, -1e30)
        ts = torch.from_numpy(g["turn_stats"].view(np.uint8).reshape(lay.n_turns, -1).copy()).cuda()
        k0_d = torch.from_numpy(k0).cuda()
        tasks = torch.arange(n_tasks, dtype=torch.int32, device="cuda")
        tto = torch.from_numpy(lay.traj_turn_off).cuda()
        stride.stride_buffer_record(buf, nt, tasks, k0_d, ts, tto)
        oracle.buffer_record(obuf, ont, np.arange(n_tasks), k0, osc["turn_mean"].astype(np.float32),
                             lay.traj_turn_off)
        gb, gn = buf.cpu().numpy(), nt.cpu().numpy()
        assert np.array_equal(gn, ont)
        for x in range(n_tasks):
            assert np.max(np.abs(gb[x, :gn[x]] - obuf[x, :ont[x]])) <= LOGP_ATOL
        # next restart point from the device record; the oracle's select on
        # the same fp32 record agrees bit for bit
        ks = torch.empty(n_tasks, dtype=torch.int32, device="cuda")
        km = torch.empty(n_tasks, dtype=torch.int32, device="cuda")
        stride.stride_select_restart(buf, nt, None, alpha, ks, km)
        torch.cuda.synchronize()
        oks, okm = oracle.select_restart(gb, gn, None, alpha)
        assert np.array_equal(ks.cpu().numpy(), oks) and np.array_equal(km.cpu().numpy(), okm)
        k0 = oks.astype(np.int32)
    assert reused > 0, "some restarts must reuse a stored prefix"
