"""The end-to-end pattern of the bench's e2e leg, checked against the oracle:
logits and tokens in pinned host memory, copied window by window on a copy
stream (an event per window), each window scored on a separate compute
stream (not the default one) once its copy has landed, with the carried
state, and the per-row outputs, state and turn statistics copied back to
pinned host memory -- twice in a row on the same buffers, the second pass's
copies waiting on the first pass's kernels.  Windows of 512 rows take the
small-window kernels, windows of 2,048 the persistent kernel."""
import numpy as np
import pytest

import synth
from gpu_helpers import compare_rows, compare_scan, oracle_batch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


def _case():
    rng = np.random.default_rng(4242)
    lens = [[int(x) for x in rng.integers(16, 400, size=int(rng.integers(2, 8)))] for _ in range(7)]
    lay = synth.layout_from_turn_lengths(lens)
    R, V = lay.rows, 4099
    S32 = rng.standard_normal((R, V), dtype=np.float32) * np.float32(3.0)
    S = synth.bf16_bits_from_f32(S32)
    T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + rng.standard_normal((R, V), dtype=np.float32))
    tok = rng.integers(0, V, R).astype(np.int32)
    return lay, S, T, tok, V


@pytest.mark.parametrize("window", [512, 2048])
def test_pinned_host_windows_on_two_streams(stride, window):
    import torch

    lay, S, T, tok, V = _case()
    R = lay.rows
    mode = stride.TURN_MEAN
    o0 = oracle_batch(S, T, tok, lay, mode, np.float32(-1e30))
    # lambda halfway between the running sums after the second and third
    # turns (a stop at the third), or below every sum of a shorter trajectory
    lam = np.array([np.float32(0.5 * (o0["turn_cum"][k0 + 1] + o0["turn_cum"][k0 + 2])) if k1 - k0 >= 3
                    else np.float32(o0["turn_cum"][k1 - 1] - 1.0)
                    for k0, k1 in zip(lay.traj_turn_off[:-1], lay.traj_turn_off[1:])], np.float32)
    o = oracle_batch(S, T, tok, lay, mode, lam)

    dev = torch.device("cuda")
    hS = torch.from_numpy(S.view(np.int16)).view(torch.bfloat16).pin_memory()
    hT = torch.from_numpy(T.view(np.int16)).view(torch.bfloat16).pin_memory()
    hk = torch.from_numpy(tok).pin_memory()
    dS = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
    dT = torch.empty_like(dS)
    dk = torch.empty(R, dtype=torch.int32, device=dev)
    offs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    lam_d = torch.from_numpy(lam).to(dev)
    st = stride.new_state(lay.n_traj, dev)
    ts = stride.new_turn_stats(lay.n_turns, dev)
    keys = ("logp_s", "logp_t", "opd", "lse_s", "lse_t", "x_s", "x_t")
    dout = {k: torch.empty(R, dtype=torch.float32, device=dev) for k in keys}
    hout = {k: torch.empty(R, dtype=torch.float32).pin_memory() for k in keys}
    hst = torch.empty((lay.n_traj, stride.STATE_DTYPE.itemsize), dtype=torch.uint8).pin_memory()
    hts = torch.empty((lay.n_turns, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8).pin_memory()
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    wins = [(a, min(R, a + window)) for a in range(0, R, window)]
    ws = torch.empty(stride.stride_score_batch_workspace_size(window), dtype=torch.uint8, device=dev)
    compute, copy = torch.cuda.Stream(), torch.cuda.Stream()
    landed = [torch.cuda.Event() for _ in wins]

    for _ in range(2):
        go = torch.cuda.Event()
        go.record(compute)  # the previous pass's kernels are done with the landing buffers
        copy.wait_event(go)
        with torch.cuda.stream(copy):
            for i, (a, b) in enumerate(wins):
                dS[a:b].copy_(hS[a:b], non_blocking=True)
                dT[a:b].copy_(hT[a:b], non_blocking=True)
                dk[a:b].copy_(hk[a:b], non_blocking=True)
                landed[i].record(copy)
        stride.stride_state_init(st, lay.n_traj, compute)
        for i, (a, b) in enumerate(wins):
            compute.wait_event(landed[i])
            stride.stride_score_batch(dS[a:b], dT[a:b], dk[a:b], *offs, a, b, mode, lam_d, st,
                                      out={k: v[a:b] for k, v in dout.items()}, turn_stats=ts,
                                      dev_status=status, workspace=ws, stream=compute)
        with torch.cuda.stream(compute):
            for k in keys:
                hout[k].copy_(dout[k], non_blocking=True)
            hst.copy_(st[: lay.n_traj], non_blocking=True)
            hts.copy_(ts[: lay.n_turns], non_blocking=True)
        compute.synchronize()
        g = {k: hout[k].numpy().copy() for k in keys}
        g["state"] = hst.numpy().view(stride.STATE_DTYPE).reshape(-1).copy()
        g["turn_stats"] = hts.numpy().view(stride.TURN_STATS_DTYPE).reshape(-1).copy()
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        compare_rows(g, o)
        compare_scan(g, o, lay, mode, lam)
