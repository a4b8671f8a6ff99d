"""stride_score_batch_noalloc: the scoring call for callers that cannot
allocate device memory (their device memory belongs to another allocator, or
their path cannot take cudaMalloc/cudaFree's implicit synchronisation).  It
uses the library's built-in scratch instead of a caller workspace.

Checked through the C ABI against stride_score_batch on the same inputs, on
two calls in a row (the scratch keeps the previous call's contents, so the
second call shows that what must start at zero is cleared), then on a
chunked pass, within the parity tolerances used for the CUDA path.  The file
is collected last so that a run that stops at the first failure has already
run every other test; it also passes on its own in a fresh process."""
from __future__ import annotations

import numpy as np
import pytest

import synth
from gpu_helpers import LOGP_ATOL, SUM_RTOL, run_batch, to_dev

pytestmark = pytest.mark.gpu


def _inputs(seed=91, V=151_936):
    rng = np.random.default_rng(seed)
    lay = synth.ragged_layout(rng, 5, (2, 6), 20, 300)
    S = synth.bf16_bits_from_f32(rng.standard_normal((lay.rows, V), dtype=np.float32) * np.float32(4.0))
    T = synth.bf16_bits_from_f32(synth.f32_from_bf16_bits(S) + rng.standard_normal((lay.rows, V), dtype=np.float32)
                                 * np.float32(0.5))
    tok = rng.integers(0, V, lay.rows).astype(np.int32)
    return lay, S, T, tok


def _noalloc(stride, St, Tt, tk, lay, mode, lam, windows):
    import torch

    offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(lay.n_traj)
    ts = stride.new_turn_stats(lay.n_turns)
    R = lay.rows
    out = {k: torch.full((R,), float("nan"), dtype=torch.float32, device="cuda") for k in stride.ROW_OUTPUT_KEYS}
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for a, b in windows:
        stride.stride_score_batch_noalloc(St[a:b], Tt[a:b], tk[a:b], *offs, a, b, mode, float(lam), st,
                                          out={k: v[a:b] for k, v in out.items()}, turn_stats=ts,
                                          dev_status=status)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["state"] = stride.state_to_numpy(st)[: lay.n_traj]
    res["turn_stats"] = stride.turn_stats_to_numpy(ts)[: lay.n_turns]
    res["status"] = int(status.item())
    return res


def _same(a, b):
    assert a["status"] == b["status"] == 0
    for k in ("logp_s", "logp_t", "opd", "lse_s", "lse_t"):
        assert np.max(np.abs(a[k] - b[k])) <= LOGP_ATOL, k
    for k in ("x_s", "x_t"):
        assert np.array_equal(a[k], b[k]), k
    for f in ("n",):
        assert np.array_equal(a["turn_stats"][f], b["turn_stats"][f])
    for f in ("sum_t", "cum"):
        x, y = a["turn_stats"][f], b["turn_stats"][f]
        assert np.all(np.abs(x - y) <= SUM_RTOL * np.abs(y) + 1e-12), f
    for f in ("stop_row", "stop_turn", "rows_seen", "stopped", "loss_tokens"):
        assert np.array_equal(a["state"][f], b["state"][f]), f
    assert np.all(np.abs(a["state"]["loss"] - b["state"]["loss"]) <= SUM_RTOL * (np.abs(b["state"]["loss"]) + 1.0))
    assert np.all(np.abs(a["state"]["cum"] - b["state"]["cum"]) <= SUM_RTOL * np.abs(b["state"]["cum"]))


@pytest.mark.parametrize("mode,lam", [(0, -20.0), (1, -600.0)])
def test_noalloc_matches_workspace_entry_point(mode, lam):
    import torch

    import paper_2609_14636_gb300 as stride

    lay, S, T, tok = _inputs()
    St, Tt = to_dev(S), to_dev(T)
    tk = torch.from_numpy(tok).cuda()
    ref = run_batch(stride, St, Tt, tk, lay, mode, lam)
    assert 0 < int((ref["state"]["stop_row"] >= 0).sum()), "the threshold should stop something"
    R = lay.rows
    first = _noalloc(stride, St, Tt, tk, lay, mode, lam, [(0, R)])
    second = _noalloc(stride, St, Tt, tk, lay, mode, lam, [(0, R)])
    _same(first, ref)
    _same(second, ref)
    cuts = [0, 37, R // 2, R - 5, R]
    chunked = _noalloc(stride, St, Tt, tk, lay, mode, lam, list(zip(cuts[:-1], cuts[1:])))
    _same(chunked, ref)


def test_noalloc_rejects_oversize_window():
    import torch

    import paper_2609_14636_gb300 as stride

    n = stride.NOALLOC_MAX_ROWS + 1
    lay = synth.layout_from_turn_lengths([[n]])
    S = torch.zeros((n, 8), dtype=torch.bfloat16, device="cuda")
    tk = torch.zeros(n, dtype=torch.int32, device="cuda")
    offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(1)
    with pytest.raises(stride.StrideError) as e:
        stride.stride_score_batch_noalloc(S, S, tk, *offs, 0, n, 0, -1.0, st)
    assert e.value.code == stride.ERR_TOO_LARGE
    assert "STRIDE_NOALLOC_MAX_ROWS" in str(e.value)
    # the largest allowed window works
    m = stride.NOALLOC_MAX_ROWS
    lay2 = synth.layout_from_turn_lengths([[m]])
    offs2 = [torch.from_numpy(a).cuda() for a in (lay2.traj_row_off, lay2.turn_row_off, lay2.traj_turn_off)]
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = {"logp_t": torch.empty(m, dtype=torch.float32, device="cuda")}
    stride.stride_score_batch_noalloc(S[:m], S[:m], tk[:m], *offs2, 0, m, 1, -1e30, st, out=out, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.allclose(out["logp_t"].cpu().numpy(), -np.log(8.0), atol=LOGP_ATOL)


def test_noalloc_empty_window_checks_arguments():
    """An empty window launches nothing but gets the workspace entry point's
    argument checks: a bad stop mode, no trajectories or missing offsets are
    rejected by both entry points alike."""
    import torch

    import paper_2609_14636_gb300 as stride

    lay = synth.layout_from_turn_lengths([[4, 3]])
    S = torch.zeros((lay.rows, 8), dtype=torch.bfloat16, device="cuda")
    tk = torch.zeros(lay.rows, dtype=torch.int32, device="cuda")
    offs = [torch.from_numpy(a).cuda().data_ptr() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(1)
    L = stride.lib()

    def both(mode, n_traj, offsets):
        a = L.stride_score_batch(S.data_ptr(), S.data_ptr(), 0, 8, 8, tk.data_ptr(), *offsets, n_traj,
                                 lay.n_turns, 2, 2, mode, None, -1.0, st.data_ptr(), None, None, None, None,
                                 None, 0, None)
        b = L.stride_score_batch_noalloc(S.data_ptr(), S.data_ptr(), 0, 8, 8, tk.data_ptr(), *offsets, n_traj,
                                         lay.n_turns, 2, 2, mode, None, -1.0, st.data_ptr(), None, None, None,
                                         None, None)
        return a, b

    assert both(0, 1, offs) == (stride.OK, stride.OK)
    assert both(7, 1, offs) == (stride.ERR_INVALID_ARG, stride.ERR_INVALID_ARG)
    assert both(0, 0, offs) == (stride.ERR_INVALID_ARG, stride.ERR_INVALID_ARG)
    assert both(0, 1, [offs[0], None, offs[2]]) == (stride.ERR_INVALID_ARG, stride.ERR_INVALID_ARG)
