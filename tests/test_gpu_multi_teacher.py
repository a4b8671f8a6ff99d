"""GPU parity of stride_score_batch_multi_teacher: the multi-teacher workload
(two domains, teacher noise from two independent streams) scored from one
teacher buffer per domain equals the same rows scored with an aligned
teacher buffer, and the oracle."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from gpu_helpers import compare_rows, compare_scan, run_batch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


@pytest.fixture(scope="module")
def case():
    """The first 6 trajectories of the multi-teacher workload, aligned and
    split by domain."""
    import torch

    w = synth.multi_teacher()
    lay = synth.sub_layout(w.layout, 6)
    R = lay.rows
    S, T, tok = synth.generate_rows(w.recipe, 0, R, device="cuda")
    dom = w.extra["domain"][:6].astype(np.uint8)
    assert set(dom.tolist()) == {0, 1}, "both domains must be present"
    row0 = np.zeros(6, np.int64)
    parts = [[], []]
    count = [0, 0]
    for i in range(6):
        a, b = int(lay.traj_row_off[i]), int(lay.traj_row_off[i + 1])
        row0[i] = count[dom[i]]
        parts[dom[i]].append(T[a:b])
        count[dom[i]] += b - a
    T_dom = [torch.cat(p).contiguous() for p in parts]
    lam = np.float32(synth.workload_lambda(w.name) / 2)  # half the 12-turn budget
    return dict(lay=lay, S=S, T=T, tok=tok, dom=dom, row0=row0, T_dom=T_dom, lam=lam)


def _run_multi(stride, c, windows):
    import torch

    lay = c["lay"]
    R = lay.rows
    offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(lay.n_traj)
    ts = stride.new_turn_stats(lay.n_turns)
    prof = stride.new_profile()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = {k: torch.full((R,), float("nan"), dtype=torch.float32, device="cuda") for k in stride.ROW_OUTPUT_KEYS}
    wmax = max(b - a for a, b in windows)
    ws = torch.empty(stride.multi_teacher_workspace_size(wmax), dtype=torch.uint8, device="cuda")
    dom = torch.from_numpy(c["dom"]).cuda()
    row0 = torch.from_numpy(c["row0"]).cuda()
    for a, b in windows:
        stride.stride_score_batch_multi_teacher(c["S"][a:b], c["T_dom"], dom, row0, c["tok"][a:b], *offs, a, b,
                                                stride.TURN_MEAN, float(c["lam"]), st,
                                                out={k: v[a:b] for k, v in out.items()}, turn_stats=ts,
                                                dev_status=status, workspace=ws, profile=prof)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["state"] = stride.state_to_numpy(st)[: lay.n_traj]
    res["turn_stats"] = stride.turn_stats_to_numpy(ts)[: lay.n_turns]
    res["status"] = int(status.item())
    res["profile"] = prof.cpu().numpy()
    return res


def test_multi_teacher_equals_aligned_and_oracle(stride, case):
    import torch

    lay = case["lay"]
    R = lay.rows
    aligned = run_batch(stride, case["S"], case["T"], case["tok"], lay, stride.TURN_MEAN, case["lam"])
    multi = _run_multi(stride, case, [(0, R)])
    chunked = _run_multi(stride, case, [(a, min(R, a + 4096)) for a in range(0, R, 4096)])
    for g in (multi, chunked):
        assert g["status"] == 0
        for k in stride.ROW_OUTPUT_KEYS:
            assert np.array_equal(g[k], aligned[k]), k  # per-row results do not depend on where T lives
        assert np.array_equal(g["state"]["stop_row"], aligned["state"]["stop_row"])
        assert np.array_equal(g["turn_stats"]["n"], aligned["turn_stats"]["n"])
    Sh = case["S"].view(torch.int16).cpu().numpy().view(np.uint16)
    Th = case["T"].view(torch.int16).cpu().numpy().view(np.uint16)
    o = oracle.row_logprobs(Sh, Th, case["tok"].cpu().numpy())
    o.update(oracle.scan_batch(o["logp_t"], o["d"], lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                               oracle.TURN_MEAN, float(case["lam"]), logp_s=o["logp_s"]))
    for g in (multi, chunked):
        compare_rows(g, o)
        compare_scan(g, o, lay, oracle.TURN_MEAN, case["lam"])
    assert int((multi["state"]["stop_row"] >= 0).sum()) > 0, "the stop rule should fire"


def test_multi_teacher_bad_rows_report(stride, case):
    import torch

    lay = case["lay"]
    c = dict(case)
    c["dom"] = case["dom"].copy()
    c["dom"][2] = 5  # no such domain
    c["row0"] = case["row0"].copy()
    c["row0"][4] = 10**9  # beyond its domain buffer
    g = _run_multi(stride, c, [(0, lay.rows)])
    assert g["status"] & stride.DEV_BAD_LAYOUT
    with pytest.raises(stride.StrideError) as e:
        offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
        stride.stride_score_batch_multi_teacher(
            case["S"], case["T_dom"], torch.from_numpy(case["dom"]).cuda(), torch.from_numpy(case["row0"]).cuda(),
            case["tok"], *offs, 0, lay.rows, 0, -1.0, stride.new_state(lay.n_traj),
            workspace=torch.empty(stride.stride_score_batch_workspace_size(lay.rows), dtype=torch.uint8,
                                  device="cuda"))
    assert e.value.code == 3  # the row table needs 8 more bytes per row


@pytest.mark.parametrize("kernel", ["auto", "stream", "split", "rows"])
def test_eight_domains_scattered_rows(stride, kernel):
    """The largest domain table (8 buffers of different lengths, two of them
    unused), trajectories reading their teacher rows from random offsets of
    their domain's buffer (ranges may overlap: the buffers are read only),
    in one window and in three; against the oracle on the teacher rows
    gathered by hand.  A ninth domain is rejected before any launch."""
    import torch

    rng = np.random.default_rng(88)
    lens = [[int(rng.integers(2, 90)) for _ in range(int(rng.integers(1, 5)))] for _ in range(12)]
    lay = synth.layout_from_turn_lengths(lens)
    R, V = lay.rows, 2048
    n_rows = np.diff(lay.traj_row_off)
    S = synth.bf16_bits_from_f32(rng.standard_normal((R, V), dtype=np.float32) * np.float32(3.0))
    dom = rng.choice([0, 1, 2, 4, 5, 7], size=lay.n_traj).astype(np.uint8)  # domains 3 and 6 unused
    L = [int(n_rows.max()) + int(rng.integers(0, 400)) for _ in range(8)]
    bufs = [synth.bf16_bits_from_f32(rng.standard_normal((L[d], V), dtype=np.float32) * np.float32(3.0))
            for d in range(8)]
    row0 = np.array([int(rng.integers(0, L[dom[i]] - n_rows[i] + 1)) for i in range(lay.n_traj)], np.int64)
    T = np.concatenate([bufs[dom[i]][row0[i]:row0[i] + n_rows[i]] for i in range(lay.n_traj)])
    tok = rng.integers(0, V, R).astype(np.int32)
    o0 = oracle_batch_multi(S, T, tok, lay, -1e30)
    lam = np.float32(np.median(o0["traj_cum"]))
    o = oracle_batch_multi(S, T, tok, lay, lam)

    def dev_bf16(a):
        return torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)

    c = dict(lay=lay, S=dev_bf16(S), tok=torch.from_numpy(tok).cuda(), dom=dom, row0=row0,
             T_dom=[dev_bf16(b) for b in bufs], lam=lam)
    stride.stride_force_batch_kernel(kernel)
    try:
        for windows in ([(0, R)], [(0, R // 3), (R // 3, (2 * R) // 3), ((2 * R) // 3, R)]):
            g = _run_multi(stride, c, windows)
            assert g["status"] == 0
            compare_rows(g, o)
            compare_scan(g, o, lay, oracle.TURN_MEAN, lam)
    finally:
        stride.stride_force_batch_kernel("auto")
    offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    ws = torch.empty(stride.multi_teacher_workspace_size(R), dtype=torch.uint8, device="cuda")
    with pytest.raises(stride.StrideError) as e:
        stride.stride_score_batch_multi_teacher(c["S"], c["T_dom"] + [c["T_dom"][0]], torch.from_numpy(dom).cuda(),
                                                torch.from_numpy(row0).cuda(), c["tok"], *offs, 0, R,
                                                stride.TURN_MEAN, float(lam), stride.new_state(lay.n_traj),
                                                workspace=ws)
    assert e.value.code == stride.ERR_INVALID_ARG


def oracle_batch_multi(S, T, tok, lay, lam):
    from gpu_helpers import oracle_batch

    return oracle_batch(S, T, tok, lay, oracle.TURN_MEAN, np.float32(lam))
