"""The scoring calls at the largest vocabulary they accept, STRIDE_MAX_VOCAB
= 2^30 logits per row (4 GB of S and T for two bf16 rows, 8 GB for one fp32
row): every batch kernel, both decode-step forms and the vocabulary-shard
pass, on 16-byte-aligned rows and on rows that are not (V = 2^30 - 3, row
stride V).  Every logit of a row equals c except the sampled token's, c +
delta, placed near the row's end (in its last whole vector, or in the
ragged tail), so a closed form gives the results at this size:
lse = c + ln(V - 1 + e^delta), logp(y) = delta - ln(V - 1 + e^delta).  One
column more is rejected before any launch."""
import math

import numpy as np
import pytest

import synth
from gpu_helpers import LOGP_ATOL, run_batch

pytestmark = pytest.mark.gpu

VMAX = 1 << 30
C_S, D_S = 0.5, 4.0    # student: every logit 0.5, the token's 4.5 (bf16-exact)
C_T, D_T = -1.0, 2.0   # teacher: every logit -1, the token's 1


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    assert s.MAX_VOCAB == VMAX
    return s


def _expect(V):
    ls = C_S + math.log(V - 1 + math.exp(D_S))
    lt = C_T + math.log(V - 1 + math.exp(D_T))
    return {"lse_s": ls, "lse_t": lt, "x_s": C_S + D_S, "x_t": C_T + D_T,
            "logp_s": C_S + D_S - ls, "logp_t": C_T + D_T - lt, "opd": (C_S + D_S - ls) - (C_T + D_T - lt)}


def _rows(torch, dtype, n_rows, V, ld, ys):
    """[n_rows, V] views (row stride ld) of fresh S and T buffers with the
    closed-form pattern; ys: the token column of each row."""
    S = torch.full((n_rows * ld,), C_S, dtype=dtype, device="cuda")
    T = torch.full((n_rows * ld,), C_T, dtype=dtype, device="cuda")
    for r, y in enumerate(ys):
        S[r * ld + y] = C_S + D_S
        T[r * ld + y] = C_T + D_T
    Sv = S.as_strided((n_rows, V), (ld, 1))
    Tv = T.as_strided((n_rows, V), (ld, 1))
    tok = torch.tensor(ys, dtype=torch.int32, device="cuda")
    return Sv, Tv, tok


def _check_rows(g, V, keys):
    e = _expect(V)
    for k in keys:
        got = np.asarray(g[k], np.float64)
        assert np.all(np.abs(got - e[k]) <= LOGP_ATOL), (k, got, e[k])


CASES = [
    # (dtype, rows, V, ld, token columns): aligned rows, tokens in the last
    # and the second-to-last vector; unaligned rows (odd stride), tokens in
    # the ragged tail; one fp32 row (4 GB per tensor: the one-CTA-per-row
    # kernel, past the persistent kernel's 2 GB row limit)
    ("bf16", 2, VMAX, VMAX + 8, [VMAX - 1, VMAX - 9]),
    ("bf16", 2, VMAX - 3, VMAX - 3, [VMAX - 4, VMAX - 7]),
    ("f32", 1, VMAX, VMAX + 4, [VMAX - 2]),
]


@pytest.mark.parametrize("case", range(len(CASES)))
def test_batch_every_kernel_at_max_vocab(stride, case):
    import torch

    dt, n, V, ld, ys = CASES[case]
    dtype = torch.bfloat16 if dt == "bf16" else torch.float32
    S, T, tok = _rows(torch, dtype, n, V, ld, ys)
    lay = synth.layout_from_turn_lengths([[n]])
    try:
        for kernel in ("auto", "stream", "split", "rows"):
            stride.stride_force_batch_kernel(kernel)
            g = run_batch(stride, S, T, tok, lay, 1, np.float32(-1e30), V=V)
            assert g["status"] == 0, kernel
            _check_rows(g, V, ("logp_s", "logp_t", "opd", "lse_s", "lse_t", "x_s", "x_t"))
            assert int(g["state"]["rows_seen"][0]) == n and int(g["state"]["stop_row"][0]) == -1
    finally:
        stride.stride_force_batch_kernel("auto")
        del S, T
        torch.cuda.empty_cache()


@pytest.mark.parametrize("case", [0, 1])
def test_steps_at_max_vocab(stride, case):
    import torch

    dt, n, V, ld, ys = CASES[case]
    S, T, tok = _rows(torch, torch.bfloat16, n, V, ld, ys)
    try:
        te = torch.zeros(n, dtype=torch.uint8, device="cuda")
        for compact in (False, True):
            st = stride.new_state(n)
            out = {k: torch.full((n,), float("nan"), dtype=torch.float32, device="cuda")
                   for k in ("logp_s", "logp_t", "opd")}
            status = torch.zeros(1, dtype=torch.int32, device="cuda")
            if compact:
                idx = torch.arange(n, dtype=torch.int32, device="cuda")
                stride.stride_score_step_compact(S, T, tok, te, idx, 1, float("-inf"), st, out=out,
                                                 dev_status=status, V=V)
            else:
                stride.stride_score_step(S, T, tok, te, 1, float("-inf"), st, out=out, dev_status=status, V=V)
            torch.cuda.synchronize()
            assert int(status.item()) == 0
            _check_rows({k: v.cpu().numpy() for k, v in out.items()}, V, ("logp_s", "logp_t", "opd"))
            s = stride.state_to_numpy(st)
            assert np.all(np.abs(s["cum"][:n] - _expect(V)["logp_t"]) <= LOGP_ATOL)
    finally:
        del S, T
        torch.cuda.empty_cache()


def test_shard_pass_at_max_vocab(stride):
    import torch

    dt, n, V, ld, ys = CASES[0]
    S, T, tok = _rows(torch, torch.bfloat16, n, V, ld, ys)
    try:
        parts = torch.empty((1, n, 6), dtype=torch.float32, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        stride.stride_partial_lse(S, T, tok, 0, parts[0], dev_status=status, V_shard=V)
        lp_s = torch.empty(n, dtype=torch.float32, device="cuda")
        lp_t = torch.empty(n, dtype=torch.float32, device="cuda")
        stride.stride_combine_partials(parts, logp_s=lp_s, logp_t=lp_t, dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        _check_rows({"logp_s": lp_s.cpu().numpy(), "logp_t": lp_t.cpu().numpy()}, V, ("logp_s", "logp_t"))
        # one column more: rejected before any launch
        with pytest.raises(stride.StrideError) as e:
            stride.stride_partial_lse(S, T, tok, 0, parts[0], V_shard=VMAX + 1)
        assert e.value.code == stride.ERR_INVALID_ARG
        lay = synth.layout_from_turn_lengths([[n]])
        offs = [torch.from_numpy(a).cuda() for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
        ws = torch.empty(stride.stride_score_batch_workspace_size(n), dtype=torch.uint8, device="cuda")
        with pytest.raises(stride.StrideError) as e:
            stride.stride_score_batch(S, T, tok, *offs, 0, n, 1, -1.0, stride.new_state(1), workspace=ws,
                                      V=VMAX + 1)
        assert e.value.code == stride.ERR_INVALID_ARG
        with pytest.raises(stride.StrideError) as e:
            stride.stride_score_step(S, T, tok, torch.zeros(n, dtype=torch.uint8, device="cuda"), 1, -1.0,
                                     stride.new_state(n), V=VMAX + 1)
        assert e.value.code == stride.ERR_INVALID_ARG
    finally:
        del S, T
        torch.cuda.empty_cache()
