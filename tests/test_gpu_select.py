"""GPU parity of stride_select_restart against the oracle: bit-exact k* and
K_max (the inputs are fp32 records; both sides compare in fp32)."""
from __future__ import annotations

import json
import math
from pathlib import Path

import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu
GOLD = Path(__file__).resolve().parent / "golden"


@pytest.fixture(scope="module")
def stride():
    import paper_2609_14636_gb300 as s

    return s


def _run(stride, means, n_turns, mask, alpha):
    import torch

    m = torch.from_numpy(np.ascontiguousarray(means, np.float32)).cuda()
    nt = torch.from_numpy(np.ascontiguousarray(n_turns, np.int32)).cuda()
    mk = None if mask is None else torch.from_numpy(np.ascontiguousarray(mask, np.uint8)).cuda()
    ks = torch.full((means.shape[0],), -7, dtype=torch.int32, device="cuda")
    km = torch.full((means.shape[0],), -7, dtype=torch.int32, device="cuda")
    stride.stride_select_restart(m, nt, mk, alpha, ks, km)
    torch.cuda.synchronize()
    return ks.cpu().numpy(), km.cpu().numpy()


def _f(x):
    return {"-inf": -math.inf, "nan": math.nan}.get(x, x) if isinstance(x, str) else float(x)


def test_select_golden(stride):
    for c in json.loads((GOLD / "select_cases.json").read_text())["cases"]:
        means = np.array([[_f(v) for v in c["means"]]], np.float32)
        nt = np.array([c.get("n_turns", means.shape[1])], np.int32)
        mask = None if c["mask"] is None else np.array([c["mask"]], np.uint8)
        ks, km = _run(stride, means, nt, mask, _f(c["alpha"]))
        assert (int(ks[0]), int(km[0])) == (c["k_star"], c["k_max"]), c["name"]


@pytest.mark.parametrize("mask_key", ["p50", "p90", None])
@pytest.mark.parametrize("alpha", [-math.inf, -6.0, -4.5])
def test_select_prefix_buffer_records(stride, mask_key, alpha):
    """10,000 stored records x 12 turns, 5% quantised values (exact ties),
    10% shorter records, masks Bernoulli(0.5) / Bernoulli(0.9) / none."""
    w = synth.multi_teacher()
    means, nt = w.extra["buffer_means"], w.extra["buffer_n_turns"]
    mask = None if mask_key is None else w.extra["buffer_masks"][mask_key]
    ks, km = _run(stride, means, nt, mask, alpha)
    oks, okm = oracle.select_restart(means, nt, mask, alpha)
    assert np.array_equal(km, okm) and np.array_equal(ks, oks)


@pytest.mark.parametrize("T_max", [1, 31, 32, 33, 100])
def test_select_long_records(stride, T_max):
    rng = np.random.default_rng(T_max)
    N = 3000
    means = np.round(rng.standard_normal((N, T_max)) * 2, 1).astype(np.float32)
    mask = (rng.random((N, T_max)) < 0.97).astype(np.uint8)
    nt = rng.integers(0, T_max + 1, N).astype(np.int32)
    for alpha in (-math.inf, -2.5):
        ks, km = _run(stride, means, nt, mask, alpha)
        oks, okm = oracle.select_restart(means, nt, mask, alpha)
        assert np.array_equal(km, okm) and np.array_equal(ks, oks)
