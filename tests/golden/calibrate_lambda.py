"""Writes tests/golden/lambda_calibration.json: the stop threshold lambda of
each ragged bf16 workload, chosen with the oracle only.

The paper sets lambda per domain by the token length of the generation unit
(Sec. 4.1, "The lambda control surface") and its values (-1 to -3, Tables 1-3)
fit per-token teacher log-probs near -0.7 (Observation 1).  The synthetic
teachers score tokens near -4 to -8, so paper-scale values do not transfer.
The reading used here: turn-mean mode (Eq. 5), lambda halfway between two
adjacent sorted values of S_{n-1} (the running sum over all turns but the
last) across the workload's trajectories, at the 40% quantile, so that about
40% of trajectories stop before their last turn and lambda sits far from any
trajectory's running sum (outside the 1e-3 tie band).

Run on a GPU machine (the inputs are generated there with torch):
  python tests/golden/calibrate_lambda.py [--out PATH] [--only NAME ...]
"""
from __future__ import annotations

import argparse
import json
import sys
import time
from pathlib import Path

import numpy as np

ROOT = Path(__file__).resolve().parents[2]
sys.path.insert(0, str(ROOT))

import oracle  # noqa: E402
import synth  # noqa: E402

QUANTILE = 0.4


def teacher_logprobs(w, device="cuda", chunk=4096) -> np.ndarray:
    import torch

    R = w.layout.rows
    lp = np.empty(R)
    lib = oracle.get()
    for r0 in range(0, R, chunk):
        r1 = min(R, r0 + chunk)
        _, T, tok = synth.generate_rows(w.recipe, r0, r1 - r0, device=device)
        Th = T.view(torch.int16).cpu().numpy().view(np.uint16)
        o = lib.row_logprobs(None, Th, tok.cpu().numpy())
        lp[r0:r1] = o["logp_t"]
        del T, tok, Th
    return lp


def calibrate(w, lp: np.ndarray) -> dict:
    lay = w.layout
    sc = oracle.scan_batch(lp, None, lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off,
                           oracle.TURN_MEAN, -1e300)
    last = lay.traj_turn_off[1:] - 1
    s_prev = sc["turn_cum"][last - 1]  # every workload here has >= 2 turns per trajectory
    v = np.sort(s_prev)
    k = int(round(QUANTILE * len(v)))
    lam = np.float32(0.5 * (v[k - 1] + v[k]))
    frac = float(np.mean(s_prev < float(lam)))
    gap = float(np.min(np.abs(sc["turn_cum"] - float(lam))))
    return {"lambda": float(lam), "quantile": QUANTILE, "early_stop_fraction": frac,
            "min_distance_to_any_turn_sum": gap, "trajectories": lay.n_traj, "rows": lay.rows}


def main():
    import torch

    ap = argparse.ArgumentParser()
    ap.add_argument("--out", default=str(ROOT / "tests" / "golden" / "lambda_calibration.json"))
    ap.add_argument("--only", nargs="*")
    args = ap.parse_args()
    out = Path(args.out)
    res = json.loads(out.read_text()) if out.exists() else {}
    for make in (synth.batch_scoring, synth.long_agentic, synth.multi_teacher):
        w = make()
        if args.only and w.name not in args.only:
            continue
        t0 = time.time()
        lp = teacher_logprobs(w)
        r = calibrate(w, lp)
        r["torch"] = torch.__version__
        r["oracle_seconds"] = time.time() - t0
        res[w.name] = r
        print(w.name, r, flush=True)
        out.write_text(json.dumps(res, indent=1) + "\n")


if __name__ == "__main__":
    main()
