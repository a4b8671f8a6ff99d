"""Benchmark of the STRIDE scoring path on GB300.

One step = one pass of the whole scoring path over the batch-scoring
workload: 64 trajectories x 8 turns, turn lengths U{64..512} (148,909 rows),
V = 151,936 bf16 student and teacher logits resident in HBM (90.5 GB, far
more than L2, so no flush is needed between steps).  A step initialises the
per-trajectory state and runs stride_score_batch over all rows (per-row
log-probs, OPD signal, turn statistics, running turn-mean sum, first
crossing of lambda).

Reported: scored tokens/s (device-timed, CUDA events on the launching
stream), the same metric end to end through the C ABI from pinned host
buffers (host->device copy of the step's logits and tokens, device->host
copy of its results), the roofline of the fused scoring kernel against the
measured HBM copy bandwidth, and the fp64 CPU oracle timed on this host's
cores on a bounded sample.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (under torchrun) every rank scores its own replica of the
workload; there is no collective on the data path ("weak" scaling).
--impl reference times the oracle (the only reference this path has) on a
bounded sample per step.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time
from pathlib import Path

import numpy as np

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = "scored tokens/sec and achieved HBM GB/s (% of GB300 peak) at V=151,936 bf16"  # value: tokens/s; GB/s and its fraction: roofline
UNIT = "tokens/s"


def algorithmic_bytes_per_row(V: int, elem: int = 2) -> int:
    # S row + T row read once, token id read, three fp32 outputs written,
    # ~8 B amortised per-turn / per-trajectory state and statistics
    return 2 * V * elem + 4 + 12 + 8


def measured_peaks() -> dict:
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        return json.loads(p.read_text())
    return {}


def kernel_traffic_record() -> tuple[float | None, str]:
    """DRAM traffic per launch of the fused kernel from the committed ncu
    summary, valid only while the kernel source is unchanged."""
    src = ROOT / "paper_2609_14636_gb300" / "csrc"
    h = hashlib.sha256()
    for f in ("score_batch_stream.cu", "row_scan.cuh", "stride_device.cuh", "mbarrier.cuh"):
        h.update((src / f).read_bytes())
    digest = h.hexdigest()[:16]
    rec = ROOT / "profiles" / "score_batch_traffic.txt"
    if not rec.exists():
        return None, digest
    kv = {}
    for line in rec.read_text().splitlines():
        if ":" in line:
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    if kv.get("source_sha256_16") != digest:
        return None, digest
    try:
        return float(kv["dram_bytes_per_row"]), digest
    except (KeyError, ValueError):
        return None, digest


class ClockSampler:
    """nvidia-smi clock / throttle sampling while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = Path(os.environ.get("TMPDIR", "/tmp")) / f"stride_clocks_{os.getpid()}.csv"

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self) -> dict:
        if self.proc is None or not self.path.exists():
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["clock sampling unavailable"]}
        rows = [l.split(",") for l in self.path.read_text().splitlines() if l.strip()]
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax = float(r[2])
            except ValueError:
                continue
            for n, v in zip(names, r[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        try:
            self.path.unlink()
        except OSError:
            pass
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


def max_over_ranks(ms: float, device=None) -> float:
    """The slowest rank's time (the whole job finishes when it does)."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(rows_per_rank: int, world: int, ms_per_step: float) -> float:
    """Tokens scored by all ranks per second of the slowest rank's step."""
    return world * rows_per_rank / (ms_per_step * 1e-3)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def cpu_oracle_rate(S_dev, T_dev, tok_dev, lay, lam, budget_s: float, chunk: int = 1024) -> dict:
    """Oracle rows/s on a bounded sample: consecutive 1,024-row chunks of the
    workload, copied device->host, until ~budget_s of oracle time."""
    import oracle
    import torch

    lib = oracle.get()
    threads = oracle.default_threads()
    rows_done, t_oracle = 0, 0.0
    R = S_dev.shape[0]
    r0 = 0
    while t_oracle < budget_s and r0 < R:
        r1 = min(R, r0 + chunk)
        Sh = S_dev[r0:r1].view(torch.int16).cpu().numpy().view(np.uint16)
        Th = T_dev[r0:r1].view(torch.int16).cpu().numpy().view(np.uint16)
        th = tok_dev[r0:r1].cpu().numpy()
        t0 = time.perf_counter()
        o = lib.row_logprobs(Sh, Th, th, nthreads=threads)
        t_oracle += time.perf_counter() - t0
        rows_done += r1 - r0
        r0 = r1
        del Sh, Th, o
    return {"value": rows_done / t_oracle, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"first {rows_done} rows of the workload (fp64 log-softmax gather of S and T, "
                      f"{threads} threads), {t_oracle:.1f} s"}


def run_reference(args) -> None:
    """--impl reference: the fp64 CPU oracle, as it stands, on a bounded
    sample of the workload per step (1,024 rows of its logits)."""
    ws, rank, local = dist_env()
    if rank != 0:
        return
    import torch

    import oracle
    import synth

    w = synth.batch_scoring()
    rows = 1024
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    S, T, tok = synth.generate_rows(w.recipe, 0, rows, device=dev)
    Sh = S.view(torch.int16).cpu().numpy().view(np.uint16)
    Th = T.view(torch.int16).cpu().numpy().view(np.uint16)
    th = tok.cpu().numpy()
    lay = synth.layout_from_turn_lengths([[rows]])
    lib = oracle.get()
    threads = oracle.default_threads()
    lam = float(load_lambda(w)[0])

    def step():
        o = lib.row_logprobs(Sh, Th, th, nthreads=threads)
        lib.scan_batch(o["logp_t"], o["d"], lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off, 0, lam)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    value = rows * args.steps / dt
    line = {"metric": METRIC, "value": value, "unit": UNIT, "impl": "reference", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": w.name, "sample_rows_per_step": rows},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"{rows} rows of the workload per step, fp64 oracle, {threads} threads"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def load_lambda(w) -> np.ndarray:
    """Per-trajectory lambda: the oracle calibration of the workload
    (tests/golden/lambda_calibration.json), else its provisional value."""
    import synth

    return np.full(w.layout.n_traj, np.float32(synth.workload_lambda(w.name)), np.float32)


WORKLOADS = ("batch_scoring", "long_agentic", "multi_teacher", "decode_step", "select", "tiny_reference",
             "vocab_parallel")


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=WORKLOADS, default="batch_scoring",
                    help="batch_scoring is the headline; the others measure the remaining rows of the path")
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--e2e-rows", type=int, default=8192)
    ap.add_argument("--max-rows", type=int, default=0,
                    help="score only the leading whole trajectories that fit (small profiling cases)")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
        return
    if args.workload == "decode_step":
        run_decode(args)
    elif args.workload == "tiny_reference":
        run_tiny(args)
    elif args.workload == "select":
        run_select(args)
    elif args.workload == "vocab_parallel":
        run_vocab_parallel(args)
    else:
        run_batch(args)


def _setup_rank():
    import torch

    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    return ws, rank, local, torch.device("cuda", local)


def _common_line(args, ws, ms_step, value, unit=UNIT, metric=METRIC, dtype="bf16"):
    return {"metric": metric, "value": value, "unit": unit, "n_gpus": ws, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": dtype, "data": "synthetic"}


def run_batch(args) -> None:
    """Ragged batch scoring: the headline workload (all rows in one window), or
    the long-agentic / multi-teacher workloads resident in HBM and scored in
    their 16,384-row windows with the carried state."""
    import torch

    ws, rank, local, dev = _setup_rank()
    if ws > 1:
        import torch.distributed as dist

    import paper_2609_14636_gb300 as stride
    import synth

    w = {"batch_scoring": synth.batch_scoring, "long_agentic": synth.long_agentic,
         "multi_teacher": synth.multi_teacher}[args.workload]()
    lay = w.layout
    if args.max_rows > 0:
        lay = synth.sub_layout(lay, synth.first_trajectories(lay, args.max_rows))
    R, V = lay.rows, w.recipe.V
    lam = load_lambda(w)[: lay.n_traj]

    # ---- workload resident in HBM --------------------------------------
    S = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
    T = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
    tok = torch.empty(R, dtype=torch.int32, device=dev)
    t_gen = time.perf_counter()
    CH = 8192
    for r0 in range(0, R, CH):
        r1 = min(R, r0 + CH)
        synth.generate_rows(w.recipe, r0, r1 - r0, device=dev, out_S=S[r0:r1], out_T=T[r0:r1], out_tok=tok[r0:r1])
    torch.cuda.synchronize()
    t_gen = time.perf_counter() - t_gen
    offs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    lam_d = torch.from_numpy(lam).to(dev)
    st = stride.new_state(lay.n_traj, dev)
    ts = stride.new_turn_stats(lay.n_turns, dev)
    out = {k: torch.empty(R, dtype=torch.float32, device=dev) for k in ("logp_s", "logp_t", "opd")}
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    chunk = int(w.extra.get("chunk_rows", R))
    windows = [(a, min(R, a + chunk)) for a in range(0, R, chunk)]
    wsb = torch.empty(stride.stride_score_batch_workspace_size(min(chunk, R)), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step(ev=None):
        stride.stride_state_init(st, lay.n_traj, stream)
        if ev is not None:
            ev[0].record(stream)
        for a, b in windows:
            stride.stride_score_batch(S[a:b], T[a:b], tok[a:b], *offs, a, b, stride.TURN_MEAN, lam_d, st,
                                      out={k: v[a:b] for k, v in out.items()}, turn_stats=ts,
                                      dev_status=status, workspace=wsb, stream=stream)
        if ev is not None:
            ev[1].record(stream)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())} after warm-up")
    early = stride.state_to_numpy(st)[: lay.n_traj]
    n_turns_traj = np.diff(lay.traj_turn_off)
    early_frac = float(np.mean((early["stop_turn"] >= 0) & (early["stop_turn"] < n_turns_traj - 1)))

    # ---- device-timed steps ---------------------------------------------
    kev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        time.sleep(0.25)
        e0.record(stream)
        for i in range(args.steps):
            step(kev[i])
        e1.record(stream)
        torch.cuda.synchronize()
        time.sleep(0.05)
    if ws > 1:
        dist.barrier()
    ms_total = max_over_ranks(e0.elapsed_time(e1), dev)
    k_ms = [a.elapsed_time(b) for a, b in kev]
    ms_step = ms_total / args.steps
    value = whole_job_rate(R, ws, ms_step)

    # the same scoring calls with the within-turn profile (Observation 1)
    # accumulated too, outside the timed steps above
    prof = stride.new_profile(dev)
    pev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(5)]
    for a, b in pev:
        stride.stride_state_init(st, lay.n_traj, stream)
        a.record(stream)
        for wa, wb in windows:
            stride.stride_score_batch(S[wa:wb], T[wa:wb], tok[wa:wb], *offs, wa, wb, stride.TURN_MEAN, lam_d, st,
                                      out={k: v[wa:wb] for k, v in out.items()}, turn_stats=ts,
                                      dev_status=status, workspace=wsb, stream=stream, profile=prof)
        b.record(stream)
    torch.cuda.synchronize()
    ms_with_profile = statistics.mean(a.elapsed_time(b) for a, b in pev)

    # ---- roofline of the fused kernel -------------------------------------
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs", 6800.0)
    bpr = algorithmic_bytes_per_row(V)
    k_avg = statistics.mean(k_ms)  # all windows of one step
    achieved = bpr * R / (k_avg * 1e-3) / 1e9
    dram_per_row, digest = kernel_traffic_record()
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": None if dram_per_row is None else dram_per_row * R,
                "algorithmic_bytes_per_launch": bpr * R, "kernel_ms_mean": k_avg,
                "kernel_ms_min": min(k_ms), "kernel": "score_batch_stream_kernel<bf16>",
                "kernel_ms_mean_with_profile": ms_with_profile,
                "peak_source": "MEASURED_PEAKS.json hbm_gbs (of measured)" if "hbm_gbs" in peaks else "fallback 6.8 TB/s"}

    # ---- end to end from pinned host buffers ------------------------------
    e2e = None
    if rank == 0 or ws > 1:
        # the first trajectories up to e2e_rows rows, as a caller holding them in host memory would
        n_tr = int(np.searchsorted(lay.traj_row_off, args.e2e_rows, side="right") - 1)
        n_tr = max(1, min(n_tr, lay.n_traj))
        Re = int(lay.traj_row_off[n_tr])
        n_tu = int(lay.traj_turn_off[n_tr])
        hS = torch.empty((Re, V), dtype=torch.bfloat16, pin_memory=True)
        hT = torch.empty((Re, V), dtype=torch.bfloat16, pin_memory=True)
        hk = torch.empty(Re, dtype=torch.int32, pin_memory=True)
        hS.copy_(S[:Re])
        hT.copy_(T[:Re])
        hk.copy_(tok[:Re])
        hout = {k: torch.empty(Re, dtype=torch.float32, pin_memory=True) for k in out}
        hst = torch.empty((n_tr, stride.STATE_DTYPE.itemsize), dtype=torch.uint8, pin_memory=True)
        hts = torch.empty((n_tu, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, pin_memory=True)
        dS, dT, dk = S[:Re], T[:Re], tok[:Re]  # device landing buffers (the resident workload's first rows)
        eoffs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off[: n_tr + 1], lay.turn_row_off[: n_tu + 1],
                                                        lay.traj_turn_off[: n_tr + 1])]
        est = stride.new_state(n_tr, dev)
        ets = stride.new_turn_stats(n_tu, dev)
        eout = {k: v[:Re] for k, v in out.items()}

        # Host->device copies of window i+1 (copy stream) overlap the scoring of
        # window i (compute stream); the carried state makes the windows exact.
        ew = min(1024, chunk)
        ewin = [(a, min(Re, a + ew)) for a in range(0, Re, ew)]
        cstream = torch.cuda.Stream(device=dev)
        landed = [torch.cuda.Event() for _ in ewin]

        def e2e_step():
            go = torch.cuda.Event()
            go.record(stream)  # the previous step's kernels are done with the landing buffers
            cstream.wait_event(go)
            with torch.cuda.stream(cstream):
                for i, (a, b) in enumerate(ewin):
                    dS[a:b].copy_(hS[a:b], non_blocking=True)
                    dT[a:b].copy_(hT[a:b], non_blocking=True)
                    dk[a:b].copy_(hk[a:b], non_blocking=True)
                    landed[i].record(cstream)
            stride.stride_state_init(est, n_tr, stream)
            for i, (a, b) in enumerate(ewin):
                stream.wait_event(landed[i])
                stride.stride_score_batch(dS[a:b], dT[a:b], dk[a:b], *eoffs, a, b, stride.TURN_MEAN, lam_d[:n_tr],
                                          est, out={k: v[a:b] for k, v in eout.items()}, turn_stats=ets,
                                          dev_status=status, workspace=wsb, stream=stream)
            for k in hout:
                hout[k].copy_(eout[k], non_blocking=True)
            hst.copy_(est[:n_tr], non_blocking=True)
            hts.copy_(ets[:n_tu], non_blocking=True)

        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        # Each step is timed on its own and the median reported: the host link
        # is shared with the rest of the machine, and a transient stall of one
        # step should not stand for the path.
        n_e = max(3, min(args.steps, 7))
        e_evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_e)]
        for a, b in e_evs:
            a.record(stream)
            e2e_step()
            b.record(stream)
        torch.cuda.synchronize()
        e_all = sorted(a.elapsed_time(b) for a, b in e_evs)
        e_ms = statistics.median(e_all)
        h2d = 2 * Re * V * 2 + Re * 4
        d2h = Re * 4 * len(hout) + n_tr * stride.STATE_DTYPE.itemsize + n_tu * stride.TURN_STATS_DTYPE.itemsize
        e2e = {"value": ws * Re / (e_ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": e_ms, "ms_per_step_min": e_all[0], "ms_per_step_max": e_all[-1],
               "timing": f"median of {n_e} steps, each timed on its own", "windows": len(ewin),
               "sample": f"first {n_tr} trajectories ({Re} rows) of the workload held in pinned host memory; H2D of "
                         f"S, T, tokens in {len(ewin)} windows overlapped with scoring, D2H of per-row outputs, "
                         f"state and turn stats, all inside the timed region"}
        del hS, hT

    # ---- oracle on this host's cores (rank 0, N = 1 only) ------------------
    cpu = None
    if rank == 0 and ws == 1:
        cpu = cpu_oracle_rate(S, T, tok, lay, lam, args.cpu_budget)

    if rank == 0:
        clocks = clk.summary()
        line = _common_line(args, ws, ms_step, value)
        line.update({
            "config": {"workload": w.name if args.max_rows <= 0 else f"{w.name} (first {lay.n_traj} trajectories)",
                       "windows": len(windows), "window_rows": chunk,
                       "trajectories": lay.n_traj, "turns": lay.n_turns, "rows": R,
                       "vocab": V, "logits": "bf16 student + bf16 teacher, resident in HBM",
                       "bytes_resident": 2 * R * V * 2, "stop_mode": "turn_mean",
                       "lambda": float(lam[0]), "early_stop_fraction": early_frac,
                       "l2": f"inputs ({2 * R * V * 2 / 1e9:.1f} GB) larger than L2 (129 MB): no flush",
                       "lambda_source": "tests/golden/lambda_calibration.json (oracle, 40% quantile)",
                       "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU",
                       "generation_s": t_gen},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clocks,
            "gpu_launches": (1 + len(windows)) * args.steps,
        })
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.destroy_process_group()


def run_vocab_parallel(args, n_shards: int = 4) -> None:
    """The batch-scoring workload with its logits split by vocabulary into
    n_shards column shards, as a tensor-parallel teacher and student would
    hold them: stride_partial_lse on every shard (each shard a column range
    of the resident [rows, V] buffers, row stride V), stride_combine_partials,
    stride_scan_logprobs.  On one GPU the shards run one after another, so a
    step reads the same logit bytes as the fused path."""
    import torch

    ws, rank, local, dev = _setup_rank()
    import paper_2609_14636_gb300 as stride
    import synth

    w = synth.batch_scoring()
    lay = w.layout
    if args.max_rows > 0:
        lay = synth.sub_layout(lay, synth.first_trajectories(lay, args.max_rows))
    R, V = lay.rows, w.recipe.V
    lam = load_lambda(w)[: lay.n_traj]
    S = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
    T = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
    tok = torch.empty(R, dtype=torch.int32, device=dev)
    for r0 in range(0, R, 8192):
        r1 = min(R, r0 + 8192)
        synth.generate_rows(w.recipe, r0, r1 - r0, device=dev, out_S=S[r0:r1], out_T=T[r0:r1], out_tok=tok[r0:r1])
    offs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    lam_d = torch.from_numpy(lam).to(dev)
    st = stride.new_state(lay.n_traj, dev)
    ts = stride.new_turn_stats(lay.n_turns, dev)
    parts = torch.empty((n_shards, R, 6), dtype=torch.float32, device=dev)
    lps, lpt, opd = (torch.empty(R, dtype=torch.float32, device=dev) for _ in range(3))
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    wsb = torch.empty(stride.stride_score_batch_workspace_size(R), dtype=torch.uint8, device=dev)
    # shard k: columns [cuts[k], cuts[k+1]), cut on 16-byte boundaries
    cuts = [((V * k // n_shards) // 8) * 8 for k in range(n_shards)] + [V]
    stream = torch.cuda.current_stream()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(4)]

    def step(timed=False):
        stride.stride_state_init(st, lay.n_traj, stream)
        if timed:
            evs[0].record(stream)
        for k in range(n_shards):
            c0, c1 = cuts[k], cuts[k + 1]
            stride.stride_partial_lse(S[:, c0:c1], T[:, c0:c1], tok, c0, parts[k], dev_status=status, stream=stream)
        if timed:
            evs[1].record(stream)
        stride.stride_combine_partials(parts, logp_s=lps, logp_t=lpt, dev_status=status, stream=stream)
        if timed:
            evs[2].record(stream)
        stride.stride_scan_logprobs(lps, lpt, *offs, 0, R, stride.TURN_MEAN, lam_d, st, opd=opd, turn_stats=ts,
                                    dev_status=status, workspace=wsb, stream=stream)
        if timed:
            evs[3].record(stream)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}")
    steps = max(1, min(args.steps, 30))
    t_part, t_comb, t_scan = [], [], []
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        time.sleep(0.25)
        e0.record(stream)
        for _ in range(steps):
            step(timed=True)
            torch.cuda.synchronize()
            t_part.append(evs[0].elapsed_time(evs[1]))
            t_comb.append(evs[1].elapsed_time(evs[2]))
            t_scan.append(evs[2].elapsed_time(evs[3]))
        e1.record(stream)
        torch.cuda.synchronize()
        time.sleep(0.05)
    ms_step = max_over_ranks(statistics.mean(a + b + c for a, b, c in zip(t_part, t_comb, t_scan)), dev)
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs", 6800.0)
    part_bytes = R * (2 * V * 2 + n_shards * (4 + 24))  # every shard's logits, tokens, partials written
    part_ms = statistics.mean(t_part)
    achieved = part_bytes / (part_ms * 1e-3) / 1e9
    if rank == 0:
        line = _common_line(args, ws, ms_step, whole_job_rate(R, ws, ms_step))
        line.update({
            "config": {"workload": f"{w.name} in {n_shards} vocabulary shards", "rows": R, "vocab": V,
                       "shards": n_shards, "shard_columns": [cuts[k + 1] - cuts[k] for k in range(n_shards)],
                       "stop_mode": "turn_mean", "lambda": float(lam[0]),
                       "l2": f"inputs ({2 * R * V * 2 / 1e9:.1f} GB) larger than L2 (129 MB): no flush",
                       "timing": "per step: the shards' partial passes, the combine and the scan, each "
                                 "bracketed by CUDA events; the step is their sum (state init excluded)"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": None, "algorithmic_bytes_per_launch": part_bytes / n_shards,
                         "kernel": "partial_lse_kernel<bf16> (one CTA per row and shard)",
                         "ms_partials": part_ms, "ms_combine": statistics.mean(t_comb),
                         "ms_scan": statistics.mean(t_scan),
                         "peak_source": "MEASURED_PEAKS.json hbm_gbs (of measured)" if "hbm_gbs" in peaks
                         else "fallback 6.8 TB/s"},
            "clocks": clk.summary(), "gpu_launches": steps * (1 + n_shards + 2),
        })
        print(json.dumps(line), flush=True)


def _graph(fn):
    """Capture fn() (a sequence of library calls on the current stream) in a
    CUDA graph."""
    import torch

    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn()  # warm: first calls on a device do their one-time set-up here
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    with torch.cuda.graph(g):
        fn()
    torch.cuda.synchronize()
    return g


def decode_compact_schedule(stride, S, T, tok, turn_end, B, ring, lam, dev):
    """Live sets of a compacted decode sweep: run it once step by step,
    reading each step's stop flags back (as a rollout engine does before it
    batches the next step's live sequences).  Step s scores the live
    rollouts' rows as rows 0..n-1 of slab s mod ring.  Returns the per-step
    row counts and the concatenated rollout ids and turn-end flags."""
    import torch

    st = stride.new_state(B, dev)
    sn = torch.empty(B, dtype=torch.uint8, device=dev)
    live = np.arange(B, dtype=np.int32)
    counts, idx, te = [], [], []
    for s in range(turn_end.shape[0]):
        n = live.shape[0]
        counts.append(n)
        if n == 0:
            continue
        j = s % ring
        it = torch.from_numpy(live).to(dev)
        tc = torch.from_numpy(np.ascontiguousarray(turn_end[s][live])).to(dev)
        stride.stride_score_step_compact(S[j * B:j * B + n], T[j * B:j * B + n], tok[j * B:j * B + n], tc, it,
                                         stride.TURN_MEAN, lam, st, stopped_now=sn)
        fired = sn[:n].cpu().numpy()
        idx.append(live.copy())
        te.append(turn_end[s][live])
        live = live[fired == 0]
    return np.array(counts), np.concatenate(idx), np.concatenate(te).astype(np.uint8)


def run_decode(args) -> None:
    """Decode steps: B = 256 rollouts x 4,096 steps, a ring of 16 distinct
    [256, V] step slabs (more bytes than L2), turn ends every U{96..768}
    steps.  Two forms of the same sweep, each replayed as one CUDA graph:
    compacted (stride_score_step_compact over the live rollouts' rows only;
    the reported value) and masked (stride_score_step over all 256 rows,
    stopped rollouts masked).  Also a 64-step all-active graph (lambda =
    -inf), which shows the kernel at full activity."""
    import torch

    ws, rank, local, dev = _setup_rank()
    import paper_2609_14636_gb300 as stride
    import synth

    w = synth.decode_steps()
    B, ring, n_steps = w["B"], w["ring"], w["steps"]
    V = w["recipe"].V
    S, T, tok = synth.generate_rows(w["recipe"], 0, ring * B, device=dev)
    te = torch.from_numpy(w["turn_end"]).to(dev)
    st = stride.new_state(B, dev)
    out = {k: torch.empty(B, dtype=torch.float32, device=dev) for k in ("logp_s", "logp_t", "opd")}
    sn = torch.empty(B, dtype=torch.uint8, device=dev)
    tout = torch.empty((B, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)

    def sweep(lam, steps):
        stride.stride_state_init(st, B)
        for i in range(steps):
            j = i % ring
            stride.stride_score_step(S[j * B:(j + 1) * B], T[j * B:(j + 1) * B], tok[j * B:(j + 1) * B], te[i],
                                     stride.TURN_MEAN, lam, st, out=out, stopped_now=sn, turn_out=tout,
                                     dev_status=status)

    counts, idx_np, te_np = decode_compact_schedule(stride, S, T, tok, w["turn_end"], B, ring, w["lam_turn"], dev)
    idx_all = torch.from_numpy(idx_np).to(dev)
    te_all = torch.from_numpy(te_np).to(dev)
    offs = np.concatenate([[0], np.cumsum(counts)])

    def sweep_compact():
        stride.stride_state_init(st, B)
        for i in range(n_steps):
            n = int(counts[i])
            if n == 0:
                continue
            j, a = i % ring, int(offs[i])
            stride.stride_score_step_compact(S[j * B:j * B + n], T[j * B:j * B + n], tok[j * B:j * B + n],
                                             te_all[a:a + n], idx_all[a:a + n], stride.TURN_MEAN, w["lam_turn"], st,
                                             out=out, stopped_now=sn, turn_out=tout, dev_status=status)

    g_full = _graph(lambda: sweep(float("-inf"), 64))
    g_run = _graph(lambda: sweep(w["lam_turn"], n_steps))
    g_cmp = _graph(sweep_compact)
    stream = torch.cuda.current_stream()
    reps = max(1, min(args.steps, 10))
    for _ in range(max(3, args.warmup)):
        g_full.replay()
    g_run.replay()
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}")
    scored = int(stride.state_to_numpy(st)["rows_seen"][:B].sum())
    g_cmp.replay()
    torch.cuda.synchronize()
    scored_c = int(stride.state_to_numpy(st)["rows_seen"][:B].sum())
    if int(status.item()) != 0 or scored_c != int(counts.sum()):
        raise RuntimeError(f"compacted sweep: status {int(status.item())}, rows {scored_c} vs {int(counts.sum())}")
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(g, n):
        a.record(stream)
        for _ in range(n):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / n

    with ClockSampler(local) as clk:
        time.sleep(0.25)
        ms_cmp = timed(g_cmp, reps)
        ms_sweep = timed(g_run, reps)
        ms_full = timed(g_full, 20)
        time.sleep(0.05)
    ms_cmp = max_over_ranks(ms_cmp, dev)
    ms_sweep = max_over_ranks(ms_sweep, dev)
    bpr = algorithmic_bytes_per_row(V)
    peak = measured_peaks().get("hbm_gbs", 6800.0)
    us_step_full = 1e3 * ms_full / 64
    full_gbs = B * bpr / (us_step_full * 1e-6) / 1e9
    cmp_gbs = scored_c * bpr / (ms_cmp * 1e-3) / 1e9
    value = ws * scored_c / (ms_cmp * 1e-3)
    launched = int((counts > 0).sum())
    if rank == 0:
        line = _common_line(args, ws, ms_cmp, value)
        line.update({
            "config": {"workload": w["name"], "rollouts": B, "decode_steps": n_steps, "ring_slabs": ring,
                       "vocab": V, "stop_mode": "turn_mean", "lambda": w["lam_turn"],
                       "form": "compacted: each step scores only the live rollouts' rows (stride_score_step_compact)",
                       "tokens_scored_per_sweep": scored_c, "steps_with_live_rollouts": launched,
                       "mean_live_rollouts": float(counts.mean()),
                       "live_rollouts_per_launched_step": {
                           q: int(np.percentile(counts[counts > 0], float(q[1:]))) for q in ("p10", "p50", "p90")},
                       "steps_all_live": int((counts == B).sum()),
                       "graph": "one CUDA graph per sweep (state init + one launch per step with live rollouts)",
                       "l2": f"ring of {ring} slabs = {2 * ring * B * V * 2 / 1e9:.2f} GB > L2: no flush"},
            "roofline": {"bound": "hbm", "achieved": cmp_gbs, "peak": peak, "unit": "GB/s", "frac": cmp_gbs / peak,
                         "traffic": None, "kernel": "score_step_kernel<bf16,vec,compact> (cluster size from the step's rows)",
                         "achieved_basis": "algorithmic bytes of the sweep's scored rows / sweep time",
                         "us_per_step_all_active": us_step_full, "all_active_gbs": full_gbs,
                         "all_active_frac": full_gbs / peak,
                         "masked_sweep": {"ms": ms_sweep, "tokens": scored, "tokens_per_s": scored / (ms_sweep * 1e-3),
                                          "gbs": scored * bpr / (ms_sweep * 1e-3) / 1e9,
                                          "frac": scored * bpr / (ms_sweep * 1e-3) / 1e9 / peak},
                         "peak_source": "MEASURED_PEAKS.json hbm_gbs (of measured)"},
            "clocks": clk.summary(), "gpu_launches": reps * (launched + 1) + reps * (n_steps + 1) + 20 * 65,
        })
        print(json.dumps(line), flush=True)


def run_select(args) -> None:
    """Restart choice over the 10,000-record prefix buffer (12 turns, masks
    Bernoulli(0.5), alpha = -6.0): one launch per call, 200 calls per graph."""
    import torch

    ws, rank, local, dev = _setup_rank()
    import paper_2609_14636_gb300 as stride
    import synth

    w = synth.multi_teacher()
    means = torch.from_numpy(w.extra["buffer_means"]).to(dev)
    nt = torch.from_numpy(w.extra["buffer_n_turns"]).to(dev)
    mask = torch.from_numpy(w.extra["buffer_masks"]["p50"]).to(dev)
    N, T_max = means.shape
    ks = torch.empty(N, dtype=torch.int32, device=dev)
    km = torch.empty(N, dtype=torch.int32, device=dev)
    calls = 200
    g = _graph(lambda: [stride.stride_select_restart(means, nt, mask, -6.0, ks, km) for _ in range(calls)])
    stream = torch.cuda.current_stream()
    for _ in range(max(3, args.warmup)):
        g.replay()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = max(1, min(args.steps, 50))
    with ClockSampler(local) as clk:
        time.sleep(0.25)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        time.sleep(0.05)
    us_call = 1e3 * a.elapsed_time(b) / (reps * calls)
    us_call = max_over_ranks(us_call, dev)
    bytes_call = N * T_max * 5 + N * 12

    # the prefix buffer's record step (Algorithm 1): 128 rollouts of 12 turns
    # each recorded into a copy of the buffer, each keeping k0 stored turns
    n_rec, turns_rec = 128, 12
    rng = np.random.default_rng(9)
    rbuf, rnt = means.clone(), nt.clone()
    tasks = torch.from_numpy(rng.choice(N, n_rec, replace=False).astype(np.int32)).to(dev)
    k0 = torch.from_numpy(rng.integers(0, 6, n_rec).astype(np.int32)).to(dev)
    rts = stride.new_turn_stats(n_rec * turns_rec, dev)
    rts_view = rts.view(-1, stride.TURN_STATS_DTYPE.itemsize)
    tt = np.zeros(n_rec * turns_rec, stride.TURN_STATS_DTYPE)
    tt["mean_t"] = rng.normal(-4.5, 1.5, n_rec * turns_rec).astype(np.float32)
    tt["n"] = 100
    rts_view.copy_(torch.from_numpy(tt.view(np.uint8).reshape(n_rec * turns_rec, -1)).to(dev))
    rturn_off = torch.arange(0, n_rec * turns_rec + 1, turns_rec, dtype=torch.int32, device=dev)
    g_rec = _graph(lambda: [stride.stride_buffer_record(rbuf, rnt, tasks, k0, rts, rturn_off) for _ in range(calls)])
    for _ in range(3):
        g_rec.replay()
    a.record(stream)
    for _ in range(reps):
        g_rec.replay()
    b.record(stream)
    torch.cuda.synchronize()
    us_record = 1e3 * a.elapsed_time(b) / (reps * calls)
    if rank == 0:
        line = _common_line(args, ws, us_call / 1e3, ws * N / (us_call * 1e-6), unit="records/s",
                            metric="restart choices/sec (10,000 x 12 records)", dtype="f32")
        line.update({
            "config": {"workload": "prefix_buffer_select_10000x12", "records": N, "turns": T_max,
                       "mask": "Bernoulli(0.5)", "alpha": -6.0, "graph": f"{calls} launches per CUDA graph"},
            "roofline": {"bound": "latency", "achieved": bytes_call / (us_call * 1e-6) / 1e9, "peak": None,
                         "unit": "GB/s", "frac": None, "traffic": None, "us_per_call": us_call,
                         "kernel": "select_restart_kernel (one warp per record)",
                         "record_us_per_call": us_record,
                         "record": f"stride_buffer_record of {n_rec} rollouts x {turns_rec} turns into the "
                                   f"{N}-record buffer (buffer_record_kernel, {calls} launches per graph)"},
            "clocks": clk.summary(), "gpu_launches": 2 * reps * calls,
        })
        print(json.dumps(line), flush=True)


def run_tiny(args) -> None:
    """The tiny reference workload: 1 trajectory x 4 turns x 128 tokens,
    V = 32,000 fp32 logits (131 MB, about the size of L2), token-sum stop
    at lambda = -200.  L2 is flushed (a 512 MB write) before every timed
    step; each step (state init + scoring, captured once in a CUDA graph so
    that host-side submission is not timed) is timed with CUDA events."""
    import torch

    import oracle
    import paper_2609_14636_gb300 as stride
    import synth

    ws, rank, local, dev = _setup_rank()
    w = synth.tiny_reference(0)
    lay = w["layout"]
    R, V = lay.rows, w["V"]
    S = torch.from_numpy(w["S"]).to(dev)
    T = torch.from_numpy(w["T"]).to(dev)
    tok = torch.from_numpy(w["tokens"]).to(dev)
    offs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
    st = stride.new_state(lay.n_traj, dev)
    ts = stride.new_turn_stats(lay.n_turns, dev)
    out = {k: torch.empty(R, dtype=torch.float32, device=dev) for k in ("logp_s", "logp_t", "opd")}
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    wsb = torch.empty(stride.stride_score_batch_workspace_size(R), dtype=torch.uint8, device=dev)
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
    # The 512 MB write leaves L2 full of dirty lines, which the step's reads
    # would then have to write back (a streaming-only kernel over the same
    # 131 MB takes 32.3-32.8 us after it); reading a clean 256 MB buffer
    # after the write evicts them outside the timed region, so the step
    # starts, like the larger workloads (inputs far above L2, no flush),
    # with none of its inputs and no dirty lines in L2.
    clean = torch.ones(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step():  # on the current stream (the capture stream while capturing)
        stride.stride_state_init(st, lay.n_traj)
        stride.stride_score_batch(S, T, tok, *offs, 0, R, stride.TOKEN_SUM, w["lam_token"], st, out=out,
                                  turn_stats=ts, dev_status=status, workspace=wsb)

    g = _graph(step)
    for _ in range(max(3, args.warmup)):
        flush.zero_()
        clean.sum()
        g.replay()
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}")

    def timed(read_after_write: bool) -> float:
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        for a, b in evs:
            flush.zero_()  # L2 flush, outside the timed events
            if read_after_write:
                clean.sum()
            a.record(stream)
            g.replay()
            b.record(stream)
        torch.cuda.synchronize()
        return statistics.mean(a.elapsed_time(b) for a, b in evs)

    with ClockSampler(local) as clk:
        time.sleep(0.25)
        ms = timed(True)
        ms_write_only = timed(False)
        time.sleep(0.05)
    ms = max_over_ranks(ms, dev)
    ms_write_only = max_over_ranks(ms_write_only, dev)
    bpr = algorithmic_bytes_per_row(V, 4)
    peak = measured_peaks().get("hbm_gbs", 6800.0)
    threads = oracle.default_threads()
    t0 = time.perf_counter()
    oracle.row_logprobs(w["S"], w["T"], w["tokens"], nthreads=threads)
    cpu_rate = R / (time.perf_counter() - t0)
    if rank == 0:
        line = _common_line(args, ws, ms, ws * R / (ms * 1e-3), dtype="f32")
        line.update({
            "config": {"workload": w["name"], "rows": R, "vocab": V, "stop_mode": "token_sum",
                       "lambda": w["lam_token"],
                       "l2": "before every timed step 512 MB written, then a clean 256 MB buffer read (inputs "
                             "131 MB; no input and no dirty line left in L2)"},
            "roofline": {"bound": "hbm", "achieved": bpr * R / (ms * 1e-3) / 1e9, "peak": peak, "unit": "GB/s",
                         "frac": bpr * R / (ms * 1e-3) / 1e9 / peak, "traffic": None,
                         "algorithmic_bytes_per_launch": bpr * R,
                         "kernel": "score_batch_split_kernel<f32> (2-CTA clusters, one wave of 1,024 CTAs) "
                                   "+ scan_logprobs_tile_kernel (4 tiles of 128 rows)",
                         "note": "512 rows on 152 SMs: a latency-bound launch; time includes state init",
                         "ms_per_step_write_flush_only": ms_write_only,
                         "frac_write_flush_only": bpr * R / (ms_write_only * 1e-3) / 1e9 / peak},
            "cpu_baseline": {"value": cpu_rate, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"all {R} rows"},
            "clocks": clk.summary(), "gpu_launches": 3 * args.steps,
            "graph": "state init + small-window scoring + tiled scan, one CUDA graph "
                     "replayed per step",
        })
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
