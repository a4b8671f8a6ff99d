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
             "vocab_parallel", "stream_floor", "step_shapes")


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=WORKLOADS, default="batch_scoring",
                    help="batch_scoring is the headline; the others measure the remaining rows of the path")
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--e2e-rows", type=int, default=16384,
                    help="e2e sample: the first whole trajectories holding at least this many rows")
    ap.add_argument("--e2e-window", type=int, default=1024, help="rows per host->device copy window in e2e")
    ap.add_argument("--teacher", choices=["domains", "aligned"], default="domains",
                    help="multi_teacher: one teacher buffer per domain (gather-free entry point) or one aligned buffer")
    ap.add_argument("--no-secondary", action="store_true", help="headline workload only")
    ap.add_argument("--rows-list", default="8,16,32,48,64,96,128,160,192,224,256", help="step_shapes: live rows")
    ap.add_argument("--shapes", default="0x0,128x4,128x6,128x8,128x12,128x16,512x4,512x8",
                    help="step_shapes: CTA threads x CTAs per row (0x0 = automatic)")
    ap.add_argument("--step-shape", default="",
                    help="decode_step: a fixed launch shape THREADSxCLUSTER for every step "
                         "(stride_force_step_shape), for comparisons; default: the library's choice")
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
    elif args.workload == "stream_floor":
        run_stream_floor(args)
    elif args.workload == "step_shapes":
        run_step_shapes(args)
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


class BatchRun:
    """A ragged bf16 workload resident in HBM and its scoring step.

    entry = "aligned": one teacher buffer row-aligned with the student rows
    (stride_score_batch); "multi_teacher": the teacher rows of each domain in
    a buffer of their own, each trajectory scored against its domain's buffer
    through stride_score_batch_multi_teacher (no gather).  The workload is
    scored in its windows (16,384 rows for the streamed workloads, all rows
    for batch scoring) with the carried state."""

    def __init__(self, w, dev, entry="aligned", max_rows=0):
        import torch

        import paper_2609_14636_gb300 as stride
        import synth

        self.stride, self.w, self.dev, self.entry = stride, w, dev, entry
        lay = w.layout
        if max_rows > 0:
            lay = synth.sub_layout(lay, synth.first_trajectories(lay, max_rows))
        self.lay = lay
        R, V = lay.rows, w.recipe.V
        self.R, self.V = R, V
        self.lam = load_lambda(w)[: lay.n_traj]
        self.S = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
        self.tok = torch.empty(R, dtype=torch.int32, device=dev)
        t0 = time.perf_counter()
        CH = 8192
        if entry == "aligned":
            self.T = torch.empty((R, V), dtype=torch.bfloat16, device=dev)
            for r0 in range(0, R, CH):
                r1 = min(R, r0 + CH)
                synth.generate_rows(w.recipe, r0, r1 - r0, device=dev, out_S=self.S[r0:r1], out_T=self.T[r0:r1],
                                    out_tok=self.tok[r0:r1])
        else:
            # each domain's teacher rows in a buffer of their own, trajectories
            # in order; generated in chunks and scattered there (set-up only)
            dom = w.extra["domain"][: lay.n_traj].astype(np.uint8)
            n_rows_traj = np.diff(lay.traj_row_off)
            row0 = np.zeros(lay.n_traj, np.int64)
            self.T_dom = []
            for j in range(2):
                sel = dom == j
                row0[sel] = np.concatenate([[0], np.cumsum(n_rows_traj[sel])[:-1]]) if sel.any() else 0
                self.T_dom.append(torch.empty((max(1, int(n_rows_traj[sel].sum())), V), dtype=torch.bfloat16,
                                              device=dev))
            self.traj_domain = torch.from_numpy(dom).to(dev)
            self.traj_T_row0 = torch.from_numpy(row0).to(dev)
            row_traj = lay.row_traj()
            Tc = torch.empty((CH, V), dtype=torch.bfloat16, device=dev)
            for r0 in range(0, R, CH):
                r1 = min(R, r0 + CH)
                synth.generate_rows(w.recipe, r0, r1 - r0, device=dev, out_S=self.S[r0:r1], out_T=Tc[: r1 - r0],
                                    out_tok=self.tok[r0:r1])
                rt = row_traj[r0:r1]
                dest = row0[rt] + (np.arange(r0, r1) - lay.traj_row_off[rt])
                for j in range(2):
                    m = np.nonzero(dom[rt] == j)[0]
                    if m.size:
                        self.T_dom[j].index_copy_(0, torch.from_numpy(dest[m]).to(dev),
                                                  Tc.index_select(0, torch.from_numpy(m).to(dev)))
            del Tc
        torch.cuda.synchronize()
        self.t_gen = time.perf_counter() - t0
        self.offs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off, lay.turn_row_off, lay.traj_turn_off)]
        self.lam_d = torch.from_numpy(self.lam).to(dev)
        self.st = stride.new_state(lay.n_traj, dev)
        self.ts = stride.new_turn_stats(lay.n_turns, dev)
        self.out = {k: torch.empty(R, dtype=torch.float32, device=dev) for k in ("logp_s", "logp_t", "opd")}
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.chunk = int(w.extra.get("chunk_rows", R))
        self.windows = [(a, min(R, a + self.chunk)) for a in range(0, R, self.chunk)]
        wbytes = (stride.stride_score_batch_workspace_size(min(self.chunk, R)) if entry == "aligned"
                  else stride.multi_teacher_workspace_size(min(self.chunk, R)))
        self.wsb = torch.empty(wbytes, dtype=torch.uint8, device=dev)

    def score(self, a, b, stream, profile=None):
        stride = self.stride
        o = {k: v[a:b] for k, v in self.out.items()}
        if self.entry == "aligned":
            stride.stride_score_batch(self.S[a:b], self.T[a:b], self.tok[a:b], *self.offs, a, b, stride.TURN_MEAN,
                                      self.lam_d, self.st, out=o, turn_stats=self.ts, dev_status=self.status,
                                      workspace=self.wsb, stream=stream, profile=profile)
        else:
            stride.stride_score_batch_multi_teacher(
                self.S[a:b], self.T_dom, self.traj_domain, self.traj_T_row0, self.tok[a:b], *self.offs, a, b,
                stride.TURN_MEAN, self.lam_d, self.st, out=o, turn_stats=self.ts, dev_status=self.status,
                workspace=self.wsb, stream=stream, profile=profile)

    def step(self, stream, ev=None, profile=None):
        self.stride.stride_state_init(self.st, self.lay.n_traj, stream)
        if ev is not None:
            ev[0].record(stream)
        for a, b in self.windows:
            self.score(a, b, stream, profile)
        if ev is not None:
            ev[1].record(stream)

    def launches_per_step(self) -> int:
        """The library's kernels in one step: the state init, then per window
        either the workspace clear and the persistent kernel (windows above
        8 rows per SM) or the small-window kernel and its scan, plus the
        teacher-row pre-pass on the multi-teacher path."""
        per = 2 * len(self.windows)  # clear + persistent, or split + scan
        if self.entry != "aligned":
            per += len(self.windows)
        return 1 + per

    def early_fraction(self) -> float:
        st = self.stride.state_to_numpy(self.st)[: self.lay.n_traj]
        n_turns_traj = np.diff(self.lay.traj_turn_off)
        return float(np.mean((st["stop_turn"] >= 0) & (st["stop_turn"] < n_turns_traj - 1)))

    def release(self):
        for k in ("S", "T", "T_dom", "tok", "out", "wsb"):
            if hasattr(self, k):
                delattr(self, k)


def time_batch(run, steps, warmup, local, dev, ws=1) -> dict:
    """Warm-up, then `steps` timed steps (CUDA events on the launching
    stream, per step and over all), clocks sampled meanwhile."""
    import torch

    stream = torch.cuda.current_stream()
    for _ in range(max(3, warmup)):
        run.step(stream)
    torch.cuda.synchronize()
    if int(run.status.item()) != 0:
        raise RuntimeError(f"device status {int(run.status.item())} after warm-up")
    kev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if ws > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        time.sleep(0.25)
        e0.record(stream)
        for i in range(steps):
            run.step(stream, kev[i])
        e1.record(stream)
        torch.cuda.synchronize()
        time.sleep(0.05)
    if ws > 1:
        dist.barrier()
    ms_total = max_over_ranks(e0.elapsed_time(e1), dev)
    k_ms = [a.elapsed_time(b) for a, b in kev]
    bpr = algorithmic_bytes_per_row(run.V)
    peak = measured_peaks().get("hbm_gbs", 6800.0)
    k_avg = statistics.mean(k_ms)
    gbs = bpr * run.R / (k_avg * 1e-3) / 1e9
    return {"ms_step": ms_total / steps, "kernel_ms_mean": k_avg, "kernel_ms_min": min(k_ms), "gbs": gbs,
            "frac": gbs / peak, "clocks": clk.summary(), "early": run.early_fraction()}


def plain_copy_rates(dev, nbytes: int = 4 << 30) -> dict:
    """This box's plain pinned host <-> device rates: one cudaMemcpyAsync of
    nbytes each way (torch copy_ from / to pinned memory), CUDA events, best
    of 3."""
    import torch

    h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    d = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    res = {}
    for name, dst, src in (("h2d_gbs", d, h), ("d2h_gbs", h, d)):
        best = None
        for _ in range(3):
            a.record(stream)
            dst.copy_(src, non_blocking=True)
            b.record(stream)
            torch.cuda.synchronize()
            t = a.elapsed_time(b)
            best = t if best is None else min(best, t)
        res[name] = nbytes / (best * 1e-3) / 1e9
    del h, d
    res["bytes"] = nbytes
    return res


def e2e_batch(run, args, dev, ws=1) -> dict:
    """The headline metric end to end through the C ABI from pinned host
    memory: the first whole trajectories holding at least args.e2e_rows rows
    are copied host->device (S, T, tokens, window by window on a copy stream,
    window i+1 landing while window i is scored), scored with the carried
    state, and their per-row outputs, states and turn stats copied back, all
    inside each timed step."""
    import torch

    stride, lay, V = run.stride, run.lay, run.V
    stream = torch.cuda.current_stream()
    n_tr = int(np.searchsorted(lay.traj_row_off, args.e2e_rows, side="left"))
    n_tr = max(1, min(n_tr, lay.n_traj))
    Re = int(lay.traj_row_off[n_tr])
    n_tu = int(lay.traj_turn_off[n_tr])
    hS = torch.empty((Re, V), dtype=torch.bfloat16, pin_memory=True)
    hT = torch.empty((Re, V), dtype=torch.bfloat16, pin_memory=True)
    hk = torch.empty(Re, dtype=torch.int32, pin_memory=True)
    hS.copy_(run.S[:Re])
    hT.copy_(run.T[:Re])
    hk.copy_(run.tok[:Re])
    hout = {k: torch.empty(Re, dtype=torch.float32, pin_memory=True) for k in run.out}
    hst = torch.empty((n_tr, stride.STATE_DTYPE.itemsize), dtype=torch.uint8, pin_memory=True)
    hts = torch.empty((n_tu, stride.TURN_STATS_DTYPE.itemsize), dtype=torch.uint8, pin_memory=True)
    dS, dT, dk = run.S[:Re], run.T[:Re], run.tok[:Re]  # landing buffers: the resident workload's first rows
    eoffs = [torch.from_numpy(a).to(dev) for a in (lay.traj_row_off[: n_tr + 1], lay.turn_row_off[: n_tu + 1],
                                                    lay.traj_turn_off[: n_tr + 1])]
    est = stride.new_state(n_tr, dev)
    ets = stride.new_turn_stats(n_tu, dev)
    eout = {k: v[:Re] for k, v in run.out.items()}
    ew = args.e2e_window
    ewin = [(a, min(Re, a + ew)) for a in range(0, Re, ew)]
    wsb = torch.empty(stride.stride_score_batch_workspace_size(ew), dtype=torch.uint8, device=dev)
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
            stride.stride_score_batch(dS[a:b], dT[a:b], dk[a:b], *eoffs, a, b, stride.TURN_MEAN, run.lam_d[:n_tr],
                                      est, out={k: v[a:b] for k, v in eout.items()}, turn_stats=ets,
                                      dev_status=run.status, workspace=wsb, stream=stream)
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
    del hS, hT, hk
    plain = plain_copy_rates(dev)
    h2d_gbs = h2d / (e_ms * 1e-3) / 1e9
    return {"value": ws * Re / (e_ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": e_ms, "ms_per_step_min": e_all[0], "ms_per_step_max": e_all[-1],
            "timing": f"median of {n_e} steps, each timed on its own", "windows": len(ewin), "window_rows": ew,
            "h2d_gbs": h2d_gbs, "plain_copy": plain, "h2d_frac_of_plain_copy": h2d_gbs / plain["h2d_gbs"],
            "sample": f"first {n_tr} trajectories ({Re} rows) of the workload held in pinned host memory; H2D of "
                      f"S, T, tokens in {len(ewin)} windows of {ew} rows on a copy stream, overlapped with "
                      f"scoring; D2H of per-row outputs, state and turn stats; all inside the timed region"}


def run_batch(args) -> None:
    """Ragged batch scoring: the headline workload (all 148,909 rows in one
    window), or the long-agentic / multi-teacher workloads resident in HBM and
    scored in their 16,384-row windows with the carried state (multi-teacher
    through stride_score_batch_multi_teacher on per-domain teacher buffers,
    or --teacher aligned for one row-aligned teacher buffer).  The default run
    adds a `secondary` object: the other workloads measured in the same
    process, each with its own clock record."""
    import torch

    ws, rank, local, dev = _setup_rank()
    import synth

    w = {"batch_scoring": synth.batch_scoring, "long_agentic": synth.long_agentic,
         "multi_teacher": synth.multi_teacher}[args.workload]()
    entry = "multi_teacher" if (args.workload == "multi_teacher" and args.teacher == "domains") else "aligned"
    run = BatchRun(w, dev, entry, args.max_rows)
    lay, R, V = run.lay, run.R, run.V
    t = time_batch(run, args.steps, args.warmup, local, dev, ws)
    value = whole_job_rate(R, ws, t["ms_step"])
    stream = torch.cuda.current_stream()

    # the same scoring calls with the within-turn profile (Observation 1)
    # accumulated too, outside the timed steps above
    prof = run.stride.new_profile(dev)
    pev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(5)]
    for ev in pev:
        run.step(stream, ev, profile=prof)
    torch.cuda.synchronize()
    ms_with_profile = statistics.mean(a.elapsed_time(b) for a, b in pev)

    # ---- roofline of the fused kernel -------------------------------------
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs", 6800.0)
    bpr = algorithmic_bytes_per_row(V)
    dram_per_row, digest = kernel_traffic_record()
    roofline = {"bound": "hbm", "achieved": t["gbs"], "peak": peak, "unit": "GB/s", "frac": t["frac"],
                "traffic": None if (dram_per_row is None or entry != "aligned") else dram_per_row * R,
                "algorithmic_bytes_per_launch": bpr * R, "kernel_ms_mean": t["kernel_ms_mean"],
                "kernel_ms_min": t["kernel_ms_min"],
                "kernel": "score_batch_stream_kernel<bf16>" + (" (teacher rows through the per-domain row table)"
                                                               if entry != "aligned" else ""),
                "kernel_ms_mean_with_profile": ms_with_profile,
                "peak_source": "MEASURED_PEAKS.json hbm_gbs (of measured)" if "hbm_gbs" in peaks else "fallback 6.8 TB/s"}

    e2e = e2e_batch(run, args, dev, ws) if entry == "aligned" and args.workload == "batch_scoring" else None
    cpu = None
    if rank == 0 and ws == 1:
        if entry == "aligned":
            cpu = cpu_oracle_rate(run.S, run.T, run.tok, lay, run.lam, args.cpu_budget)
    line = None
    if rank == 0:
        line = _common_line(args, ws, t["ms_step"], value)
        line.update({
            "config": {"workload": w.name if args.max_rows <= 0 else f"{w.name} (first {lay.n_traj} trajectories)",
                       "windows": len(run.windows), "window_rows": run.chunk,
                       "trajectories": lay.n_traj, "turns": lay.n_turns, "rows": R, "vocab": V,
                       "logits": "bf16 student + bf16 teacher, resident in HBM"
                                 + (" (teacher rows in one buffer per domain)" if entry != "aligned" else ""),
                       "entry_point": "stride_score_batch" if entry == "aligned" else "stride_score_batch_multi_teacher",
                       "bytes_resident": 2 * R * V * 2, "stop_mode": "turn_mean",
                       "lambda": float(run.lam[0]), "early_stop_fraction": t["early"],
                       "l2": f"inputs ({2 * R * V * 2 / 1e9:.1f} GB) larger than L2 (129 MB): no flush",
                       "lambda_source": "tests/golden/lambda_calibration.json (oracle, 40% quantile)",
                       "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU",
                       "generation_s": run.t_gen},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": t["clocks"],
            "gpu_launches": run.launches_per_step() * args.steps,
        })
    run.release()
    del run
    torch.cuda.empty_cache()
    if args.workload == "batch_scoring" and ws == 1 and not args.no_secondary:
        sec = measure_secondary(args, dev, local)
        if line is not None:
            line["secondary"] = sec
    if line is not None:
        print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


def _short(d: dict, keys) -> dict:
    return {k: d[k] for k in keys if k in d}


def measure_secondary(args, dev, local) -> dict:
    """The other workloads of the path, in the same process, each with its own
    clock record (fewer steps for the large ones): the tiny reference, the
    decode sweep, long agentic plus the restart choice over its turn stats,
    multi-teacher through the per-domain buffers (and the aligned buffer for
    comparison) plus the 10,000-record restart choice."""
    import torch

    import paper_2609_14636_gb300 as stride
    import synth

    sec = {}
    tl = measure_tiny(args, dev, local)
    sec["tiny_reference"] = {"tokens_per_s": tl["value"], "us_per_step": 1e3 * tl["ms_per_step"],
                             "gbs": tl["roofline"]["achieved"], "frac": tl["roofline"]["frac"],
                             "rows": tl["config"]["rows"], "clocks": tl["clocks"]}
    torch.cuda.empty_cache()
    dl = measure_decode(args, dev, local)
    r = dl["roofline"]
    sec["decode_step"] = {"tokens_per_s": dl["value"], "gbs": r["achieved"], "frac": r["frac"],
                          "form": "compacted sweep (live rollouts only), 4,096 steps, lambda = -30",
                          "ms_per_sweep": dl["ms_per_step"], "tokens_per_sweep": dl["config"]["tokens_scored_per_sweep"],
                          "us_per_step_all_active": r["us_per_step_all_active"], "all_active_frac": r["all_active_frac"],
                          "masked_sweep": r["masked_sweep"], "clocks": dl["clocks"]}
    torch.cuda.empty_cache()
    steps, warm = max(3, min(args.steps, 8)), 2

    w = synth.long_agentic()
    run = BatchRun(w, dev, "aligned")
    t = time_batch(run, steps, warm, local, dev)
    lay = run.lay
    tsn = stride.turn_stats_to_numpy(run.ts)[: lay.n_turns]  # the scoring's own turn stats
    nt = np.diff(lay.traj_turn_off).astype(np.int32)
    m = torch.from_numpy(tsn["mean_t"].reshape(lay.n_traj, -1).astype(np.float32)).to(dev)
    us_sel = time_select(m, torch.from_numpy(nt).to(dev), torch.from_numpy(w.extra["masks"]["p50"]).to(dev),
                         float("-inf"), dev)
    sec["long_agentic"] = {"tokens_per_s": run.R / (t["ms_step"] * 1e-3), "ms_per_step": t["ms_step"],
                           "gbs": t["gbs"], "frac": t["frac"], "rows": run.R, "windows": len(run.windows),
                           "select_us_16x30": us_sel, "clocks": t["clocks"]}
    run.release()
    del run
    torch.cuda.empty_cache()

    w = synth.multi_teacher()
    res = {}
    for entry in ("aligned", "multi_teacher"):
        run = BatchRun(w, dev, entry)
        t = time_batch(run, steps, warm, local, dev)
        res[entry] = {"tokens_per_s": run.R / (t["ms_step"] * 1e-3), "ms_per_step": t["ms_step"], "gbs": t["gbs"],
                      "frac": t["frac"], "clocks": t["clocks"], "rows": run.R, "windows": len(run.windows)}
        run.release()
        del run
        torch.cuda.empty_cache()
    sl = measure_select(args, dev, local)
    sec["multi_teacher"] = dict(res["multi_teacher"],
                                entry_point="stride_score_batch_multi_teacher (one teacher buffer per domain)",
                                aligned_teacher_buffer=_short(res["aligned"], ("gbs", "frac", "ms_per_step")),
                                select_us_10000x12=sl["roofline"]["us_per_call"],
                                select_clocks=sl["clocks"])
    return sec


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
    ws, rank, local, dev = _setup_rank()
    shape = getattr(args, "step_shape", "")
    if shape:
        import paper_2609_14636_gb300 as stride

        th, C = (int(v) for v in shape.split("x"))
        stride.stride_force_step_shape(th, C)
    try:
        line = measure_decode(args, dev, local, ws)
    finally:
        if shape:
            stride.stride_force_step_shape(0, 0)
    if shape:
        line["config"]["forced_step_shape"] = shape
    if rank == 0:
        print(json.dumps(line), flush=True)


def measure_decode(args, dev, local, ws=1) -> dict:
    """The decode sweeps of run_decode; returns the JSON line."""
    import torch

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
    return line


def run_select(args) -> None:
    """Restart choice over the 10,000-record prefix buffer (12 turns, masks
    Bernoulli(0.5), alpha = -6.0): one launch per call, 200 calls per graph."""
    ws, rank, local, dev = _setup_rank()
    line = measure_select(args, dev, local, ws)
    if rank == 0:
        print(json.dumps(line), flush=True)


def time_select(means, n_turns, mask, alpha, dev, calls=200, reps=20) -> float:
    """us per stride_select_restart call (a graph of `calls` launches)."""
    import torch

    import paper_2609_14636_gb300 as stride

    N = means.shape[0]
    ks = torch.empty(N, dtype=torch.int32, device=dev)
    km = torch.empty(N, dtype=torch.int32, device=dev)
    g = _graph(lambda: [stride.stride_select_restart(means, n_turns, mask, alpha, ks, km) for _ in range(calls)])
    for _ in range(3):
        g.replay()
    stream = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        g.replay()
    b.record(stream)
    torch.cuda.synchronize()
    return 1e3 * a.elapsed_time(b) / (reps * calls)


def measure_select(args, dev, local, ws=1) -> dict:
    """The restart choice and the prefix buffer's record step of run_select;
    returns the JSON line."""
    import torch

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
    return line


def run_tiny(args) -> None:
    """The tiny reference workload: 1 trajectory x 4 turns x 128 tokens,
    V = 32,000 fp32 logits (131 MB, about the size of L2), token-sum stop
    at lambda = -200.  L2 is flushed (a 512 MB write) before every timed
    step; each step (state init + scoring, captured once in a CUDA graph so
    that host-side submission is not timed) is timed with CUDA events."""
    ws, rank, local, dev = _setup_rank()
    line = measure_tiny(args, dev, local, ws)
    if rank == 0:
        print(json.dumps(line), flush=True)


def measure_tiny(args, dev, local, ws=1) -> dict:
    """The tiny-reference steps of run_tiny; returns the JSON line."""
    import torch

    import oracle
    import paper_2609_14636_gb300 as stride
    import synth

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
                               "+ scan_logprobs_tile_kernel (4 tiles of 128 rows, one 4-CTA cluster)",
                     "note": "512 rows on 152 SMs: a latency-bound launch; time includes state init",
                     "ms_per_step_write_flush_only": ms_write_only,
                     "frac_write_flush_only": bpr * R / (ms_write_only * 1e-3) / 1e9 / peak},
        "cpu_baseline": {"value": cpu_rate, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"all {R} rows"},
        "clocks": clk.summary(), "gpu_launches": 3 * args.steps,
        "graph": "state init + small-window scoring + tiled scan, one CUDA graph "
                 "replayed per step",
    })
    return line


def run_stream_floor(args) -> None:
    """Read-only floors for the scoring kernels' bytes (stride_selftest_stream_read:
    the kernels' 16-byte loads, no arithmetic):
    * long read: 2 x 8 GB, several launch shapes, best of 5 launches -- the
      measured read-only HBM rate of this GPU;
    * decode-step size: the 256 x V bf16 S and T slabs of one step (155.6 MB)
      from the decode workload's 16-slab ring, 64-launch graphs;
    * tiny-reference size: 512 x 32,000 fp32 S and T (131 MB) after the tiny
      bench's L2 flush (a 512 MB write, then a clean 256 MB read)."""
    import torch

    import paper_2609_14636_gb300 as stride
    import synth

    ws, rank, local, dev = _setup_rank()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    stream = torch.cuda.current_stream()
    shapes = [(sms * 8, 128), (1024, 128), (sms * 4, 256), (sms * 2, 512), (sms, 1024)]
    sink = torch.empty(sms * 16, dtype=torch.int32, device=dev)
    a_ev, b_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def best_ms(fn, reps, per=1):
        best = None
        for _ in range(reps):
            a_ev.record(stream)
            fn()
            b_ev.record(stream)
            torch.cuda.synchronize()
            t = a_ev.elapsed_time(b_ev) / per
            best = t if best is None else min(best, t)
        return best

    res = {}
    with ClockSampler(local) as clk:
        time.sleep(0.25)
        nb = 8 << 30
        A = torch.empty(nb, dtype=torch.uint8, device=dev).fill_(1)
        Bb = torch.empty(nb, dtype=torch.uint8, device=dev).fill_(2)
        long_read = {}
        for g, th in shapes:
            stride.stride_selftest_stream_read(A, Bb, nb, g, th, sink)
            ms = best_ms(lambda: stride.stride_selftest_stream_read(A, Bb, nb, g, th, sink), 5)
            long_read[f"{g}x{th}"] = 2 * nb / (ms * 1e-3) / 1e9
        del A, Bb
        torch.cuda.empty_cache()
        res["long_read_gbs"] = long_read

        w = synth.decode_steps()
        B, ring, V = w["B"], w["ring"], w["recipe"].V
        S, T, _ = synth.generate_rows(w["recipe"], 0, ring * B, device=dev)
        slab = B * V * 2
        step_floor = {}
        for g, th in shapes:
            gr = _graph(lambda: [stride.stride_selftest_stream_read(S[(i % ring) * B:], T[(i % ring) * B:], slab, g,
                                                                     th, sink) for i in range(64)])
            gr.replay()
            us = 1e3 * best_ms(gr.replay, 5, 64)
            step_floor[f"{g}x{th}"] = {"us": us, "gbs": 2 * slab / (us * 1e-6) / 1e9}
        del S, T
        res["decode_step_size"] = {"bytes": 2 * slab, "per_shape": step_floor}

        tw = synth.tiny_reference(0)
        tS = torch.from_numpy(tw["S"]).to(dev)
        tT = torch.from_numpy(tw["T"]).to(dev)
        flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
        clean = torch.ones(256 << 20, dtype=torch.uint8, device=dev)
        tb = tS.numel() * 4
        tiny_floor = {}
        for g, th in shapes:
            ts_ = []
            for _ in range(10):
                flush.zero_()
                clean.sum()
                a_ev.record(stream)
                stride.stride_selftest_stream_read(tS, tT, tb, g, th, sink)
                b_ev.record(stream)
                torch.cuda.synchronize()
                ts_.append(a_ev.elapsed_time(b_ev))
            us = 1e3 * statistics.median(ts_)
            tiny_floor[f"{g}x{th}"] = {"us": us, "gbs": 2 * tb / (us * 1e-6) / 1e9}
        res["tiny_reference_size"] = {"bytes": 2 * tb, "per_shape": tiny_floor,
                                      "l2": "512 MB written, then a clean 256 MB read, before each launch"}
        time.sleep(0.05)
    peak = measured_peaks().get("hbm_gbs", 6800.0)
    best = max(long_read.values())
    if rank == 0:
        line = _common_line(args, ws, 2 * nb / best / 1e6, best, unit="GB/s",
                            metric="read-only stream GB/s (the scoring kernels' loads, no arithmetic)", dtype="u8")
        line.update({"config": {"workload": "stream_floor", "long_read_bytes": 2 * nb},
                     "roofline": {"bound": "hbm", "achieved": best, "peak": peak, "unit": "GB/s",
                                  "frac": best / peak, "traffic": None,
                                  "kernel": "stream_read_kernel (stride_selftest_stream_read)",
                                  "peak_source": "MEASURED_PEAKS.json hbm_gbs (of measured; a read+write copy)"},
                     "floors": res, "clocks": clk.summary(), "gpu_launches": None})
        print(json.dumps(line), flush=True)


def run_step_shapes(args) -> None:
    """us per compacted decode step at fixed live-row counts, for the
    automatic launch shape and forced ones (stride_force_step_shape): all
    rows active (lambda = -inf), 64-step graphs over the decode workload's
    16-slab ring, median of 5 x 4 replays.  The sweep the launch-shape rule
    of the step kernel rests on."""
    import torch

    import paper_2609_14636_gb300 as stride
    import synth

    ws, rank, local, dev = _setup_rank()
    w = synth.decode_steps()
    B, ring, V = w["B"], w["ring"], w["recipe"].V
    S, T, tok = synth.generate_rows(w["recipe"], 0, ring * B, device=dev)
    st = stride.new_state(B, dev)
    idx = torch.arange(B, dtype=torch.int32, device=dev)
    te0 = torch.zeros(B, dtype=torch.uint8, device=dev)
    ns = [int(x) for x in args.rows_list.split(",")]
    shapes = [tuple(int(v) for v in x.split("x")) for x in args.shapes.split(",")]
    bpr = algorithmic_bytes_per_row(V)
    stream = torch.cuda.current_stream()
    a_ev, b_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    table = []
    with ClockSampler(local) as clk:
        for n in ns:
            row = {"rows": n}
            for th, C in shapes:
                stride.stride_force_step_shape(th, C)
                try:
                    def f():
                        stride.stride_state_init(st, B)
                        for i in range(64):
                            j = i % ring
                            stride.stride_score_step_compact(S[j * B:j * B + n], T[j * B:j * B + n],
                                                             tok[j * B:j * B + n], te0[:n], idx[:n], stride.TURN_MEAN,
                                                             float("-inf"), st)
                    g = _graph(f)
                finally:
                    stride.stride_force_step_shape(0, 0)
                for _ in range(3):
                    g.replay()
                ts_ = []
                for _ in range(5):
                    a_ev.record(stream)
                    for _ in range(4):
                        g.replay()
                    b_ev.record(stream)
                    torch.cuda.synchronize()
                    ts_.append(1e3 * a_ev.elapsed_time(b_ev) / (4 * 64))
                row["auto" if th == 0 else f"{th}x{C}"] = round(statistics.median(ts_), 2)
            table.append(row)
    if rank == 0:
        auto = {r["rows"]: r.get("auto") for r in table}
        line = _common_line(args, ws, None, None, unit="us/step", metric="decode step time by live rows and launch shape")
        line.update({"config": {"workload": "step_shapes", "vocab": V, "graph": "64 compacted steps per graph",
                                "shapes": "CTA threads x CTAs per row; auto = the library's choice"},
                     "table_us_per_step": table,
                     "auto_gbs": {n: n * bpr / (us * 1e-6) / 1e9 for n, us in auto.items() if us},
                     "clocks": clk.summary(), "gpu_launches": None})
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
