"""Seeded synthetic inputs for the STRIDE scoring path (arXiv 2609.14636).

This module holds the workload recipes only: ragged trajectory layouts, logit
distributions, Gumbel-max token sampling and the bf16 narrowing.  It contains
none of the scored method's arithmetic (no log-softmax, no turn means, no
running sums, no stop rule, no restart choice), so both the CUDA path and the
oracle can be fed from it without sharing any of the method.

The paper's own workloads (tau^2-bench rollouts of Qwen3 students and
teachers, AIME math traces) are not available here; these generators stand in
for them with the shapes the paper describes: multi-turn trajectories with
ragged turn lengths, a vocabulary of 151,936 (the Qwen3 tokenizer), a teacher
that tracks the student closely until a per-trajectory "first error" turn
(Observation 3) and drifts after it, and a token sampled from the student.

Small workloads are generated on the CPU with numpy; the bf16 workloads are
generated on the GPU with torch in fixed-size blocks, each block seeded from
(seed, block index), so any row range can be regenerated independently.
"""
from __future__ import annotations

import dataclasses
import json
import math
from pathlib import Path

import numpy as np

V_QWEN3 = 151_936
GEN_BLOCK = 512  # rows per independently seeded generation block

# lambda of each ragged bf16 workload, written by tests/golden/calibrate_lambda.py
CALIBRATION = Path(__file__).resolve().parents[1] / "tests" / "golden" / "lambda_calibration.json"
# used only until a calibration exists (a round number near the expected value)
PROVISIONAL_LAMBDA = {
    "batch_scoring_64x8_v151936_bf16": -36.0,
    "long_agentic_16x30_v151936_bf16": -170.0,
    "multi_teacher_128x12_v151936_bf16": -55.0,
}


def load_calibration(name: str) -> dict | None:
    if not CALIBRATION.exists():
        return None
    return json.loads(CALIBRATION.read_text()).get(name)


def workload_lambda(name: str) -> float:
    cal = load_calibration(name)
    return float(np.float32(cal["lambda"] if cal else PROVISIONAL_LAMBDA[name]))


def first_trajectories(lay: "Layout", max_rows: int) -> int:
    """Number of leading trajectories whose rows fit in max_rows (at least 1)."""
    n = int(np.searchsorted(lay.traj_row_off, lay.traj_row_off[0] + max_rows, side="right") - 1)
    return max(1, min(n, lay.n_traj))


def sub_layout(lay: "Layout", n_traj: int) -> "Layout":
    """The layout of the first n_traj trajectories."""
    k = int(lay.traj_turn_off[n_traj])
    return Layout(lay.traj_row_off[: n_traj + 1].copy(), lay.turn_row_off[: k + 1].copy(),
                  lay.traj_turn_off[: n_traj + 1].copy())


# --------------------------------------------------------------------------
# encoding helpers
# --------------------------------------------------------------------------
def bf16_bits_from_f32(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (IEEE round-to-nearest-even); return the raw bits."""
    x = np.ascontiguousarray(x, np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    rounding = ((u >> 16) & 1) + 0x7FFF
    out = ((u + rounding) >> 16).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def f32_from_bf16_bits(h: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(h, np.uint16).astype(np.uint32) << 16).view(np.float32)


# --------------------------------------------------------------------------
# ragged layouts
# --------------------------------------------------------------------------
@dataclasses.dataclass
class Layout:
    """Trajectory-major ragged layout.

    traj_row_off[i]..traj_row_off[i+1]   rows of trajectory i
    traj_turn_off[i]..traj_turn_off[i+1] turns of trajectory i
    turn_row_off[k]..turn_row_off[k+1]   rows of turn k
    """
    traj_row_off: np.ndarray  # int64 [n_traj+1]
    turn_row_off: np.ndarray  # int64 [n_turns+1]
    traj_turn_off: np.ndarray  # int32 [n_traj+1]

    @property
    def n_traj(self) -> int:
        return int(self.traj_row_off.shape[0] - 1)

    @property
    def n_turns(self) -> int:
        return int(self.turn_row_off.shape[0] - 1)

    @property
    def rows(self) -> int:
        return int(self.traj_row_off[-1] - self.traj_row_off[0])

    def row_traj(self) -> np.ndarray:
        r = np.arange(self.traj_row_off[0], self.traj_row_off[-1])
        return (np.searchsorted(self.traj_row_off, r, side="right") - 1).astype(np.int32)

    def row_turn(self) -> np.ndarray:
        r = np.arange(self.turn_row_off[0], self.turn_row_off[-1])
        return (np.searchsorted(self.turn_row_off, r, side="right") - 1).astype(np.int32)

    def turn_local_index(self) -> np.ndarray:
        """0-based index of each turn within its trajectory."""
        out = np.empty(self.n_turns, np.int32)
        for i in range(self.n_traj):
            a, b = self.traj_turn_off[i], self.traj_turn_off[i + 1]
            out[a:b] = np.arange(b - a)
        return out


def layout_from_turn_lengths(turn_lengths: list[list[int]]) -> Layout:
    traj_turn_off = [0]
    turn_row_off = [0]
    traj_row_off = [0]
    for lens in turn_lengths:
        for n in lens:
            turn_row_off.append(turn_row_off[-1] + int(n))
        traj_turn_off.append(traj_turn_off[-1] + len(lens))
        traj_row_off.append(turn_row_off[-1])
    return Layout(np.asarray(traj_row_off, np.int64), np.asarray(turn_row_off, np.int64),
                  np.asarray(traj_turn_off, np.int32))


def ragged_layout(rng: np.random.Generator, n_traj: int, turns: int | tuple[int, int],
                  lo: int, hi: int) -> Layout:
    """n_traj trajectories; turn count fixed (int) or uniform in [a, b]; turn
    lengths uniform integers in [lo, hi]."""
    lens = []
    for _ in range(n_traj):
        nt = turns if isinstance(turns, int) else int(rng.integers(turns[0], turns[1] + 1))
        lens.append([int(x) for x in rng.integers(lo, hi + 1, size=nt)])
    return layout_from_turn_lengths(lens)


# --------------------------------------------------------------------------
# workload descriptions
# --------------------------------------------------------------------------
@dataclasses.dataclass
class RowRecipe:
    """Per-row logit recipe for a ragged workload.

    student ~ N(0, sigma_s^2) iid, rounded to the storage dtype;
    teacher = student_stored + N(0, sigma_t[r]^2) (+ bump on one uniformly
    drawn token for rows with bump[r]), drawn from teacher stream
    stream[r], rounded to the storage dtype;
    token = argmax_j(student_stored[j] + Gumbel_j)  (Gumbel-max sampling from
    the student's softmax).
    """
    V: int
    sigma_s: float
    sigma_t: np.ndarray  # float32 [R]
    bump: np.ndarray  # bool [R]
    stream: np.ndarray  # int8 [R] teacher stream id
    stream_seeds: tuple  # seed of each teacher stream
    seed: int
    bump_value: float = 6.0


@dataclasses.dataclass
class Workload:
    name: str
    layout: Layout
    recipe: RowRecipe
    dtype: str  # "bf16" | "f32"
    mode: str  # "turn_mean" | "token_sum"
    lam: np.ndarray | None  # per-trajectory lambda (fp32); None = to be calibrated
    extra: dict = dataclasses.field(default_factory=dict)


def _error_turn_sigmas(layout: Layout, err_turn: np.ndarray, before: float, after: float) -> np.ndarray:
    sig = np.empty(layout.rows, np.float32)
    base = layout.traj_row_off[0]
    for i in range(layout.n_traj):
        a, b = layout.traj_turn_off[i], layout.traj_turn_off[i + 1]
        for j, k in enumerate(range(a, b)):
            r0, r1 = layout.turn_row_off[k] - base, layout.turn_row_off[k + 1] - base
            sig[r0:r1] = before if j < err_turn[i] else after
    return sig


def tiny_reference(seed: int = 0) -> dict:
    """1 trajectory, 4 turns x 128 tokens, V=32,000, fp32 logits, on the CPU.

    student ~ N(0, 3^2); teacher = student + N(0, 0.5^2), plus +6 on one
    uniformly drawn teacher-preferred token per row in the first two turns;
    tokens by Gumbel-max from the student.  Thresholds: token-sum lambda=-200
    (primary) and turn-mean lambda=-15.
    """
    rng = np.random.default_rng(seed)
    V, n_turn, n = 32_000, 4, 128
    lay = layout_from_turn_lengths([[n] * n_turn])
    R = lay.rows
    S = (rng.standard_normal((R, V), dtype=np.float32) * np.float32(3.0)).astype(np.float32)
    T = (S + rng.standard_normal((R, V), dtype=np.float32) * np.float32(0.5)).astype(np.float32)
    bump_rows = np.arange(R) < 2 * n
    bump_idx = rng.integers(0, V, size=R)
    T[bump_rows, bump_idx[bump_rows]] += np.float32(6.0)
    U = rng.random((R, V), dtype=np.float32)
    with np.errstate(divide="ignore"):
        G = -np.log(-np.log(U))
    tokens = np.argmax(S + G, axis=1).astype(np.int32)
    return dict(name="tiny_1x4x128_v32000_f32", S=S, T=T, tokens=tokens, layout=lay, V=V,
                lam_token=-200.0, lam_turn=-15.0)


def batch_scoring(seed: int = 2, n_traj: int = 64, turns: int = 8, lo: int = 64, hi: int = 512,
                  V: int = V_QWEN3) -> Workload:
    """64 trajectories x 8 turns, turn lengths U{64..512}, V=151,936 bf16.

    student ~ N(0, 4^2); teacher = student + N(0, 0.3^2) before a per-trajectory
    first-error turn e ~ U{0..turns-1} and + N(0, 2.5^2) from e on."""
    rng = np.random.default_rng(seed)
    lay = ragged_layout(rng, n_traj, turns, lo, hi)
    err = rng.integers(0, turns, size=n_traj)
    sig = _error_turn_sigmas(lay, err, 0.3, 2.5)
    R = lay.rows
    rec = RowRecipe(V=V, sigma_s=4.0, sigma_t=sig, bump=np.zeros(R, bool), stream=np.zeros(R, np.int8),
                    stream_seeds=(seed * 7919 + 1,), seed=seed)
    return Workload(f"batch_scoring_{n_traj}x{turns}_v{V}_bf16", lay, rec, "bf16", "turn_mean", None,
                    dict(err_turn=err))


def long_agentic(seed: int = 4, n_traj: int = 16, turns: int = 30, lo: int = 32, hi: int = 1024,
                 V: int = V_QWEN3) -> Workload:
    """16 trajectories x 30 turns, turn lengths U{32..1024}, V=151,936 bf16,
    batch-scoring teacher recipe with the divergence at e ~ U{0..29}."""
    rng = np.random.default_rng(seed)
    lay = ragged_layout(rng, n_traj, turns, lo, hi)
    err = rng.integers(0, turns, size=n_traj)
    sig = _error_turn_sigmas(lay, err, 0.3, 2.5)
    R = lay.rows
    rec = RowRecipe(V=V, sigma_s=4.0, sigma_t=sig, bump=np.zeros(R, bool), stream=np.zeros(R, np.int8),
                    stream_seeds=(seed * 7919 + 1,), seed=seed)
    mask_rng = np.random.default_rng(seed + 1000)
    masks = dict(p50=(mask_rng.random((n_traj, turns)) < 0.5).astype(np.uint8),
                 p90=(mask_rng.random((n_traj, turns)) < 0.9).astype(np.uint8))
    return Workload(f"long_agentic_{n_traj}x{turns}_v{V}_bf16", lay, rec, "bf16", "turn_mean", None,
                    dict(err_turn=err, masks=masks, chunk_rows=16_384))


def multi_teacher(seed: int = 5, n_traj: int = 128, turns: int = 12, lo: int = 64, hi: int = 512,
                  V: int = V_QWEN3, buffer_entries: int = 10_000) -> Workload:
    """128 trajectories, domain ~ Bernoulli(0.5), 12 turns x U{64..512},
    V=151,936 bf16.  Teacher noise N(0, 0.3^2) for domain 0 and N(0, 0.6^2) for
    domain 1, from two independent streams.  Plus a 10,000-entry record of
    per-turn means ~ N(-4.5, 1.5^2) with 5% quantised to force ties and masks
    ~ Bernoulli(0.5) and Bernoulli(0.9)."""
    rng = np.random.default_rng(seed)
    lay = ragged_layout(rng, n_traj, turns, lo, hi)
    dom = (rng.random(n_traj) < 0.5).astype(np.int8)
    row_dom = dom[lay.row_traj()]
    sig = np.where(row_dom == 0, np.float32(0.3), np.float32(0.6)).astype(np.float32)
    R = lay.rows
    rec = RowRecipe(V=V, sigma_s=4.0, sigma_t=sig, bump=np.zeros(R, bool), stream=row_dom,
                    stream_seeds=(50, 51), seed=seed)
    brng = np.random.default_rng(seed + 2000)
    means = (brng.standard_normal((buffer_entries, turns)) * 1.5 - 4.5).astype(np.float32)
    q = brng.random((buffer_entries, turns)) < 0.05
    means[q] = np.round(means[q] * 2.0) / 2.0  # quantised to 0.5 steps: exact ties
    n_turns = np.full(buffer_entries, turns, np.int32)
    short = brng.random(buffer_entries) < 0.1
    n_turns[short] = brng.integers(0, turns, size=int(short.sum()))
    masks = dict(p50=(brng.random((buffer_entries, turns)) < 0.5).astype(np.uint8),
                 p90=(brng.random((buffer_entries, turns)) < 0.9).astype(np.uint8))
    return Workload(f"multi_teacher_{n_traj}x{turns}_v{V}_bf16", lay, rec, "bf16", "turn_mean", None,
                    dict(domain=dom, buffer_means=means, buffer_n_turns=n_turns, buffer_masks=masks,
                         chunk_rows=16_384))


def decode_steps(seed: int = 3, B: int = 256, steps: int = 4096, ring: int = 16, V: int = V_QWEN3,
                 lo: int = 96, hi: int = 768) -> dict:
    """B=256 rollouts x 4096 decode steps, V=151,936 bf16, tiny-reference
    logit recipe (student N(0,3^2), teacher + N(0,0.5^2), +6 bump).

    The logits of step s are slab s mod ring of a ring of `ring` distinct
    [B, V] slabs (more bytes than L2); slabs with an even index carry the +6
    teacher bump on every row.  Each rollout closes a turn every U{96..768}
    steps (turn_end[s, b])."""
    rng = np.random.default_rng(seed)
    turn_end = np.zeros((steps, B), np.uint8)
    for b in range(B):
        t = -1
        while True:
            t += int(rng.integers(lo, hi + 1))
            if t >= steps:
                break
            turn_end[t, b] = 1
    R = ring * B
    slab = np.repeat(np.arange(ring), B)
    rec = RowRecipe(V=V, sigma_s=3.0, sigma_t=np.full(R, 0.5, np.float32), bump=(slab % 2 == 0),
                    stream=np.zeros(R, np.int8), stream_seeds=(seed * 7919 + 1,), seed=seed)
    return dict(name=f"decode_step_b{B}_s{steps}_v{V}_bf16", B=B, steps=steps, ring=ring,
                turn_end=turn_end, recipe=rec, lam_turn=-30.0, lam_token=-15_000.0)


# --------------------------------------------------------------------------
# GPU generation (torch), block-seeded
# --------------------------------------------------------------------------
def _block_gen(torch, device, seed: int, block: int):
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1_000_003 + int(block)) % (2**63 - 1))
    return g


def generate_rows(recipe: RowRecipe, row0: int, nrows: int, device="cuda", dtype: str = "bf16",
                  ld: int | None = None, out_S=None, out_T=None, out_tok=None):
    """Generate rows [row0, row0+nrows) of a recipe on `device` with torch.

    Returns (S, T, tokens): S/T [nrows, ld] of torch.bfloat16 (or float32) with
    columns >= V left as zero padding; tokens int32 [nrows].  Output tensors may
    be passed in to fill in place.  Rows are generated block by block
    (GEN_BLOCK rows per block), each block from its own seeded generators, so
    the result for a row does not depend on the requested range."""
    import torch

    V = recipe.V
    ld = V if ld is None else ld
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    S = out_S if out_S is not None else torch.empty((nrows, ld), dtype=tdt, device=device)
    T = out_T if out_T is not None else torch.empty((nrows, ld), dtype=tdt, device=device)
    tok = out_tok if out_tok is not None else torch.empty(nrows, dtype=torch.int32, device=device)
    if ld > V:
        S[:, V:].zero_()
        T[:, V:].zero_()
    r = row0
    end = row0 + nrows
    while r < end:
        blk = r // GEN_BLOCK
        b0 = blk * GEN_BLOCK
        b1 = b0 + GEN_BLOCK
        lo, hi = max(r, b0), min(end, b1)
        n_blk = GEN_BLOCK
        g = _block_gen(torch, device, recipe.seed, blk)
        s32 = torch.randn((n_blk, V), generator=g, device=device, dtype=torch.float32)
        s32.mul_(recipe.sigma_s)
        s_st = s32.to(tdt)
        del s32
        u = torch.rand((n_blk, V), generator=g, device=device, dtype=torch.float32)
        u.log_().neg_().log_().neg_()  # Gumbel(0,1) = -log(-log U)
        u.add_(s_st.float())
        tk = torch.argmax(u, dim=1).to(torch.int32)
        del u
        bump_idx = torch.randint(0, V, (n_blk,), generator=g, device=device)
        m = min(b1, recipe.sigma_t.shape[0]) - b0  # rows of this block inside the workload
        sig_np = np.zeros(n_blk, np.float32)
        sig_np[:m] = recipe.sigma_t[b0:b0 + m]
        str_np = np.zeros(n_blk, np.int8)
        str_np[:m] = recipe.stream[b0:b0 + m]
        bump_np = np.zeros(n_blk, bool)
        bump_np[:m] = recipe.bump[b0:b0 + m]
        t32 = s_st.float()
        noise = None
        for sid, sseed in enumerate(recipe.stream_seeds):
            if not (str_np[:m] == sid).any():
                continue
            nz = torch.randn((n_blk, V), generator=_block_gen(torch, device, sseed, blk),
                             device=device, dtype=torch.float32)
            if noise is None:
                noise = nz
            else:
                sel = torch.from_numpy(str_np == sid).to(device)
                noise = torch.where(sel[:, None], nz, noise)
            del nz
        if noise is not None:
            noise.mul_(torch.from_numpy(sig_np).to(device)[:, None])
            t32.add_(noise)
        if bump_np.any():
            rows_idx = torch.arange(n_blk, device=device)
            add = torch.from_numpy(np.where(bump_np, np.float32(recipe.bump_value), np.float32(0.0))).to(device)
            t32[rows_idx, bump_idx] += add
        t_st = t32.to(tdt)
        del t32, noise
        S[lo - row0:hi - row0, :V] = s_st[lo - b0:hi - b0]
        T[lo - row0:hi - row0, :V] = t_st[lo - b0:hi - b0]
        tok[lo - row0:hi - row0] = tk[lo - b0:hi - b0]
        r = hi
    return S, T, tok


def describe_recipe() -> str:
    return __doc__ or ""


__all__ = [
    "V_QWEN3", "GEN_BLOCK", "Layout", "RowRecipe", "Workload", "bf16_bits_from_f32", "f32_from_bf16_bits",
    "layout_from_turn_lengths", "ragged_layout", "tiny_reference", "batch_scoring", "long_agentic",
    "multi_teacher", "decode_steps", "generate_rows", "load_calibration", "workload_lambda",
    "first_trajectories", "sub_layout",
]
