"""Benchmark of the entropic-time batched decode step on GB300.

One step = one pass of the whole hot path over one batch:
  score every key page (eti_score_blocks) -> keep set, budget, compaction and
  kept-token normaliser (eti_prune_blocks) -> GQA paged decode over the kept
  blocks (eti_paged_decode) -> entropy / entropic time / temperature /
  threshold / sample (eti_entropy_temp_sample).
The step runs overlapped, as a serving loop would issue it: the sampling call
on one stream and the attention half (score, keep set, decode) of each of two
sub-batches (the batch's halves) on a stream of its own, all forked at the
step's start and joined before its end; the same four calls over the whole
batch on one stream give `ms_per_step_sequential`.
The workload is the Llama-3-8B-shaped layer step (64 sequences, 32 query /
8 kv heads, head_dim 128, page 16, context lengths uniform in [1024, 8192],
vocabulary 128,256) with seeded synthetic inputs.

Prints ONE JSON line (rank 0).  Timing: W warm-up steps, then K timed steps;
before every step a buffer of twice the L2 size is written and another one
read (L2 flush, write-backs settled outside the timed region); each timed
step is bracketed by one pair of CUDA events on the launching stream (no
event between its calls, so each kernel keeps its programmatic launch overlap
with the one before), and a separate pass with an event between calls gives
the per-kernel times behind `roofline`.  `value` = sequences decoded per
second per layer step over all ranks (each rank decodes its own batch: weak
scaling).  The clock sampler runs over the timed steps and a further
--clock-seconds of the same step back to back (`clocks`, `clock_pass`).

Beside the headline step the line carries: `dense_baseline` (the same batch
decoded densely by the same library call), `sampling` (the entropy / sample
pass against the HBM peak and against a read-only pass over the same logits),
`e2e` (host buffers, copies inside the timed region, with a stage breakdown),
`workloads` (tiny, long_ctx, mixed_batch and llama3_70b at H_target 0.1, 0.3
and 0.5 log V: step time, tokens/s, kept fraction, per-kernel times and
fractions of the peak), `keep_sweep`, `estimators` and `cpu_baseline`.

--impl reference times the fp64 CPU oracle on a bounded sample of the same
workload (the paper has no reference implementation).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# The overlapped step runs on several streams at once (the sampling call and
# one per sub-batch, the copy stream of the end-to-end step); with the driver's
# default of 8 hardware work queues, two of them could share a queue and run
# one after the other (a per-process draw).  Before CUDA starts:
os.environ.setdefault("CUDA_DEVICE_MAX_CONNECTIONS", "32")

import numpy as np
import torch

import workloads

METRIC = "paged-decode tokens/s per layer-step"
UNIT = "tokens/s"
SUB_BATCHES = 2      # sub-batches of the overlapped step, each on its own stream


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


def shard_workload(w: workloads.Workload, rank: int) -> workloads.Workload:
    """Each rank decodes its own batch of the same shape (independent sequences)."""
    return w.scaled(seed=w.seed + 7919 * rank) if rank else w


def aggregate(per_rank_step_s: list[float], B: int) -> tuple[float, float]:
    """Whole-job throughput from every rank's step time: all ranks' sequences
    over the slowest rank's time."""
    slowest = max(per_rank_step_s)
    return B * len(per_rank_step_s) / slowest, slowest


def aggregate_e2e(e2e: dict, B: int, world: int, device) -> dict:
    """The end-to-end figure for the whole job: every rank's sequences over the
    slowest rank's step, and every rank's copies (unchanged at one rank)."""
    if world == 1:
        return e2e
    s = max_over_ranks(e2e["ms_per_step"] / 1e3, world, device)
    return dict(e2e, value=round(B * world / s, 1), ms_per_step=round(s * 1e3, 4),
                h2d_bytes_per_step=e2e["h2d_bytes_per_step"] * world,
                d2h_bytes_per_step=e2e["d2h_bytes_per_step"] * world)


def max_over_ranks(x: float, world: int, device) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while it runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int, log_path: str | None = None):
        self.index, self.log_path, self.proc, self.lines = index, log_path, None, []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.index), "-lms", "100"], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
            self._t = threading.Thread(target=self._read, daemon=True)
            self._t.start()
            t0 = time.time()
            while not self.lines and time.time() - t0 < 10 and self.proc.poll() is None:
                time.sleep(0.02)           # the timed region starts once sampling runs
        except (FileNotFoundError, OSError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self._t.join(timeout=2)
        if self.log_path and self.lines:
            with open(self.log_path, "w") as f:
                f.write("\n".join(self.lines) + "\n")

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
def algorithmic_bytes(w, L: np.ndarray, kept_blocks: int) -> dict:
    """Compulsory DRAM bytes per call of each kernel (see the design notes)."""
    g = w.Hq // w.Hkv
    nb = -(-L // w.P)
    tokens_slots = int(nb.sum()) * w.P                   # token slots of all blocks
    k_bytes = int(L.sum()) * w.Hkv * w.D * 2             # every key read once
    q_bytes = w.B * w.Hq * w.D * 2
    score_bytes = tokens_slots * w.Hq * 4                # x_i written for every slot
    stats_bytes = int(nb.sum()) * w.Hq * 16
    kept_slots = kept_blocks * w.P
    return {
        "score": k_bytes + q_bytes + score_bytes + stats_bytes,
        "prune": stats_bytes + int(nb.sum()) * w.Hkv * 5,
        # kept V pages + their scores + the bf16 output
        "decode": kept_slots * w.D * 2 + kept_slots * g * 4 + w.B * w.Hq * w.D * 2,
        "sample": w.B * w.V * 4,
    }


def kept_attention_mass(stats: torch.Tensor, keep_mask: torch.Tensor, ctx_lens: torch.Tensor,
                        P: int) -> dict:
    """Share of each query head's attention (softmax over all of its sequence's
    tokens) that falls in the kept blocks, from the scorer's block stats
    [B][Hkv][max_blocks][g][(m, l - 1, u, e)] and the keep mask: with
    l_b = 1 + (l - 1), Z = sum_b l_b e^{m_b - M} over the sequence's blocks and
    the kept share = the same sum over the kept blocks / Z.  Sequences without
    tokens are left out.  A diagnostic of reading A, whose block score can be
    small for a block holding one dominant token."""
    B, Hkv, mb, g, _ = stats.shape
    nb = (ctx_lens.to(torch.int64) + P - 1) // P
    valid = (torch.arange(mb, device=stats.device)[None, :] < nb[:, None])[:, None, :, None]
    m = stats[..., 0].double()
    ok = valid & torch.isfinite(m)
    M = torch.where(ok, m, torch.full_like(m, -math.inf)).amax(dim=2, keepdim=True)
    w = torch.where(ok, (1.0 + stats[..., 1].double()) * torch.exp(m - M), torch.zeros_like(m))
    Z = w.sum(dim=2)
    kept = keep_mask.to(torch.bool)[..., None] & ok
    frac = torch.where(kept, w, torch.zeros_like(w)).sum(dim=2) / Z
    frac = frac[(nb > 0)[:, None, None].expand_as(frac) & torch.isfinite(frac)]
    if frac.numel() == 0:
        return {"mean": None, "min": None}
    return {"mean": round(float(frac.mean()), 5), "min": round(float(frac.min()), 5)}


def source_digest(paths) -> str:
    """sha256 of the code of these source files: comments and blank lines are
    left out, so a change of wording is not a change of kernel."""
    import hashlib
    import re
    h = hashlib.sha256()
    for path in paths:
        with open(os.path.join(ROOT, path)) as f:
            for line in f:
                code = re.sub(r"/\*.*?\*/", "", line).split("//")[0].strip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()


def ncu_traffic(kernel):
    """DRAM bytes per launch from the committed ncu record, if the kernel's
    code is unchanged since that capture (else None)."""
    rec = ncu_record(kernel)
    return rec["bytes"] if rec else None


def run_estimators(eti, lg, step, prm, w, flush_l2, stream, k=64, reps=50):
    """Time eti_topk_entropy (L2 flushed before each call) and correlate H~ and H^
    with the exact entropy of the same rows (Pearson r over the batch)."""
    B = w.B
    f32 = torch.float32
    Ht, Hh, tm = (torch.empty(B, dtype=f32, device=lg["logits"].device) for _ in range(3))
    err = torch.empty(B, dtype=torch.int32, device=lg["logits"].device)
    tau = lg["tau"].clone()
    step.sample(lg["logits"], lg["T_in"], lg["H_prev"], tau, lg["H_target"], params=prm, seed=w.seed)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
    for i in range(reps + 3):
        flush_l2()
        if i >= 3:
            ev[i - 3][0].record(stream)
        eti.eti_topk_entropy(lg["logits"], lg["T_in"], k, Ht, Hh, err, tail_mass=tm)
        if i >= 3:
            ev[i - 3][1].record(stream)
    torch.cuda.synchronize()
    ms = statistics.median(e[0].elapsed_time(e[1]) for e in ev)
    H = step.H.double().cpu().numpy()
    r_t = float(np.corrcoef(H, Ht.double().cpu().numpy())[0, 1])
    r_h = float(np.corrcoef(H, Hh.double().cpu().numpy())[0, 1])
    return {"k": k, "topk_entropy_ms": round(ms, 5),
            "topk_entropy_gbs": round(B * w.V * 4 / (ms / 1e3) / 1e9, 1),
            "pearson_r_H_tilde_vs_H": round(r_t, 5), "pearson_r_H_hat_vs_H": round(r_h, 5),
            "mean_tail_mass": round(float(tm.double().mean().item()), 6),
            "note": "one CTA per row: the k-th largest thread maximum bounds the k-th logit, the "
                    "tokens above it are sorted (1 pass from HBM, 1 from L2); the exact entropy + "
                    "sample pass is kernels_ms['sample']; schedule_ms: Section 3.1 priority and "
                    "admission of half the batch"}


def run_schedule(eti, step, kv, w, stream, reps=50):
    """Median time of eti_schedule (Section 3.1 priority + admission of half
    the batch) on the step's entropy flow, kept counts and context lengths."""
    dev = step.dH.device
    ema = torch.zeros(w.B, dtype=torch.float32, device=dev)
    pr = torch.empty(w.B, dtype=torch.float32, device=dev)
    adm = torch.empty(w.B, dtype=torch.uint8, device=dev)
    urg = torch.ones(w.B, dtype=torch.float32, device=dev)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
    for i in range(reps + 3):
        if i >= 3:
            ev[i - 3][0].record(stream)
        eti.eti_schedule(step.dH, ema, w.B // 2, pr, adm, kept_cnt=step.kept_cnt, P=w.P,
                         ctx_lens=kv["ctx_lens"], urgency=urg)
        if i >= 3:
            ev[i - 3][1].record(stream)
    torch.cuda.synchronize()
    return round(statistics.median(e[0].elapsed_time(e[1]) for e in ev), 5)


def workload_desc(w) -> str:
    """The workload as `config.workload` names it (both arms print the same)."""
    return f"{w.name}: B={w.B} Hq={w.Hq} Hkv={w.Hkv} D={w.D} P={w.P} {ctx_desc(w)} V={w.V}"


def ctx_desc(w) -> str:
    """The workload's context-length distribution, as printed in `config`."""
    kind = w.ctx[0]
    if kind == "list":
        return "ctx " + "/".join(str(x) for x in w.ctx[1])
    return f"ctx {'log-U' if kind == 'loguniform' else 'U'}[{w.ctx[1]},{w.ctx[2]}]"


def run_keep_sweep(eti, device, flush_l2, stream, peak, fracs=(0.1, 0.25, 0.5, 1.0), reps=10):
    """The long-context step of the paper's sweep (8 sequences, contexts
    U[32768, 131072]): theta = +inf and B_min = ceil(f * n_b) of the longest
    sequence, so every sequence keeps its min(B_min, n_b) best blocks.  The
    decode reads only the kept blocks: its time against the kept fraction is
    the saving the method buys; the scorer's full read of K is the fixed cost
    of the rule.  Median of `reps` calls, L2 flushed before each."""
    w = workloads.WORKLOADS["long_ctx"]
    kv = workloads.make_kv(w, device)
    g = w.Hq // w.Hkv
    st = eti.DecodeStep(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, w.V, device=device)
    stats = torch.empty((w.B, w.Hkv, w.max_blocks, g, 4), dtype=torch.float32, device=device)
    shape = (w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks)
    theta = torch.full((w.B,), float("inf"), dtype=torch.float32, device=device)
    L = kv["ctx_lens"].cpu().numpy()
    nb = -(-L // w.P)
    total = int(nb.sum()) * w.Hkv

    def timed(fn):
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
        for i in range(reps + 2):
            flush_l2()
            if i >= 2:
                ev[i - 2][0].record(stream)
            fn()
            if i >= 2:
                ev[i - 2][1].record(stream)
        torch.cuda.synchronize()
        return statistics.median(e[0].elapsed_time(e[1]) for e in ev)

    def score():
        eti.eti_score_blocks(kv["q"], kv["k_cache"], kv["block_table"], kv["ctx_lens"], kv["scale"],
                             stats, token_scores=st.token_scores, num_pages=kv["num_pages"])

    def decode():
        eti.eti_paged_decode(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                             kv["scale"], st.out, st.err_dec, st.ws_dec, kept_idx=st.kept_idx,
                             kept_cnt=st.kept_cnt, token_scores=st.token_scores,
                             kept_norm=st.kept_norm, num_pages=kv["num_pages"])

    score_ms = timed(score)
    # the baseline the rule is measured against: dense decode over every block
    # (q.K and p.V in one pass, K and V of every block read once)
    ws_dense = torch.empty(eti.paged_decode_workspace_size(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, False),
                           dtype=torch.uint8, device=device)
    out_dense = torch.empty_like(st.out)

    def dense():
        eti.eti_paged_decode(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                             kv["scale"], out_dense, st.err_dec, ws_dense, num_pages=kv["num_pages"])

    dense_ms = timed(dense)
    kv_bytes = int(L.sum()) * w.Hkv * w.D * 2 * 2 + 2 * w.B * w.Hq * w.D * 2
    points = []
    for f in fracs:
        B_min = int(math.ceil(f * int(nb.max())))

        def prune():
            eti.eti_prune_blocks(stats, kv["block_table"], kv["ctx_lens"], shape, theta, B_min, st.keep_mask,
                                 st.kept_idx, st.kept_cnt, st.err_attn, kept_norm=st.kept_norm,
                                 num_pages=kv["num_pages"])

        prune_ms = timed(prune)
        kept = int(st.kept_cnt.sum().item())
        ms = timed(decode)
        byt = algorithmic_bytes(w, L, kept)["decode"]
        step_ms = score_ms + prune_ms + ms
        points.append({"f": f, "B_min": B_min, "kept_fraction": round(kept / total, 4),
                       "decode_ms": round(ms, 5), "decode_gbs": round(byt / (ms / 1e3) / 1e9, 1),
                       "frac": round(byt / (ms / 1e3) / 1e9 / peak, 4), "prune_ms": round(prune_ms, 5),
                       "attention_ms": round(step_ms, 5), "speedup_vs_dense": round(dense_ms / step_ms, 3)})
    sbytes = algorithmic_bytes(w, L, 0)["score"]
    del kv, st, stats, ws_dense, out_dense
    torch.cuda.empty_cache()
    return {"workload": f"{w.name}: B={w.B} Hq={w.Hq} Hkv={w.Hkv} D={w.D} P={w.P} "
                        f"{ctx_desc(w)}",
            "theta": "+inf", "score_ms": round(score_ms, 5),
            "score_gbs": round(sbytes / (score_ms / 1e3) / 1e9, 1),
            "dense_decode_ms": round(dense_ms, 5),
            "dense_decode_gbs": round(kv_bytes / (dense_ms / 1e3) / 1e9, 1), "points": points,
            "note": "decode over the kept blocks only (kept V pages + their scores); the scorer "
                    "reads every key whatever f is; attention_ms = score + prune + decode, against "
                    "a dense decode that reads K and V of every block"}


def pool_for(w, device) -> int | None:
    """The workload's page pool, capped to the largest power of two of pages
    (K + V) within a quarter of the free HBM: the mixed-batch recipe's 2^21
    pages would need 256 GB.  None: exactly the pages the sequences use."""
    if w.pool is None:
        return None
    free, _ = torch.cuda.mem_get_info(device)
    page_bytes = 2 * w.Hkv * w.P * w.D * 2
    cap = int(0.25 * free // page_bytes)
    return min(w.pool, 1 << max(10, cap.bit_length() - 1))


def sub_batches(B: int, n: int, weights=None) -> list[tuple[int, int]]:
    """Contiguous runs [lo, hi) that cover sequences 0 .. B-1 in order, never
    empty (fewer runs than n when B < n): as even in count as possible, or,
    with per-sequence `weights` (the blocks each reads), cut where the
    running weight crosses each i/n of the total."""
    n = max(1, min(n, B))
    if weights is None:
        bounds = [round(i * B / n) for i in range(n + 1)]
    else:
        cum = np.concatenate([[0.0], np.cumsum(np.asarray(weights, dtype=np.float64))])
        bounds = [0]
        for i in range(1, n):
            k = int(np.searchsorted(cum, cum[-1] * i / n))            # first prefix >= the target
            if k > 0 and abs(cum[k - 1] - cum[-1] * i / n) <= abs(cum[k] - cum[-1] * i / n):
                k -= 1
            bounds.append(min(max(k, bounds[-1] + 1), B - (n - i)))   # non-empty runs
        bounds.append(B)
    return list(zip(bounds[:-1], bounds[1:]))


class StepRunner:
    """One workload's inputs, buffers and the four calls of the step (score
    -> keep set -> decode over the kept blocks -> entropy / sample)."""

    def __init__(self, eti, w, device, prm, stream, H_target_frac=None):
        self.eti, self.w, self.prm, self.stream = eti, w, prm, stream
        self.pool = pool_for(w, device)
        self.kv = workloads.make_kv(w, device, pool=self.pool)
        self.lg = workloads.make_logits(w, device)
        if H_target_frac is not None:
            self.lg["H_target"].fill_(H_target_frac * math.log(w.V))
        g = w.Hq // w.Hkv
        self.step = eti.DecodeStep(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, w.V, device=device)
        self.stats = torch.empty((w.B, w.Hkv, w.max_blocks, g, 4), dtype=torch.float32, device=device)
        self.shape = (w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks)
        self.B_min = 1
        # threshold of this step: theta_next of the previous step's entropy (same logits)
        tau0 = self.lg["tau"].clone()
        self.step.sample(self.lg["logits"], self.lg["T_in"], self.lg["H_prev"], tau0, self.lg["H_target"],
                         params=prm, seed=w.seed)
        self.theta = self.step.theta_next.clone()
        self.L = self.kv["ctx_lens"].cpu().numpy()
        self.total_blocks = int((-(-self.L // w.P)).sum()) * w.Hkv
        # sub-batches of the overlapped step: contiguous runs of the batch whose
        # calls write into views of the same outputs, each with its own decode
        # workspace (two calls in flight must not share one)
        self.parts = []
        for lo, hi in sub_batches(w.B, SUB_BATCHES, weights=-(-self.L // w.P)):
            ws = torch.empty(eti.paged_decode_workspace_size(hi - lo, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, True),
                             dtype=torch.uint8, device=device)
            self.parts.append((lo, hi, (hi - lo, w.Hq, w.Hkv, w.D, w.P, w.max_blocks), ws))

    def attention_part(self, lo, hi, shape, ws, q=None, theta=None):
        """Score, keep set and decode of sequences [lo, hi) on the current
        stream (q and theta: the whole batch's, if not the runner's own)."""
        eti, kv, st = self.eti, self.kv, self.step
        q = (kv["q"] if q is None else q)[lo:hi]
        theta = (self.theta if theta is None else theta)[lo:hi]
        bt, cl = kv["block_table"][lo:hi], kv["ctx_lens"][lo:hi]
        eti.eti_score_blocks(q, kv["k_cache"], bt, cl, kv["scale"], self.stats[lo:hi],
                             token_scores=st.token_scores[lo:hi], num_pages=kv["num_pages"])
        eti.eti_prune_blocks(self.stats[lo:hi], bt, cl, shape, theta, self.B_min,
                             st.keep_mask[lo:hi], st.kept_idx[lo:hi], st.kept_cnt[lo:hi], st.err_attn[lo:hi],
                             kept_norm=st.kept_norm[lo:hi], num_pages=kv["num_pages"])
        eti.eti_paged_decode(q, kv["k_cache"], kv["v_cache"], bt, cl, kv["scale"], st.out[lo:hi],
                             st.err_dec[lo:hi], ws, kept_idx=st.kept_idx[lo:hi], kept_cnt=st.kept_cnt[lo:hi],
                             token_scores=st.token_scores[lo:hi], kept_norm=st.kept_norm[lo:hi],
                             num_pages=kv["num_pages"])

    def run(self, ev=None, offset=0, sched=None):
        """One step; with `ev` (5 events) an event between the calls, all four
        on the launching stream.  With `sched` = (side, subs) the step is
        overlapped: the sampling call (which reads only the logits and the
        per-sequence state) runs on `side`, and the attention half of each
        sub-batch (score, keep set, decode) on its own stream of `subs`; all
        fork at the step's start and the launching stream waits for them before
        the step ends."""
        eti, kv, st, w = self.eti, self.kv, self.step, self.w
        s = self.stream
        if sched is not None:
            side, subs = sched
            side.wait_stream(s)                  # fork
            st.sample(self.lg["logits"], self.lg["T_in"], self.lg["H_prev"], self.lg["tau"],
                      self.lg["H_target"], params=self.prm, seed=w.seed, offset=offset, stream=side)
            for part, sub in zip(self.parts, subs):
                sub.wait_stream(s)
                with torch.cuda.stream(sub):
                    self.attention_part(*part)
            for sub in subs[:len(self.parts)]:
                s.wait_stream(sub)               # join
            s.wait_stream(side)
            return
        if ev is not None:
            ev[0].record(s)
        eti.eti_score_blocks(kv["q"], kv["k_cache"], kv["block_table"], kv["ctx_lens"], kv["scale"],
                             self.stats, token_scores=st.token_scores, num_pages=kv["num_pages"])
        if ev is not None:
            ev[1].record(s)
        eti.eti_prune_blocks(self.stats, kv["block_table"], kv["ctx_lens"], self.shape, self.theta, self.B_min,
                             st.keep_mask, st.kept_idx, st.kept_cnt, st.err_attn, kept_norm=st.kept_norm,
                             num_pages=kv["num_pages"])
        if ev is not None:
            ev[2].record(s)
        eti.eti_paged_decode(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                             kv["scale"], st.out, st.err_dec, st.ws_dec, kept_idx=st.kept_idx,
                             kept_cnt=st.kept_cnt, token_scores=st.token_scores, kept_norm=st.kept_norm,
                             num_pages=kv["num_pages"])
        if ev is not None:
            ev[3].record(s)
        st.sample(self.lg["logits"], self.lg["T_in"], self.lg["H_prev"], self.lg["tau"], self.lg["H_target"],
                  params=self.prm, seed=w.seed, offset=offset)
        if ev is not None:
            ev[4].record(s)

    def kept(self) -> int:
        return int(self.step.kept_cnt.sum().item())


def timed_median(fn, flush_l2, stream, reps):
    """Median CUDA-event time (ms) of fn over reps calls, L2 flushed before each."""
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
    for i in range(reps + 2):
        flush_l2()
        if i >= 2:
            ev[i - 2][0].record(stream)
        fn()
        if i >= 2:
            ev[i - 2][1].record(stream)
    torch.cuda.synchronize()
    return statistics.median(e[0].elapsed_time(e[1]) for e in ev)


NAMES = ("score", "prune", "decode", "sample")


def kernel_pass(r, flush_l2, n, offset0):
    """Per-call times (ms, mean over n steps) from a pass with an event between calls."""
    evb = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(n)]
    for i in range(n):
        flush_l2()
        r.run(evb[i], offset=offset0 + i)
    torch.cuda.synchronize()
    return {nm: statistics.mean(evb[i][j].elapsed_time(evb[i][j + 1]) for i in range(n))
            for j, nm in enumerate(NAMES)}


def dense_decode_ms(r, flush_l2, reps=20):
    """The baseline the keep set is measured against: eti_paged_decode without
    kept lists (every block: q.K scored and p.V accumulated over K and V of
    every block, in the same library call)."""
    eti, kv, w = r.eti, r.kv, r.w
    ws = torch.empty(eti.paged_decode_workspace_size(w.B, w.Hq, w.Hkv, w.D, w.P, w.max_blocks, False),
                     dtype=torch.uint8, device=kv["q"].device)
    out = torch.empty_like(r.step.out)
    err = torch.empty_like(r.step.err_dec)

    def dense():
        eti.eti_paged_decode(kv["q"], kv["k_cache"], kv["v_cache"], kv["block_table"], kv["ctx_lens"],
                             kv["scale"], out, err, ws, num_pages=kv["num_pages"])
    ms = timed_median(dense, flush_l2, r.stream, reps)
    del ws, out, err
    return ms


def timed_steps(r, flush_l2, steps, offset0, sched=None):
    """Mean CUDA-event time (ms) of `steps` steps, L2 flushed before each."""
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(steps)]
    for i in range(steps):
        flush_l2()
        evs[i][0].record(r.stream)
        r.run(offset=offset0 + i, sched=sched)
        evs[i][1].record(r.stream)
    torch.cuda.synchronize()
    return statistics.mean(e[0].elapsed_time(e[1]) for e in evs)


def workload_summary(r, flush_l2, peak, steps, warmup, sched, offset0=0):
    """Step time, throughput, kept fraction and per-kernel times / fractions of
    the HBM peak for one workload (same timing rules as the main line)."""
    w = r.w
    for i in range(warmup):
        flush_l2()
        r.run(offset=offset0 + i, sched=sched)
    ms = timed_steps(r, flush_l2, steps, offset0 + warmup, sched)
    ms_seq = timed_steps(r, flush_l2, min(steps, 50), offset0 + warmup + steps)
    per = kernel_pass(r, flush_l2, min(steps, 50), offset0 + warmup + steps)
    kept = r.kept()
    ab = algorithmic_bytes(w, r.L, kept)
    gbs = {n: ab[n] / (per[n] / 1e3) / 1e9 for n in NAMES}
    out = {"workload": workload_desc(w), "steps": steps, "ms_per_step": round(ms, 5),
           "ms_per_step_sequential": round(ms_seq, 5),
           "tokens_per_s": round(w.B / (ms / 1e3), 1),
           "kept_fraction": round(kept / max(1, r.total_blocks), 4),
           "kernels_ms": {n: round(v, 5) for n, v in per.items()},
           "kernels_gbs": {n: round(v, 1) for n, v in gbs.items()},
           "kernels_frac_of_peak": {n: round(v / peak, 4) for n, v in gbs.items()}}
    if r.pool is not None:
        out["page_pool"] = r.pool
    return out


def read_floor(lg, flush_l2, stream, reps=50):
    """A size-matched read-only floor for the sampling pass: torch.sum over the
    same logits, L2 flushed before each call (median ms, GB/s)."""
    ms = timed_median(lambda: lg["logits"].sum(), flush_l2, stream, reps)
    byt = lg["logits"].numel() * 4
    return {"kernel": "torch.sum over the same logits", "ms": round(ms, 5),
            "gbs": round(byt / (ms / 1e3) / 1e9, 1)}


def ncu_record(kernel):
    """The committed ncu record of a kernel (bytes, instructions, ...), if its
    code is unchanged since that capture (else None)."""
    try:
        rec = json.load(open(os.path.join(ROOT, "profiles", "ncu_traffic.json")))[kernel]
        digest = source_digest(rec["sources"])
    except (OSError, KeyError, TypeError, ValueError):
        return None
    return rec if digest == rec["sha256"] else None


def run_gpu(args):
    import paper_2603_03310_gb300 as eti

    rank, world, local = dist_env()
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=device)
    eti.load()
    w = shard_workload(workloads.WORKLOADS[args.workload], rank)
    if args.batch:
        w = w.scaled(B=args.batch)   # a reduced case of the same shape (for profiling)
    prm = eti.ctrl_params()
    stream = torch.cuda.current_stream()
    # the overlapped step: the sampling call on one stream, each sub-batch's
    # attention half on another, of higher priority (the attention half is
    # the step's critical path; the sampling call fills the SMs it leaves)
    sched = (torch.cuda.Stream(device=device, priority=0),
             [torch.cuda.Stream(device=device, priority=-1) for _ in range(SUB_BATCHES)])
    r = StepRunner(eti, w, device, prm, stream)
    nparts = len(r.parts)
    L2 = torch.cuda.get_device_properties(device).L2_cache_size
    flush_w = torch.empty(max(2 * L2, 256 << 20), dtype=torch.uint8, device=device)
    flush_r = torch.ones(max(2 * L2, 256 << 20) // 4, dtype=torch.int32, device=device)

    def flush_l2():
        """Write a buffer of 2x L2, then read another one: the step's data is
        evicted and the flush's own dirty lines are written back before the
        timed region instead of inside its first kernel."""
        flush_w.zero_()
        flush_r.sum()

    try:
        peak, peak_src = float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        peak, peak_src = 6800.0, "fallback"

    for i in range(args.warmup):
        flush_l2()
        r.run(offset=i, sched=sched)
    torch.cuda.synchronize()
    kept = r.kept()
    total_blocks = r.total_blocks
    # the timed steps carry one event pair each (no event between the calls, so
    # every kernel keeps its programmatic launch overlap with the one before);
    # the per-kernel breakdown comes from a separate pass with an event per call
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    clock_log = None
    if args.clock_log:
        clock_log = args.clock_log.replace("{rank}", str(rank))
        os.makedirs(os.path.dirname(os.path.abspath(clock_log)), exist_ok=True)
    off = args.warmup
    with ClockSampler(local, clock_log) as clk:
        t0 = time.perf_counter()
        for i in range(args.steps):
            flush_l2()
            evs[i][0].record(stream)
            r.run(offset=off + i, sched=sched)
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        timed_samples = len(clk.lines)
        off += args.steps
        # the same step back to back for args.clock_seconds more, so that the
        # clock record holds enough samples whatever K is
        cp = None
        if args.clock_seconds > 0:
            ncp, t1 = 0, time.perf_counter()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            while time.perf_counter() - t1 < args.clock_seconds:
                for _ in range(50):
                    flush_l2()
                    r.run(offset=off + ncp, sched=sched)
                    ncp += 1
                torch.cuda.synchronize()
            e1.record(stream)
            torch.cuda.synchronize()
            off += ncp
            cp = {"steps": ncp, "seconds": round(time.perf_counter() - t1, 3),
                  "ms_per_step_with_flush": round(e0.elapsed_time(e1) / ncp, 5)}
    if world > 1:
        dist.barrier()
    step_ms = [evs[i][0].elapsed_time(evs[i][1]) for i in range(args.steps)]
    clocks = clk.summary()
    if clocks is not None:
        clocks["timed_region_samples"] = timed_samples
    if cp is not None and clocks is not None:
        cp["sm_mhz_median"] = clocks["sm_mhz"]
    mean_ms = kernel_pass(r, flush_l2, min(args.steps, 300), off)
    off += min(args.steps, 300)
    seq_ms = timed_steps(r, flush_l2, min(args.steps, 300), off)   # the four calls on one stream
    off += min(args.steps, 300)
    # share of the attention the keep set retains (outside the timed region;
    # a diagnostic never fails the run)
    try:
        kept_mass = kept_attention_mass(r.stats, r.step.keep_mask, r.kv["ctx_lens"], w.P)
    except Exception as ex:
        kept_mass = {"error": f"{type(ex).__name__}: {ex}"}
    ms_local = statistics.mean(step_ms)
    ms = max_over_ranks(ms_local, world, device)
    value, _ = aggregate([ms / 1e3] * world, w.B)
    if cp is not None:
        cp["kcycles_per_step"] = round(ms * (clocks or {}).get("sm_mhz", 0.0), 1)
    abytes = algorithmic_bytes(w, r.L, kept)
    dom = max(mean_ms, key=mean_ms.get)
    achieved = {n: abytes[n] / (mean_ms[n] / 1e3) / 1e9 for n in NAMES}
    rec_name = {"score": "score_blocks", "prune": "prune_finalize", "decode": "paged_decode",
                "sample": "entropy_sample"}
    rec = ncu_record(rec_name[dom])
    traffic = args.traffic if args.traffic is not None else (rec["bytes"] if rec else None)
    roof = {"kernel": {"score": "score_blocks", "prune": "prune_finalize",
                       "decode": "paged_decode (plan + decode; split segments merged in-kernel)",
                       "sample": "entropy_temp_sample (ticket clear + pass)"}[dom],
            "bound": "hbm", "achieved": round(achieved[dom], 1), "peak": peak, "unit": "GB/s",
            "frac": round(achieved[dom] / peak, 4), "peak_source": peak_src,
            "bytes_per_launch": abytes[dom], "ms_per_launch": round(mean_ms[dom], 5),
            "traffic": traffic,
            "traffic_note": "ncu dram read+write per launch of the main kernel (profiles/), "
                            "null if its source changed since the capture"}

    # the keep set against dense attention on the same batch (paper Section 6.7)
    attn_ms = mean_ms["score"] + mean_ms["prune"] + mean_ms["decode"]
    dms = dense_decode_ms(r, flush_l2)
    dense = {"dense_decode_ms": round(dms, 5), "attention_ms": round(attn_ms, 5),
             "speedup_vs_dense": round(dms / attn_ms, 3),
             "note": "attention_ms = score + keep set + decode over the kept blocks (kernels_ms); "
                     "dense = eti_paged_decode without kept lists on the same batch (every block "
                     "scored, then K and V of every block)"}
    # the sampling pass against a read-only pass over the same bytes
    floor = read_floor(r.lg, flush_l2, stream)
    srec = ncu_record("entropy_sample")
    sampling = {"ms": round(mean_ms["sample"], 5), "gbs": round(achieved["sample"], 1),
                "frac_of_peak": round(achieved["sample"] / peak, 4), "read_floor": floor,
                "frac_of_read_floor": round(floor["ms"] / mean_ms["sample"], 4),
                "inst_per_logit": (round(srec["inst_executed"] * 32 / (w.B * w.V), 2)
                                   if srec and srec.get("inst_executed") else None),
                "inst_note": "smsp__inst_executed x 32 lanes / logits of the pass kernel, from the "
                             "committed ncu record (null if the kernel changed since)"}

    # top-k entropy estimators (Section 2.1) on the same logits: cost next to the
    # exact pass, and how they track the exact entropy of the step
    est = None
    if not args.no_estimators:
        est = run_estimators(eti, r.lg, r.step, prm, w, flush_l2, stream)
        est["schedule_ms"] = run_schedule(eti, r.step, r.kv, w, stream)

    # end to end through the public API: host (pinned) inputs -> device -> step -> host results
    e2e = None if args.no_e2e else run_e2e(eti, r, args, device)
    if e2e is not None:
        e2e = aggregate_e2e(e2e, w.B, world, device)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, r.kv, r.lg, r.theta, r.B_min, budget_s=args.cpu_budget)
    main_desc = workload_desc(w)
    del r
    torch.cuda.empty_cache()

    sweep = None if args.no_sweep else run_keep_sweep(eti, device, flush_l2, stream, peak)

    # the other workloads (the same step and timing rules, fewer steps)
    others = None
    if not args.no_workloads:
        others = {}
        ksteps = max(20, min(args.steps, 200))
        for name in ("tiny", "long_ctx", "mixed_batch", "llama3_70b"):
            if name == args.workload:
                continue
            ow = shard_workload(workloads.WORKLOADS[name], rank)
            fracs = (0.1, 0.3, 0.5) if name == "llama3_70b" else (None,)
            res = []
            for f in fracs:
                ro = StepRunner(eti, ow, device, prm, stream, H_target_frac=f)
                s = workload_summary(ro, flush_l2, peak, ksteps, 5, sched)
                if f is not None:
                    s["H_target"] = f"{f} log V"
                res.append(s)
                del ro
                torch.cuda.empty_cache()
            others[name] = res[0] if len(res) == 1 else {"H_target_sweep": res}

    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16/fp32",
        "data": "synthetic (seeded; Llama-3-8B-shaped layer step)",
        "ms_per_step_sequential": round(seq_ms, 5),
        "config": {"workload": main_desc,
                   "streams": f"the sampling call on one stream and the attention half (score, keep set, "
                              f"decode) of each of {nparts} sub-batches (contiguous runs of the batch with "
                              f"about equal blocks) on its own, of higher priority, all forked at the step's "
                              f"start and joined before its end event; ms_per_step_sequential: the four "
                              f"calls over the whole batch on one stream",
                   "global_batch": w.B * world, "l2": "flushed before every step (2x L2 write, then 2x L2 read)",
                   "parallelism": f"replicas x{world} (independent batches)", "B_min": 1,
                   "theta": "theta_next of the step's own entropy (defaults)",
                   "kept_fraction": round(kept / max(1, total_blocks), 4)},
        "roofline": roof,
        "kernels_ms": {n: round(v, 5) for n, v in mean_ms.items()},
        "kernels_ms_note": "per call, from a separate pass with an event between calls (the timed "
                           "steps have none, so their sum can exceed ms_per_step)",
        "kernels_gbs": {n: round(v, 1) for n, v in achieved.items()},
        "entropy_sample_gbs": round(achieved["sample"], 1),
        "sampling": sampling,
        "attention_tbs": round((abytes["score"] + abytes["decode"]) / (attn_ms / 1e3) / 1e12, 3),
        "dense_baseline": dense,
        "gpu_launches": (5 * nparts + 2) * args.steps,
        "launches_per_step": {"score_blocks": nparts, "clear_words (keep-set error words)": nparts,
                              "prune_finalize": nparts, "decode_plan": nparts,
                              "paged_decode": nparts, "ets_clear (sampling tickets)": 1,
                              "entropy_sample": 1},
        "e2e": e2e,
        "estimators": est,
        "keep_sweep": sweep,
        "workloads": others,
        "kept_attention_mass": kept_mass,
        "wall_s_timed_region": round(wall, 4),
        "clocks": clocks,
        "clock_pass": cp,
    }
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_e2e(eti, r, args, device):
    """Same metric through the public API from pinned host buffers: per step the
    step's inputs (q, logits, per-sequence state, threshold) go host -> device and
    its results (attention output, token, entropy, temperature, threshold) come
    back.  Returns the figure and the time of each stage (an eager pass with
    events at the stage boundaries)."""
    # One byte buffer per direction for the small per-step data, so each
    # direction costs one copy (a small copy costs ~12 us whatever its size):
    #   [q | T_in H_prev H_target theta | tau theta_next tok H T_out surprisal err]
    # goes up as far as tau (q, the state, tau) and comes back from tau on.
    w, kv, lg, step, prm = r.w, r.kv, r.lg, r.step, r.prm
    B = w.B
    qb = kv["q"].numel() * 2
    row = B * 4
    n_in, n_all = qb + 5 * row, qb + 11 * row
    d_io = torch.zeros(n_all, dtype=torch.uint8, device=device)
    d_q = d_io[:qb].view(torch.bfloat16).view(kv["q"].shape)
    rows = d_io[qb:].view(torch.float32).view(11, B)
    T_in, H_prev, H_tgt, th, tau = rows[0], rows[1], rows[2], rows[3], rows[4]
    th_next, H_out, T_out, surp = rows[5], rows[7], rows[8], rows[9]
    tok, err = rows[6].view(torch.int32), rows[10].view(torch.int32)
    d_io[:qb].view(torch.bfloat16).copy_(kv["q"].reshape(-1))
    rows[:5].copy_(torch.stack([lg["T_in"], lg["H_prev"], lg["H_target"], r.theta, lg["tau"]]))
    h_in = d_io[:n_in].cpu().pin_memory()
    h_res = torch.empty(n_all - (qb + 4 * row), dtype=torch.uint8).pin_memory()
    h_logits = lg["logits"].cpu().pin_memory()
    d_logits = torch.empty_like(lg["logits"])
    h_out = torch.empty(step.out.shape, dtype=step.out.dtype).pin_memory()
    off_dev = torch.zeros(1, dtype=torch.int64, device=device)   # Philox offset, advanced by each call

    # The small inputs go up first; the logits (the bulk of the bytes) then go
    # up on a second stream, where the sampling call follows them and its
    # results come down, all while the attention half runs (each sub-batch's
    # on a stream of its own, as in the device-resident step); the attention
    # output comes down on the second stream once both are done.
    # The whole step (copies and calls, both streams) is captured once in a CUDA
    # graph and replayed every step, as a serving loop would; the sampling
    # offset lives in device memory (the call advances it), so every replay
    # draws fresh numbers.  If the capture is refused the same body runs eagerly.
    main = torch.cuda.current_stream()
    copy = torch.cuda.Stream(device=device)
    subs = [torch.cuda.Stream(device=device) for _ in r.parts]
    ev_out = torch.cuda.Event()
    stages = ("start", "logits_up_start", "logits_up_end", "small_up_end", "attention_end", "out_down_end",
              "sample_end", "results_down_end", "end")

    def body(cur, mk=None):
        rec = (lambda name, s: mk[name].record(s)) if mk is not None else (lambda name, s: None)
        rec("start", cur)
        # the small inputs go first: both uploads use the same copy engine, in
        # the order they are issued, and the attention half waits only for these
        d_io[:n_in].copy_(h_in, non_blocking=True)
        rec("small_up_end", cur)
        copy.wait_stream(cur)                                  # fork
        with torch.cuda.stream(copy):
            rec("logits_up_start", copy)
            d_logits.copy_(h_logits, non_blocking=True)
            rec("logits_up_end", copy)
            eti.eti_entropy_temp_sample(d_logits, T_in, H_prev, tau, H_tgt, tok, H_out, T_out, err,
                                        step.ws_ets, params=prm, seed=w.seed, offset_dev=off_dev,
                                        theta_next=th_next, tok_surprisal=surp, stream=copy)
            rec("sample_end", copy)
            h_res.copy_(d_io[qb + 4 * row:], non_blocking=True)
            rec("results_down_end", copy)
        for part, sub in zip(r.parts, subs):
            sub.wait_stream(cur)
            with torch.cuda.stream(sub):
                r.attention_part(*part, q=d_q, theta=th)
        for sub in subs:
            cur.wait_stream(sub)
        ev_out.record(cur)
        rec("attention_end", cur)
        with torch.cuda.stream(copy):
            copy.wait_event(ev_out)
            h_out.copy_(step.out, non_blocking=True)
            rec("out_down_end", copy)
        cur.wait_stream(copy)                                  # join
        rec("end", cur)

    for _ in range(args.warmup):
        body(main)
        main.synchronize()
    # where the time of one step goes (eager, events at the stage boundaries)
    n_bd = 20
    marks = [{s: torch.cuda.Event(enable_timing=True) for s in stages} for _ in range(n_bd)]
    for i in range(n_bd):
        body(main, marks[i])
        main.synchronize()

    def span(a, b):
        return statistics.median(m[a].elapsed_time(m[b]) for m in marks)
    breakdown = {
        "logits_upload_ms": span("logits_up_start", "logits_up_end"),
        "small_upload_ms": span("start", "small_up_end"),
        "attention_ms": span("small_up_end", "attention_end"),
        "out_download_ms": span("attention_end", "out_down_end"),
        "sample_ms": span("logits_up_end", "sample_end"),
        "results_download_ms": span("sample_end", "results_down_end"),
        "sampling_side_done_after_attention_ms": span("attention_end", "results_down_end"),
        "device_span_ms": span("start", "end"),
    }
    breakdown = {k: round(v, 4) for k, v in breakdown.items()}
    breakdown["note"] = ("eager pass with events at the stage boundaries (median of 20); the logits "
                         "upload, the sampling call and its results download run on a second stream "
                         "beside the attention half; sampling_side_done_after_attention_ms < 0 means "
                         "that side finished first; out_download_ms includes any wait for it")
    mode = "cuda graph replay (copies and calls of one step; sampling offset in device memory)"
    graph, gs = None, torch.cuda.Stream(device=device)
    try:
        gs.wait_stream(main)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=gs):
            body(gs)
        graph.replay()                 # on the current stream, like every replay below
        torch.cuda.synchronize()
    except Exception as ex:                                    # capture refused: eager steps
        graph = None
        mode = f"eager (graph capture refused: {type(ex).__name__})"
        torch.cuda.synchronize()
    o0 = int(off_dev.item())
    toks = []
    times = []
    for i in range(args.steps):
        t0 = time.perf_counter()
        if graph is not None:
            # replay() launches on the current stream (not the capture stream):
            # wait for the whole device, so each step's results are on the host
            graph.replay()
            torch.cuda.synchronize()
        else:
            body(main)
            main.synchronize()
        times.append(time.perf_counter() - t0)
        if i < 2:
            toks.append(h_res[2 * row:3 * row].view(torch.int32).clone())
    s = statistics.mean(times)
    bi = h_in.numel() + h_logits.numel() * 4
    bo = h_out.numel() * 2 + h_res.numel()
    breakdown["host_and_launch_ms"] = round(s * 1e3 - breakdown["device_span_ms"], 4)
    return {"value": round(w.B / s, 1), "unit": UNIT, "ms_per_step": round(s * 1e3, 4),
            "h2d_bytes_per_step": int(bi), "d2h_bytes_per_step": int(bo), "mode": mode,
            "offset_advanced": int(off_dev.item()) - o0,
            "fresh_tokens_per_replay": bool(len(toks) == 2 and not torch.equal(toks[0], toks[1])),
            "breakdown": breakdown,
            "l2": "not flushed: every step uploads its logits and reads "
                  f"{(key_bytes(w, kv) / 1e9):.2f} GB of keys plus the kept values, more than the L2"}


def key_bytes(w, kv) -> int:
    """Bytes of the key pages a step reads (every block of every sequence)."""
    L = kv["ctx_lens"].cpu().numpy()
    return int((-(-L // w.P)).sum()) * w.Hkv * w.P * w.D * 2


# ---------------------------------------------------------------------------
def oracle_step(w, sub, lg_np, theta_np, B_min, seqs, seed):
    """One decode step of the oracle on the given sequences (host arrays)."""
    import oracle
    r = oracle.score_prune(sub["q"], sub["k_cache"], sub["block_table"], sub["ctx_lens"],
                           sub["scale"], theta_np[seqs], B_min)
    oracle.paged_attention(sub["q"], sub["k_cache"], sub["v_cache"], sub["block_table"],
                           sub["ctx_lens"], sub["scale"], r["keep_mask"])
    oracle.entropy_temp_sample(lg_np["logits"][seqs], lg_np["T_in"][seqs], lg_np["H_prev"][seqs],
                               lg_np["tau"][seqs], lg_np["H_target"][seqs], seed=seed)


def _oracle_sample(w, kv, lg, theta, budget_s):
    """Pick a sample of sequences so one oracle step takes about budget_s seconds."""
    import oracle
    oracle.build()
    lg_np = {k: (v.cpu().numpy() if torch.is_tensor(v) else v) for k, v in lg.items()}
    theta_np = theta.cpu().numpy() if torch.is_tensor(theta) else theta
    n = 1
    while True:
        seqs = list(range(n))
        sub = workloads.gather_sequences(kv, seqs)
        t0 = time.perf_counter()
        oracle_step(w, sub, lg_np, theta_np, 1, seqs, w.seed)
        dt = time.perf_counter() - t0
        if n >= w.B or dt > budget_s / 4:
            break
        n = min(w.B, max(n + 1, int(n * min(8.0, budget_s / 2 / max(dt, 1e-3)))))
    return seqs, sub, lg_np, theta_np, dt


def cpu_baseline(w, kv, lg, theta, B_min, budget_s=15.0):
    import oracle
    seqs, sub, lg_np, theta_np, dt = _oracle_sample(w, kv, lg, theta, budget_s)
    t0 = time.perf_counter()
    reps = 0
    while True:
        oracle_step(w, sub, lg_np, theta_np, B_min, seqs, w.seed)
        reps += 1
        if time.perf_counter() - t0 > budget_s / 2:
            break
    s = (time.perf_counter() - t0) / reps
    return {"value": round(len(seqs) / s, 3), "unit": UNIT, "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": f"{len(seqs)} of {w.B} sequences of the same workload, full step "
                      f"(scores + keep set + attention + entropy/sample), {reps} rep(s), fp64 C + OpenMP"}


def run_reference(args):
    """The oracle as the reference arm, on this host's cores, rank 0 only."""
    rank, world, local = dist_env()
    if rank != 0:
        return
    import oracle
    oracle.build()
    w = workloads.WORKLOADS[args.workload]
    kv = workloads.make_kv(w, "cpu")
    lg = workloads.make_logits(w, "cpu")
    r = oracle.entropy_temp_sample(lg["logits"].numpy(), lg["T_in"].numpy(), lg["H_prev"].numpy(),
                                   lg["tau"].numpy(), lg["H_target"].numpy(), seed=w.seed)
    theta = r["theta_next"].astype(np.float32)
    budget = max(1.0, args.cpu_budget / max(1, args.steps + args.warmup))
    seqs, sub, lg_np, theta_np, _ = _oracle_sample(w, kv, lg, theta, budget)
    for _ in range(args.warmup):
        oracle_step(w, sub, lg_np, theta_np, 1, seqs, w.seed)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_step(w, sub, lg_np, theta_np, 1, seqs, w.seed)
        times.append(time.perf_counter() - t0)
    s = statistics.mean(times)
    v = round(len(seqs) / s, 3)
    sample = (f"{len(seqs)} of {w.B} sequences per step, full step (scores + keep set + "
              f"attention + entropy/sample), fp64 C + OpenMP")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(s * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; Llama-3-8B-shaped layer step)",
        "config": {"workload": workload_desc(w), "global_batch": w.B,
                   "oracle_sample": f"{len(seqs)} of {w.B} sequences per step"},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", choices=("eti", "reference"), default="eti")
    ap.add_argument("--workload", default="llama3_8b", choices=sorted(workloads.WORKLOADS))
    ap.add_argument("--cpu-budget", type=float, default=15.0,
                    help="seconds of oracle work for the CPU baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the long-context keep-fraction sweep (decode time against kept blocks)")
    ap.add_argument("--no-estimators", action="store_true",
                    help="skip the top-k entropy estimator line")
    ap.add_argument("--batch", type=int, default=None,
                    help="run the workload with this many sequences instead (a reduced case of the "
                         "same shape, e.g. for an ncu capture that must stay small)")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the other four workloads (tiny, long_ctx, mixed_batch, llama3_70b)")
    ap.add_argument("--clock-seconds", type=float, default=2.0,
                    help="seconds of back-to-back steps after the timed ones, under the clock sampler")
    ap.add_argument("--clock-log", default=None,
                    help="also write the raw nvidia-smi clock samples of the timed region to this "
                         "CSV file ({rank} is replaced by the rank)")
    ap.add_argument("--traffic", type=float, default=None,
                    help="ncu dram bytes per launch of the dominant kernel, if measured")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "eti":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
