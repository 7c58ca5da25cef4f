#!/usr/bin/env python3
"""Benchmark of one EfficientEdit verification step (arXiv 2506.02780, Sec. III-A)
on GB300: reuse-span match, tree prepare, L layers of tree-masked paged
attention, LM head + argmax + acceptance, KV compaction -- all in libee's
sm_103a kernels, captured as one CUDA graph per step.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config 7b]
    python bench.py --impl reference ...      # the fp64 CPU oracle, bounded sample

Prints one JSON line (rank 0).  value = verify steps/s over all ranks (each
rank verifies its own independent sequence batch: weak scaling, no data-path
collective); draft_tokens_per_s = steps/s x draft nodes per step (roots
excluded).  Inputs are seeded synthetic arrays of the configuration's shapes
(the paper's CanItEdit / CodeIF-Bench workloads are stood in for by them).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "verify steps/s and draft tokens verified/s at 1 GB300; % HBM roofline"
UNIT = "verify steps/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="7b", choices=["7b", "batched", "33b", "tiny", "long", "sweep"],
                    help="workload of the timed step (sweep: --profile only, the match, tree and "
                         "compaction kernels at the sweep's sizes)")
    ap.add_argument("--graphs", type=int, default=8, help="graphs replayed round-robin")
    ap.add_argument("--e2e-steps", type=int, default=300)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-rows", action="store_true",
                    help="skip the sweep-size measurement of the match, tree and compaction kernels")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the 33b and batched configurations timed after the headline")
    ap.add_argument("--no-variants", action="store_true",
                    help="skip the step variants (entropy k=3, k=5; in-place speculative K/V)")
    ap.add_argument("--profile", action="store_true",
                    help="run --steps eager steps and exit (for ncu captures: few launches, no timing)")
    ap.add_argument("--layers", type=int, default=None,
                    help="--profile only: build the workload with this many layers (small captures)")
    return ap.parse_args()


# DRAM bytes (read + write) per launch from one ncu capture of the kernel as it
# now stands (profiles/ names the capture); a kernel changed since has no entry.
TRAFFIC = {
    ("tree_verify_attn", "7b"): 9062144,          # profiles/attn_tc_7b.md
    ("tree_verify_attn", "33b"): 161879296,       # profiles/attn_tc_33b.md
    ("tree_verify_attn", "batched"): 246827008,   # profiles/attn_tc_batched.md
    ("lmhead_accept", "7b"): 1096552192,          # profiles/lmhead_accept_7b.md
    ("lmhead_accept", "long"): 1107782912,        # profiles/lmhead_accept_long.md
    ("chain_verify_attn", "long"): 30021120,      # profiles/attn_chain_long.md
}


def rank_seed(config, rank):
    """Seed of the synthetic batch a rank verifies: every rank owns an independent
    batch of sequences (the path partitions by sequence, so ranks never exchange
    data; only the timing scalar is reduced)."""
    return W.BASE_SEED + W.CONFIG_NAMES.index(config) + 1000 * rank


def reduce_max(value, world, device=None):
    """Max of a float over all ranks (identity when world == 1)."""
    if world <= 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ----------------------------------------------------------------------------
# algorithmic bytes and flops (what one launch must move / compute)
# ----------------------------------------------------------------------------

def algorithmic(w):
    Ts = np.diff(w.node_off)
    d, g = w.head_dim, w.n_q // w.n_kv
    depth = []
    for s in range(w.B):
        p = w.parent[w.node_off[s]:w.node_off[s + 1]]
        dep = np.zeros(len(p), np.int64)
        for i in range(1, len(p)):
            dep[i] = dep[p[i]] + 1
        depth.append(dep)
    keys = sum(int(w.ctx_len[s]) * int(Ts[s]) + int((depth[s] + 1).sum()) for s in range(w.B))
    total = w.total_nodes
    attn_bytes = (2 * int(w.ctx_len.sum()) * w.n_kv * d * 2          # K and V context, read once
                  + total * w.n_q * d * 2 + 2 * total * w.n_kv * d * 2  # Q, tree K/V
                  + total * w.n_q * d * 4)                              # fp32 output
    attn_flops = 4 * keys * w.n_q * d                                   # QK^T and PV, per layer
    lm_bytes = w.vocab * w.hidden * 2 + total * w.hidden * 2 + total * 4 * 2
    lm_flops = 2 * total * w.hidden * w.vocab
    acc = w.planted_accept
    comp_bytes = int((acc + 1).sum()) * w.layers * w.n_kv * d * 2 * 2 * 2  # K+V, read+write
    match_bytes = int(w.orig_off[-1]) * 4
    return dict(attn_bytes=attn_bytes, attn_flops=attn_flops, lm_bytes=lm_bytes, lm_flops=lm_flops,
                comp_bytes=comp_bytes, match_bytes=match_bytes, draft_nodes=int((Ts - 1).sum()))


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------

class ClockSampler:
    """nvidia-smi samples of the SM clock and the throttle reasons every 20 ms,
    each with its timestamp.  start() returns once the first sample is in (so
    sampling is live before the region begins), mark_begin()/mark_end()
    bracket the timed region on the host clock, and stop() summarises the
    samples taken inside it (see summarize_clock_rows)."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    PERIOD_MS = 20

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.file = None
        self.t_begin = None
        self.t_end = None

    def start(self, wait_s=3.0):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", delete=False, suffix=".csv")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", str(self.PERIOD_MS)],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        t0 = time.time()
        while time.time() - t0 < wait_s and self.proc.poll() is None:
            if os.path.getsize(self.file.name) > 0:
                break
            time.sleep(0.01)

    def mark_begin(self):
        self.t_begin = time.time()

    def mark_end(self):
        self.t_end = time.time()

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [r.split(",") for r in self.file.read().strip().splitlines() if r.strip()]
        self.file.close()
        os.unlink(self.file.name)
        return summarize_clock_rows(rows, self.t_begin, self.t_end)


def _clock_row_time(stamp):
    """nvidia-smi's timestamp ("YYYY/MM/DD HH:MM:SS.mmm", local time) in seconds
    since the epoch, or None."""
    import datetime
    try:
        return datetime.datetime.strptime(stamp.strip(), "%Y/%m/%d %H:%M:%S.%f").timestamp()
    except ValueError:
        return None


def summarize_clock_rows(rows, t_begin=None, t_end=None):
    """Median SM clock, maximum clock, active throttle reasons and sample count
    of the rows taken inside [t_begin, t_end] (host clock).  A region shorter
    than the sampling period may hold none: then the nearest sample before and
    the nearest after it stand in (``samples`` counts the rows used,
    ``samples_in_region`` those inside).  Without marks every row counts."""
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    parsed = []
    for r in rows:
        try:
            parsed.append((_clock_row_time(r[0]), float(r[1]), float(r[2]),
                           {nm for nm, v in zip(names, r[5:9]) if v.strip().lower() == "active"}))
        except (ValueError, IndexError):
            continue
    if not parsed:
        return None
    use, inside = parsed, None
    if t_begin is not None and t_end is not None and all(p[0] is not None for p in parsed):
        inside = [p for p in parsed if t_begin <= p[0] <= t_end]
        use = inside
        if not inside:
            before = [p for p in parsed if p[0] < t_begin]
            after = [p for p in parsed if p[0] > t_end]
            use = ([max(before, key=lambda p: p[0])] if before else []) + \
                  ([min(after, key=lambda p: p[0])] if after else [])
        if not use:
            return None
    out = {"sm_mhz": float(np.median([p[1] for p in use])), "sm_max_mhz": max(p[2] for p in use),
           "reasons": sorted(set().union(*(p[3] for p in use))), "samples": len(use)}
    if inside is not None:
        out["samples_in_region"] = len(inside)
        out["region_ms"] = round(1e3 * (t_end - t_begin), 2)
    return out


BAD_CLOCK_REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")


def clocks_rejected(clk, low=0.8):
    """Why a timed region's clock record voids its number, or None when it
    stands: a hardware or thermal slowdown seen during the region, or a median
    SM clock below ``low`` of the maximum with no reason given (a clock lock
    left behind by another user of the GPU).  sw_power_cap is kept (normal under
    a dense load on a power-capped part) and noted in the record."""
    if not clk:
        return None
    bad = [r for r in clk.get("reasons", []) if r in BAD_CLOCK_REASONS]
    if bad:
        return ",".join(bad)
    mx = clk.get("sm_max_mhz", 0.0)
    if mx > 0 and clk.get("sm_mhz", mx) < low * mx and not clk.get("reasons"):
        return "sm clocks %.0f of %.0f MHz with no reason" % (clk["sm_mhz"], mx)
    return None


# ----------------------------------------------------------------------------
# CPU baseline: the fp64 oracle on a bounded sample, scaled to a full step
# ----------------------------------------------------------------------------

def oracle_step_time(w, attn_nodes=None, lm_rows=None):
    """Time the oracle on a sample of one step and scale it to the full step.

    Sample: attention of ``attn_nodes`` tree nodes (all heads) of layer 0, the
    LM head over vocabulary rows 0..lm_rows-1, compaction of layer 0; match,
    tree structure and acceptance whole.  Returns (full-step seconds, sampled
    seconds, description)."""
    import oracle as O
    n_att = w.total_nodes if attn_nodes is None else max(1, min(int(attn_nodes), w.total_nodes))
    rows_n = max(1, w.vocab // 16) if lm_rows is None else max(1, min(int(lm_rows), w.vocab))
    nodes = np.linspace(0, w.total_nodes - 1, n_att).round().astype(int).tolist()
    raw = lambda x: x.detach().cpu().contiguous().view(torch.int16).numpy()  # noqa: E731
    chain = w.max_T > 128     # linear drafts verified in place (long reuse drafts)
    if chain:                 # set-up, not timed: the drafts' K/V where a K/V projection writes them
        pk, pv = O.tree_kv_to_cache(raw(w.k_tree[:1]), raw(w.v_tree[:1]), raw(w.k_cache[:1]),
                                    raw(w.v_cache[:1]), w.block_table, w.ctx_len, w.node_off)
        pk_t, pv_t = torch.from_numpy(pk[0]).view(torch.bfloat16), torch.from_numpy(pv[0]).view(torch.bfloat16)
    t0 = time.perf_counter()
    O.match_reuse(w.orig_tokens, w.orig_off, w.tail, w.cursor, w.max_matches)
    t1 = time.perf_counter()
    if not chain:
        depth, anc = O.tree_prepare(w.parent, w.node_off)
    t2 = time.perf_counter()
    if chain:
        O.chain_attention(w.q[0], pk_t, pv_t, w.block_table, w.ctx_len, w.node_off, nodes=nodes)
    else:
        O.tree_attention(w.q[0], w.k_tree[0], w.v_tree[0], w.k_cache[0], w.v_cache[0], w.block_table,
                         w.ctx_len, w.node_off, anc, nodes=nodes)
    t3 = time.perf_counter()
    logits, _ = O.lm_head_logits(w.hidden_states, w.lm_w, rows=slice(0, rows_n))
    am = np.argmax(logits, axis=1).astype(np.int32)
    t4 = time.perf_counter()
    if chain:
        acc, path, bonus = O.accept_chain(am, w.draft_tok, w.node_off, w.max_T)
    else:
        acc, path, bonus = O.accept_path(am, w.draft_tok, w.parent, w.node_off, w.max_T)
    t5 = time.perf_counter()
    if chain:
        O.kv_compact_inplace(pk, pv, w.block_table, w.ctx_len, w.node_off, path, acc)
    else:
        O.kv_compact(raw(w.k_tree[:1]), raw(w.v_tree[:1]), raw(w.k_cache[:1]), raw(w.v_cache[:1]),
                     w.block_table, w.ctx_len, w.node_off, path, acc)
    t6 = time.perf_counter()
    a_scale = w.layers * w.total_nodes / n_att
    l_scale = w.vocab / rows_n
    full = ((t1 - t0) + (t2 - t1) + a_scale * (t3 - t2) + l_scale * (t4 - t3) + (t5 - t4)
            + w.layers * (t6 - t5))
    sample = (f"{w.name}: attention of {n_att}/{w.total_nodes} nodes of layer 0 of {w.layers} "
              f"(x{a_scale:.1f}), LM head over vocab rows 0..{rows_n - 1} of {w.vocab} (x{l_scale:.1f}), "
              f"compaction of layer 0 (x{w.layers}), match/tree/acceptance whole; sampled work "
              f"{t6 - t0:.2f} s scaled to one full step")
    return full, t6 - t0, sample


def oracle_repeat(w, budget_s):
    """The default sample (every node of layer 0, 1/16 of the vocabulary)
    repeated until about ``budget_s`` seconds of CPU work, each repetition
    scaled to one full step.  Returns (mean full-step seconds, description)."""
    fulls, spent_all, sample = [], 0.0, ""
    while not fulls or (spent_all < budget_s and len(fulls) < 200):
        full, spent, sample = oracle_step_time(w)
        fulls.append(full)
        spent_all += spent
    return float(np.mean(fulls)), f"{sample}; repeated {len(fulls)} times ({spent_all:.1f} s of CPU work), mean"


def oracle_single_thread(config, layers, vocab, budget_s=10.0, timeout_s=120):
    """The same oracle sample timed in a child process held to one thread
    (BLAS, OpenMP and torch; no GPU visible).  The child draws the
    configuration's inputs on the CPU with only what the sample reads -- layer
    0 and the first 1/16 of the vocabulary's weight rows -- and scales by the
    full layer count and vocabulary.  Never raises: a failure is reported in
    the returned record."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               NUMEXPR_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    code = ("import json, sys, torch\n"
            "torch.set_num_threads(1)\n"
            f"sys.path.insert(0, {ROOT!r})\n"
            "import bench, workloads as W\n"
            f"w = W.build({config!r}, device='cpu', layers=1, vocab={max(1, int(vocab) // 16)})\n"
            f"w.layers, w.vocab = {int(layers)}, {int(vocab)}\n"
            f"full, sample = bench.oracle_repeat(w, {float(budget_s)!r})\n"
            "print(json.dumps({'full_s': full, 'sample': sample}))\n")
    try:
        r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                           timeout=timeout_s)
        if r.returncode != 0:
            return {"error": (r.stderr or "")[-300:]}
        d = json.loads(r.stdout.strip().splitlines()[-1])
        return {"value": round(1.0 / d["full_s"], 6), "unit": UNIT, "cores": 1, "kind": "oracle",
                "sample": d["sample"] + " (one thread, inputs drawn on the CPU)"}
    except Exception as e:  # timing the baseline must never fail the benchmark
        return {"error": f"{type(e).__name__}: {e}"[:300]}


def oracle_sample_size(w, budget_s):
    """(attention nodes, LM-head vocabulary rows) of an oracle sample that takes
    about ``budget_s`` seconds: unit costs are calibrated on a minimal sample
    (one node, 256 rows) and both parts grown by the same factor."""
    probe_nodes, probe_rows = 1, min(w.vocab, 256)
    _, spent, _ = oracle_step_time(w, attn_nodes=probe_nodes, lm_rows=probe_rows)
    grow = max(1.0, budget_s / max(spent, 1e-4))
    return (max(1, min(w.total_nodes, int(probe_nodes * grow))),
            max(1, min(w.vocab, int(probe_rows * grow))))


SWEEP_TEXT = ("sweep: 32 sequences of 65,536-token code (30% in repeated 8-token segments), n in {2, 4, 8}; "
              "accept lengths U[1, 128] compacted over 28 layers of 7B-shaped K/V")


def sweep_inputs(dev, n, layers):
    """The reuse-matching and compaction sweep at full size (one seed per n)."""
    return W.build("sweep", device=dev, n=n, layers=layers,
                   seed=W.BASE_SEED + W.CONFIG_NAMES.index("sweep") + n)


def sweep_rows(dev, stream, copies=16, reps=32):
    """The hot path's small kernels at the sweep's sizes.  Device time per call
    from a CUDA graph of `reps` calls between two events (the best of 5
    replays).  The match cycles through `copies` copies of the code (134 MB,
    more than L2 holds, so every call reads from DRAM); one compaction moves more
    than L2 holds.  Algorithmic bytes: the code from each cursor on (4 B a token)
    for the match; K and V of every committed entry read and written, all
    layers, for the compaction; parents in, depth and ancestor masks out for the
    tree."""
    import paper_2506_02780_gb300 as E
    peaks, src = load_peaks()
    hbm = peaks["hbm_gbs"]
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device=dev)  # noqa: E731

    def timed(fn):
        with torch.cuda.stream(stream):
            fn(0)
            stream.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for k in range(reps):
                    fn(k)
            g.replay()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            best = float("inf")
            for _ in range(5):
                a.record(stream)
                g.replay()
                b.record(stream)
                b.synchronize()
                best = min(best, a.elapsed_time(b) / reps)
        return best * 1e-3          # seconds per call

    def row(sec, nbytes, **extra):
        gbs = nbytes / sec / 1e9
        return dict(us=round(sec * 1e6, 2), bytes=int(nbytes), achieved_gbs=round(gbs, 1),
                    frac=round(gbs / hbm, 4), **extra)

    out = {"workload": SWEEP_TEXT, "peak": f"HBM copy {hbm} GB/s ({src})", "match_reuse": {}}
    for n in (2, 4, 8):
        w = sweep_inputs(dev, n, 28 if n == 4 else 1)
        orig = [i32(w.orig_tokens) for _ in range(copies)]
        off = torch.as_tensor(w.orig_off, device=dev)
        tail, cur = i32(w.tail), i32(w.cursor)
        mp = torch.empty((w.B, 16), dtype=torch.int32, device=dev)
        nm = torch.empty(w.B, dtype=torch.int32, device=dev)
        ws = E.new_workspace(w.B, w.total_nodes, 1, 0, device=dev)
        sec = timed(lambda k: E.ee_match_reuse(orig[k % copies], off, tail, cur, 16, mp, nm, ws, stream))
        region = sum(int(w.orig_off[s + 1] - w.orig_off[s]) - int(w.cursor[s]) for s in range(w.B))
        out["match_reuse"][f"n{n}"] = row(sec, 4 * region)
        if E.ee_read_errors(ws):
            raise RuntimeError("device error in the match sweep")
        if n == 4:
            parent, node_off = i32(w.parent), i32(w.node_off)
            depth = torch.empty(w.total_nodes, dtype=torch.int32, device=dev)
            anc = torch.empty((w.total_nodes, 2), dtype=torch.int64, device=dev)
            sec = timed(lambda k: E.ee_tree_prepare(parent, node_off, depth, anc, ws, stream))
            out["tree_prepare"] = row(sec, w.total_nodes * (4 + 4 + 16) + 4 * (w.B + 1), nodes=w.total_nodes)
            path = np.full((w.B, w.max_T), -1, np.int32)
            for s in range(w.B):
                path[s, :len(w.planted_path[s])] = w.planted_path[s]
            path_d, acc_d, bt, ctx = i32(path), i32(w.planted_accept), i32(w.block_table), i32(w.ctx_len)
            ctx_out = torch.empty(w.B, dtype=torch.int32, device=dev)
            dst = torch.empty((w.B, w.max_T), dtype=torch.int32, device=dev)
            sec = timed(lambda k: E.ee_kv_compact(w.k_tree, w.v_tree, w.k_cache, w.v_cache, bt, ctx, ctx_out,
                                                  node_off, path_d, acc_d, dst, ws, stream))
            entries = int((np.asarray(w.planted_accept) + 1).sum())
            out["kv_compact"] = row(sec, entries * w.layers * w.n_kv * w.head_dim * 2 * 2 * 2, entries=entries,
                                    layers=w.layers)
            if E.ee_read_errors(ws):
                raise RuntimeError("device error in the compaction sweep")
        del w, orig
    torch.cuda.empty_cache()
    return out


def oracle_rows_time():
    """The oracle on the sweep's rows: the match (n = 4) whole, the compaction
    of 2 of the 28 layers scaled by 14."""
    import oracle as O
    w = sweep_inputs("cpu", 4, 2)
    raw = lambda x: x.detach().cpu().contiguous().view(torch.int16).numpy()  # noqa: E731
    path = np.full((w.B, w.max_T), -1, np.int32)
    for s in range(w.B):
        path[s, :len(w.planted_path[s])] = w.planted_path[s]
    t0 = time.perf_counter()
    O.match_reuse(w.orig_tokens, w.orig_off, w.tail, w.cursor, 16)
    t1 = time.perf_counter()
    O.kv_compact(raw(w.k_tree), raw(w.v_tree), raw(w.k_cache), raw(w.v_cache), w.block_table, w.ctx_len,
                 w.node_off, path, w.planted_accept)
    t2 = time.perf_counter()
    return {"match_reuse_n4_s": round(t1 - t0, 4), "kv_compact_s": round((t2 - t1) * 14, 4),
            "sample": "sweep, n = 4: the match whole; the compaction of 2 of the 28 layers (x14)"}


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ----------------------------------------------------------------------------
# our arm
# ----------------------------------------------------------------------------

def run_profile(args, local_rank):
    """Eager steps only: every libee kernel launches --steps times, nothing else runs
    between them, no graphs and no timing (what an ncu capture wants)."""
    import paper_2506_02780_gb300 as E
    from paper_2506_02780_gb300 import build as B
    from paper_2506_02780_gb300 import step as S
    B.build_lib()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    if args.config == "sweep":
        # the match (n = 4), tree and compaction kernels, each --steps times
        w = sweep_inputs(dev, 4, 28 if args.layers is None else args.layers)
        i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device=dev)  # noqa: E731
        ws = E.new_workspace(w.B, w.total_nodes, 1, 0, device=dev)
        mp = torch.empty((w.B, 16), dtype=torch.int32, device=dev)
        nm = torch.empty(w.B, dtype=torch.int32, device=dev)
        depth = torch.empty(w.total_nodes, dtype=torch.int32, device=dev)
        anc = torch.empty((w.total_nodes, 2), dtype=torch.int64, device=dev)
        path = np.full((w.B, w.max_T), -1, np.int32)
        for s in range(w.B):
            path[s, :len(w.planted_path[s])] = w.planted_path[s]
        ctx_out = torch.empty(w.B, dtype=torch.int32, device=dev)
        dst = torch.empty((w.B, w.max_T), dtype=torch.int32, device=dev)
        orig, off, tail, cur = (i32(w.orig_tokens), torch.as_tensor(w.orig_off, device=dev), i32(w.tail),
                                i32(w.cursor))
        parent, node_off, path_d, acc_d = i32(w.parent), i32(w.node_off), i32(path), i32(w.planted_accept)
        bt, ctx = i32(w.block_table), i32(w.ctx_len)
        torch.cuda.synchronize(dev)
        for _ in range(args.steps):
            E.ee_match_reuse(orig, off, tail, cur, 16, mp, nm, ws)
            E.ee_tree_prepare(parent, node_off, depth, anc, ws)
            E.ee_kv_compact(w.k_tree, w.v_tree, w.k_cache, w.v_cache, bt, ctx, ctx_out, node_off, path_d, acc_d,
                            dst, ws)
        torch.cuda.synchronize(dev)
        bits = E.ee_read_errors(ws)
        print(json.dumps({"profile": "sweep", "steps": args.steps, "device_errors": bits}), flush=True)
        return 0 if bits == 0 else 1
    over = {} if args.layers is None else {"layers": args.layers}
    w = W.build(args.config, device=dev, **over)
    st = S.from_workload(w, device=dev, keep_layers=False)
    torch.cuda.synchronize(dev)
    for _ in range(args.steps):
        st.run()
    torch.cuda.synchronize(dev)
    bits = E.ee_read_errors(st.ws)
    print(json.dumps({"profile": args.config, "steps": args.steps, "device_errors": bits,
                      "accept_len": st.accept_len.tolist()}), flush=True)
    return 0 if bits == 0 else 1


def run_ours(args, rank, world, local_rank):
    import paper_2506_02780_gb300 as E
    from paper_2506_02780_gb300 import build as B
    from paper_2506_02780_gb300 import step as S
    B.build_lib()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    w = W.build(args.config, seed=rank_seed(args.config, rank), device=dev)
    alg = algorithmic(w)
    st = S.from_workload(w, device=dev, keep_layers=False)
    stream = torch.cuda.Stream(device=dev)
    L = w.layers

    # Two graph pools of the same step: plain graphs (no event nodes, they time
    # the headline) and graphs with three external timing events (before the
    # first attention layer, after the last one, after the LM head) that time
    # the kernels live.  An event node between kernels costs several
    # microseconds, so the headline is never taken from instrumented graphs.
    try:
        mk = lambda: torch.cuda.Event(enable_timing=True, external=True)  # noqa: E731
        mk()
        phase_events = True
    except TypeError:
        phase_events = False
    plain, graphs, evsets = [], [], []
    with torch.cuda.stream(stream):
        st.run(stream)
        stream.synchronize()
        for _ in range(max(1, args.graphs)):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                run_instrumented(st, stream, None)
            plain.append(g)
            if phase_events:
                g = torch.cuda.CUDAGraph()
                evs = [mk() for _ in range(3)]
                with torch.cuda.graph(g, stream=stream):
                    run_instrumented(st, stream, evs)
                graphs.append(g)
                evsets.append(evs)
    stream.synchronize()
    assert E.ee_read_errors(st.ws, stream) == 0

    G = len(plain)
    acc_ms = np.zeros(2)
    n_acc = 0

    def harvest(j):
        nonlocal n_acc
        evs = evsets[j]
        evs[-1].synchronize()
        acc_ms[0] += evs[0].elapsed_time(evs[1])
        acc_ms[1] += evs[1].elapsed_time(evs[2])
        n_acc += 1

    def timed(pool, steps, harvest_fn=None):
        """Replay `steps` graphs round-robin between two events; ms per step."""
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        pending = [False] * len(pool)
        with torch.cuda.stream(stream):
            t0.record(stream)
            for i in range(steps):
                j = i % len(pool)
                if harvest_fn and pending[j]:
                    harvest_fn(j)
                pool[j].replay()
                pending[j] = True
            t1.record(stream)
        t1.synchronize()
        if harvest_fn:
            for j in range(len(pool)):
                if pending[j]:
                    harvest_fn(j)
        return t0.elapsed_time(t1) / steps

    for i in range(args.warmup):
        plain[i % G].replay()
        if phase_events:
            graphs[i % G].replay()
    stream.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clocks = ClockSampler(dev.index)
    if not args.no_clocks:
        clocks.start()
    torch.cuda.synchronize(dev)
    clocks.mark_begin()
    ms_step = timed(plain, args.steps)
    torch.cuda.synchronize(dev)
    clocks.mark_end()
    ms_step = reduce_max(ms_step, world, dev)
    ms_step_instr = timed(graphs, max(1, args.steps // 2), harvest) if phase_events else None
    torch.cuda.synchronize(dev)
    if world > 1:
        torch.distributed.barrier()
    clk = None if args.no_clocks else clocks.stop()
    # a region whose clocks void it is measured once more (every rank agrees)
    why = clocks_rejected(clk)
    if reduce_max(1.0 if why else 0.0, world, dev) > 0:
        first = {"ms_per_step": round(ms_step, 5), "clocks": clk, "rejected": why or "on another rank"}
        if world > 1:
            torch.distributed.barrier()
        clocks = ClockSampler(dev.index)
        clocks.start()
        torch.cuda.synchronize(dev)
        clocks.mark_begin()
        ms_step = timed(plain, args.steps)
        torch.cuda.synchronize(dev)
        clocks.mark_end()
        ms_step = reduce_max(ms_step, world, dev)
        if world > 1:
            torch.distributed.barrier()
        clk = clocks.stop() or {}
        clk["remeasured_after"] = first

    # the same step under the entropy-aware rule (Sec. III-B) for the generated
    # branches, with the paper's two settings of k (Sec. IV-E: 3 and 5)
    variants = {}
    if not args.no_variants and w.lm_w is not None and not st.chain:   # the rules take trees
        for k in (3, 5):
            sv = S.from_workload(w, device=dev, keep_layers=False, verify=("entropy", k))
            pool = []
            with torch.cuda.stream(stream):
                sv.run(stream)
                stream.synchronize()
                for _ in range(2):
                    g = torch.cuda.CUDAGraph()
                    with torch.cuda.graph(g, stream=stream):
                        sv.run(stream)
                    pool.append(g)
            for i in range(max(3, args.warmup // 4)):
                pool[i % 2].replay()
            stream.synchronize()
            ms_v = timed(pool, max(8, args.steps // 4))
            assert E.ee_read_errors(sv.ws, stream) == 0
            variants[f"entropy_k{k}"] = {
                "value": round(world * 1e3 / ms_v, 2), "ms_per_step": round(ms_v, 5),
                "accept_len": [int(a) for a in sv.accept_len.cpu().tolist()[:8]],
                "greedy_accept_len": [int(a) for a in st.accept_len.cpu().tolist()[:8]]}
            del pool, sv
    # the same step with in-place speculative K/V: the tree's K/V already in the
    # cache after each context, compaction moving only the path entries that are
    # out of place (none for a reuse chain)
    if not args.no_variants and not st.chain:     # linear drafts are verified in place already
        sv = S.from_workload(w, device=dev, keep_layers=False, inplace_kv=True)
        pool = []
        with torch.cuda.stream(stream):
            sv.run(stream)
            stream.synchronize()
            for _ in range(2):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    sv.run(stream)
                pool.append(g)
        for i in range(max(3, args.warmup // 4)):
            pool[i % 2].replay()
        stream.synchronize()
        ms_v = timed(pool, max(8, args.steps // 4))
        assert E.ee_read_errors(sv.ws, stream) == 0
        variants["inplace_kv"] = {
            "value": round(world * 1e3 / ms_v, 2), "ms_per_step": round(ms_v, 5),
            "attention_launch": E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, int(w.ctx_len.max()),
                                               inplace=True),
            "accept_len": [int(a) for a in sv.accept_len.cpu().tolist()[:8]]}
        del pool, sv
    if not args.no_variants and not st.chain and args.config == "7b":
        variants["edit_session"] = session_variant(w, dev, stream)
    assert E.ee_read_errors(st.ws, stream) == 0

    # ---- end to end: host inputs -> device -> step -> host results ---------
    e2e = run_e2e(st, plain[0], stream, args.e2e_steps, dev, world)

    # the match, tree and compaction kernels at the sweep's sizes (after the timed regions)
    rows = None if (args.no_rows or rank != 0) else sweep_rows(dev, stream)

    peaks, peak_src = load_peaks()
    per = (acc_ms / max(n_acc, 1)) if phase_events and n_acc else None
    kernels = {}
    rl = {}
    roofline = None
    if per is not None:
        attn_ms = float(per[0]) / L
        kernels = {
            "attention_per_layer_us": round(1e3 * attn_ms, 2),
            "attention_all_layers_us": round(1e3 * float(per[0]), 2),
            "lmhead_accept_us": round(1e3 * float(per[1]), 2),
            "instrumented_ms_per_step": round(ms_step_instr, 5),
            "note": "kernel phases timed live by three external events per step in a second "
                    "pass; attention per layer includes the launch gap between layers",
        }
        hbm = peaks["hbm_gbs"]
        tf = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
        cand = {
            "lmhead_accept": dict(ms=float(per[1]), bytes=alg["lm_bytes"], flops=alg["lm_flops"],
                                  launches=1),
            ("chain_verify_attn" if st.chain else "tree_verify_attn"):
                dict(ms=attn_ms, bytes=alg["attn_bytes"], flops=alg["attn_flops"], launches=L),
        }
        for name, c in cand.items():
            t_s = c["ms"] * 1e-3
            gbs = c["bytes"] / t_s / 1e9
            tfs = c["flops"] / t_s / 1e12
            if c["bytes"] / (hbm * 1e9) >= c["flops"] / (tf * 1e12):
                rl[name] = {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm, "unit": "GB/s",
                            "frac": round(gbs / hbm, 4)}
            else:
                rl[name] = {"bound": "tensor", "achieved": round(tfs, 2), "peak": tf, "unit": "TFLOP/s",
                            "frac": round(tfs / tf, 4)}
            rl[name].update({"hbm_frac": round(gbs / hbm, 4), "us_per_launch": round(1e3 * c["ms"], 2),
                             "share_of_step": round(c["ms"] * c["launches"] / ms_step_instr, 4),
                             "peak_source": f"{peak_src} ({'copy' if rl[name]['unit'] == 'GB/s' else 'sustained'})",
                             "traffic": TRAFFIC.get((name, args.config))})
        dom = max(cand, key=lambda n: cand[n]["ms"] * cand[n]["launches"])
        roofline = dict(rl[dom], kernel=dom)
    step_rl = None
    if rank == 0:
        hbm = peaks["hbm_gbs"]
        tf = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
        # the step against the HBM roofline on the K/V and LM-head weight bytes it must read, and
        # against the sum of its two big kernels' own floors (each the larger of bytes / HBM peak
        # and flops / tensor peak)
        kvw = w.layers * 2 * int(w.ctx_len.sum()) * w.n_kv * w.head_dim * 2 + w.vocab * w.hidden * 2
        floor_s = (w.layers * max(alg["attn_bytes"] / (hbm * 1e9), alg["attn_flops"] / (tf * 1e12))
                   + max(alg["lm_bytes"] / (hbm * 1e9), alg["lm_flops"] / (tf * 1e12)))
        step_rl = {"kv_weight_bytes": kvw, "achieved_gbs": round(kvw / (ms_step * 1e-3) / 1e9, 1),
                   "hbm_frac": round(kvw / (ms_step * 1e-3) / (hbm * 1e9), 4),
                   "floor_us": round(floor_s * 1e6, 1), "frac_of_floor": round(floor_s / (ms_step * 1e-3), 4),
                   "peaks": f"{peak_src}: HBM copy {hbm} GB/s, bf16 sustained {tf} TFLOP/s"}

    steps_per_s = world * 1e3 / ms_step
    out = {
        "metric": METRIC, "value": round(steps_per_s, 2), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; stands in for CanItEdit / CodeIF-Bench edit sessions)",
        "config": dict(W.describe(w), workload=args.config + ": " + _config_text(args.config),
                       l2="inputs larger than L2 (%.2f GB touched per step)" %
                          ((alg["lm_bytes"] + w.layers * alg["attn_bytes"]) / 1e9),
                       parallelism=f"replicas x{world}",
                       attention_launch=E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, int(w.ctx_len.max()),
                                                       inplace="chain" if st.chain else False)),
        "draft_tokens_per_s": round(steps_per_s * alg["draft_nodes"], 1),
        "roofline": roofline, "roofline_kernels": rl, "step_roofline": step_rl, "kernels": kernels,
        "e2e": e2e, "gpu_launches": st.launches_per_step() * args.steps, "clocks": clk,
        "verify_variants": variants,
        "row_kernels": rows,
        "planted_accept": [int(a) for a in w.planted_accept[:8]],
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        full, sample = oracle_repeat(w, 10.0)
        out["cpu_baseline"] = {"value": round(1.0 / full, 6), "unit": UNIT, "cores": cpu_cores(),
                               "kind": "oracle", "sample": sample,
                               "threads_note": "numpy fp64, default BLAS threading",
                               "single_thread": oracle_single_thread(args.config, w.layers, w.vocab)}
        if rows is not None:
            out["cpu_baseline"]["rows"] = oracle_rows_time()
    return out


def time_config(name, args, rank, dev, stream, steps):
    """The same step on another configuration (33b, batched), timed like the
    headline in the same process: plain CUDA graphs for ms_per_step, graphs with
    three external events for the attention and LM-head phases, its own clock
    record, and its roofline figures (per kernel: the bound of the larger of
    bytes / HBM peak and flops / tensor peak; per step: the literal HBM fraction
    on K/V and weight bytes and the fraction of the attainable floor)."""
    import paper_2506_02780_gb300 as E
    from paper_2506_02780_gb300 import step as S
    w = W.build(name, seed=rank_seed(name, rank), device=dev)
    alg = algorithmic(w)
    st = S.from_workload(w, device=dev, keep_layers=False)
    L = w.layers
    mk = lambda: torch.cuda.Event(enable_timing=True, external=True)  # noqa: E731
    plain, instr, evsets = [], [], []
    with torch.cuda.stream(stream):
        st.run(stream)
        stream.synchronize()
        for _ in range(2):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                run_instrumented(st, stream, None)
            plain.append(g)
            g = torch.cuda.CUDAGraph()
            evs = [mk() for _ in range(3)]
            with torch.cuda.graph(g, stream=stream):
                run_instrumented(st, stream, evs)
            instr.append(g)
            evsets.append(evs)
    stream.synchronize()
    assert E.ee_read_errors(st.ws, stream) == 0

    def timed(pool, n):
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            t0.record(stream)
            for i in range(n):
                pool[i % len(pool)].replay()
            t1.record(stream)
        t1.synchronize()
        return t0.elapsed_time(t1) / n

    for i in range(max(3, args.warmup // 4)):
        plain[i % 2].replay()
        instr[i % 2].replay()
    stream.synchronize()
    clocks = ClockSampler(dev.index)
    if not args.no_clocks:
        clocks.start()
    torch.cuda.synchronize(dev)
    clocks.mark_begin()
    ms = timed(plain, steps)
    torch.cuda.synchronize(dev)
    clocks.mark_end()
    clk = None if args.no_clocks else clocks.stop()
    acc = np.zeros(2)
    n = max(2, steps // 4)
    for i in range(n):
        instr[i % 2].replay()
        evs = evsets[i % 2]
        evs[-1].synchronize()
        acc += [evs[0].elapsed_time(evs[1]), evs[1].elapsed_time(evs[2])]
    acc /= n
    assert E.ee_read_errors(st.ws, stream) == 0
    peaks, peak_src = load_peaks()
    hbm = peaks["hbm_gbs"]
    tf = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
    attn_s, lm_s = 1e-3 * acc[0] / L, 1e-3 * acc[1]
    rl = {}
    for kname, t_s, nb, nf in (("tree_verify_attn", attn_s, alg["attn_bytes"], alg["attn_flops"]),
                               ("lmhead_accept", lm_s, alg["lm_bytes"], alg["lm_flops"])):
        gbs, tfs = nb / t_s / 1e9, nf / t_s / 1e12
        floor = max(nb / (hbm * 1e9), nf / (tf * 1e12))
        bound = "hbm" if nb / (hbm * 1e9) >= nf / (tf * 1e12) else "tensor"
        rl[kname] = {"bound": bound, "achieved": round(gbs if bound == "hbm" else tfs, 2),
                     "peak": hbm if bound == "hbm" else tf, "unit": "GB/s" if bound == "hbm" else "TFLOP/s",
                     "frac": round((gbs / hbm) if bound == "hbm" else (tfs / tf), 4),
                     "hbm_frac": round(gbs / hbm, 4), "frac_of_floor": round(floor / t_s, 4),
                     "us_per_launch": round(1e6 * t_s, 2), "traffic": TRAFFIC.get((kname, name))}
    kvw = L * 2 * int(w.ctx_len.sum()) * w.n_kv * w.head_dim * 2 + w.vocab * w.hidden * 2
    floor_s = (L * max(alg["attn_bytes"] / (hbm * 1e9), alg["attn_flops"] / (tf * 1e12))
               + max(alg["lm_bytes"] / (hbm * 1e9), alg["lm_flops"] / (tf * 1e12)))
    out = {"workload": name + ": " + _config_text(name), "ms_per_step": round(ms, 5),
           "value": round(1e3 / ms, 3), "unit": UNIT, "steps": steps,
           "draft_tokens_per_s": round(1e3 / ms * alg["draft_nodes"], 1),
           "kernels": {"attention_per_layer_us": round(1e6 * attn_s, 2), "lmhead_accept_us": round(1e6 * lm_s, 2)},
           "roofline": dict(rl["tree_verify_attn"], kernel="tree_verify_attn"), "roofline_kernels": rl,
           "step_roofline": {"kv_weight_bytes": kvw, "hbm_frac": round(kvw / (ms * 1e-3) / (hbm * 1e9), 4),
                             "floor_us": round(floor_s * 1e6, 1), "frac_of_floor": round(floor_s / (ms * 1e-3), 4),
                             "peaks": f"{peak_src}: HBM copy {hbm} GB/s, bf16 sustained {tf} TFLOP/s"},
           "attention_launch": E.ee_attn_plan(w.B, w.max_T, w.n_q, w.n_kv, int(w.ctx_len.max())),
           "clocks": clk, "config": W.describe(w)}
    why = clocks_rejected(clk)
    if why:
        out["clocks_rejected"] = why
    return out


def session_variant(w, dev, stream, K=16, replays=6):
    """A whole edit session at the workload's shapes on the device (EditSession):
    the workload's original code, an edited version of it (a replaced span, an
    insertion, a deletion) as the synthetic target's greedy text, a committed
    prefix of 200 tokens over a 4096-token context, trees of one reuse chain of
    24 per match point (2) plus a 4-token generated branch from a noisy draft
    model.  The device loop replays K captured steps at a time; the host loop
    replays one step and reads the committed length back every step."""
    import paper_2506_02780_gb300 as E
    from paper_2506_02780_gb300.session import EditSession
    rng = np.random.default_rng(11)
    c = np.asarray(w.orig_tokens[w.orig_off[0]:w.orig_off[1]], np.int32)
    cp = list(c)
    cp[700:705] = rng.integers(0, w.vocab, 5).tolist()
    cp[1500:1500] = rng.integers(0, w.vocab, 9).tolist()
    del cp[2300:2306]
    cp = np.asarray(cp, np.int32)
    P0, ctx0, G, n = 200, 4096, 4, w.n
    chain_len, nbr = 24, 2
    T = 1 + nbr * chain_len + G
    npg = -(-(ctx0 + len(cp) + 64 * T) // 16)
    L, n_kv = w.layers, w.n_kv
    g = torch.Generator(device=dev).manual_seed(11)
    kc = torch.empty((L, npg, n_kv, 16, 128), dtype=torch.bfloat16, device=dev).normal_(0, 0.088, generator=g)
    vc = torch.empty_like(kc).normal_(0, 0.088, generator=g)
    bt = torch.randperm(npg, generator=g, device=dev).int().reshape(1, npg)
    w_unit = (w.lm_w.float() / w.lm_w.float().norm(dim=1, keepdim=True)).bfloat16()
    cap = len(cp) + 64 * T * 4
    cp_pad = torch.zeros((1, cap + T + G), dtype=torch.int64, device=dev)
    cp_pad[0, :len(cp)] = torch.as_tensor(cp)

    def target_forward(ss):
        want = cp_pad[0, ss.out_len.long()[0] + ss.depth.long()]
        ss.hidden.copy_(w_unit[want] * 12.0)

    def draft_proposal(ss):
        k = ss.out_len.long()[:, None] + torch.arange(G, device=dev)[None, :]
        t = cp_pad.gather(1, k)
        ss.gen_tok.copy_(torch.where((k % 5) == 0, (t + 1) % w.vocab, t).int())

    def make():
        ss = EditSession(orig_tokens=torch.as_tensor(c, device=dev),
                         orig_off=torch.as_tensor([0, len(c)], dtype=torch.int64, device=dev),
                         committed=[cp[:P0].tolist()], ctx_len=[ctx0], k_cache=kc, v_cache=vc, block_table=bt,
                         lm_w=w.lm_w, n_q=w.n_q, n=n, chain_len=chain_len, n_branches=nbr, gen_len=G, cap=cap,
                         target_forward=target_forward, draft_proposal=draft_proposal, max_ctx=npg * 16 - T)
        ss.q.normal_(0, 1, generator=g)
        ss.k_tree.normal_(0, 0.088, generator=g)
        ss.v_tree.normal_(0, 0.088, generator=g)
        with torch.cuda.stream(stream):
            ss.step(stream)
        stream.synchronize()
        return ss

    dl = make()
    dl.capture(K, stream)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    len0 = int(dl.out_len[0])
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(replays):
            dl.replay()
        t1.record(stream)
    t1.synchronize()
    ms_dev = t0.elapsed_time(t1) / (K * replays)
    toks = int(dl.out_len[0]) - len0
    assert E.ee_read_errors(dl.ws, stream) == 0
    ok = bool(np.array_equal(dl.out_tok[0, :int(dl.out_len[0])].cpu().numpy(), cp[:int(dl.out_len[0])]))
    del dl
    hl = make()
    hl.capture(1, stream)
    steps = K * replays
    t_host = time.perf_counter()
    for _ in range(steps):
        hl.replay()
        int(hl.out_len[0])                 # the host reads the state back each step
    ms_host = (time.perf_counter() - t_host) * 1e3 / steps
    assert E.ee_read_errors(hl.ws, stream) == 0
    return {"device_loop_steps_per_s": round(1e3 / ms_dev, 2), "device_loop_ms_per_step": round(ms_dev, 5),
            "committed_tokens_per_s": round(toks / (ms_dev * K * replays) * 1e3, 1),
            "tokens_per_step": round(toks / (K * replays), 2), "steps_per_graph": K,
            "host_loop_steps_per_s": round(1e3 / ms_host, 2), "committed_text_ok": ok,
            "tree_nodes": T, "launches_per_step": hl.launches_per_step()}


def run_instrumented(st, stream, evs):
    """One step; with `evs` (three events) recorded before the first attention
    layer, after the last one and after the LM head (inside capture)."""
    st.run(stream, marks=(lambda k: evs[k].record(stream)) if evs else None)


def _clone_step(st):
    """A second VerifyStep with its own per-step input buffers, outputs and
    workspace, sharing the resident state (KV cache, block table, original code,
    LM-head weight) -- the second buffer set of the pipelined end-to-end loop."""
    from paper_2506_02780_gb300 import step as S
    x = st.inp
    c = {n: x[n].clone() for n in ("tail", "cursor", "parent", "node_off", "draft_tok", "ctx_len", "q",
                                    "k_tree", "v_tree", "hidden")}
    return S.VerifyStep(orig_tokens=x["orig_tokens"], orig_off=x["orig_off"], tail=c["tail"],
                        cursor=c["cursor"], parent=c["parent"], node_off=c["node_off"],
                        draft_tok=c["draft_tok"], ctx_len=c["ctx_len"], block_table=x["block_table"],
                        q=c["q"], k_tree=c["k_tree"], v_tree=c["v_tree"], k_cache=x["k_cache"],
                        v_cache=x["v_cache"], hidden=c["hidden"], lm_w=x["lm_w"], max_ctx=st.max_ctx,
                        max_T=st.max_T, max_matches=st.max_matches, keep_layers=False,
                        inplace_kv=st.inplace_kv, chain=st.chain, lm_packed=st.lm_packed)


def run_e2e(st, graph, stream, steps, dev, world):
    """Same metric through the public API with host buffers: every step copies its
    inputs (tail, cursor, tree, per-layer q / tree K/V, hidden states) from pinned
    host memory, replays the step and copies its results back to pinned host memory.

    e2e: two buffer sets, as a server interleaving independent batches does --
    step i+1's input copies run on a copy stream while step i computes, and the
    host reads step i's results (accept lengths) once they have arrived, one step
    later.  e2e_serial: one buffer set; copy, replay, read back, synchronise."""
    names_in = ["tail", "cursor", "parent", "node_off", "draft_tok", "ctx_len", "q", "k_tree", "v_tree",
                "hidden"]
    host_in = {n: st.inp[n].detach().cpu().pin_memory() for n in names_in}

    def outs_of(s):
        # accept_len, path, bonus, argmax, match_pos, n_matches, ctx_out: views of one buffer
        return [s.outputs]
    acc0 = st.out_layout["accept_len"][0]    # where accept_len[0] sits in it
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())

    # serial: one buffer set
    outs = outs_of(st)
    host_out = [torch.empty(o.shape, dtype=o.dtype).pin_memory() for o in outs]
    d2h = sum(t.numel() * t.element_size() for t in host_out)

    def one():
        with torch.cuda.stream(stream):
            for n in names_in:
                st.inp[n].copy_(host_in[n], non_blocking=True)
            graph.replay()
            for ho, o in zip(host_out, outs):
                ho.copy_(o, non_blocking=True)
        stream.synchronize()

    for _ in range(5):
        one()
    if world > 1:
        torch.distributed.barrier()
    t0 = time.perf_counter()
    for _ in range(steps):
        one()
    dt_serial = reduce_max(time.perf_counter() - t0, world, dev)

    # pipelined: two buffer sets, copies on their own stream
    st2 = _clone_step(st)
    with torch.cuda.stream(stream):
        st2.run(stream)
        stream.synchronize()
        graph2 = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph2, stream=stream):
            st2.run(stream)
    stream.synchronize()
    sets = [(st, graph, outs, host_out), (st2, graph2, outs_of(st2),
                                          [torch.empty(o.shape, dtype=o.dtype).pin_memory()
                                           for o in outs_of(st2)])]
    copy_stream = torch.cuda.Stream(device=dev)    # host -> device inputs
    back_stream = torch.cuda.Stream(device=dev)    # device -> host results
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    computed = [torch.cuda.Event(), torch.cuda.Event()]
    done = [torch.cuda.Event(), torch.cuda.Event()]
    seen = []

    def pipelined(n):
        for i in range(n):
            j = i % 2
            s_, g_, o_, ho_ = sets[j]
            with torch.cuda.stream(copy_stream):
                if i >= 2:
                    copy_stream.wait_event(done[j])       # set j's previous step: computed and read back
                for nm in names_in:
                    s_.inp[nm].copy_(host_in[nm], non_blocking=True)
                copied[j].record(copy_stream)
            with torch.cuda.stream(stream):
                stream.wait_event(copied[j])
                g_.replay()
                computed[j].record(stream)
            with torch.cuda.stream(back_stream):               # overlaps the next step's compute
                back_stream.wait_event(computed[j])
                for ho, o in zip(ho_, o_):
                    ho.copy_(o, non_blocking=True)
                done[j].record(back_stream)
            if i >= 1:                                     # the previous step's results, on the host
                k = (i - 1) % 2
                done[k].synchronize()
                seen.append(int(sets[k][3][0][acc0]))
        done[(n - 1) % 2].synchronize()
        seen.append(int(sets[(n - 1) % 2][3][0][acc0]))
        torch.cuda.synchronize(dev)

    pipelined(6)
    if world > 1:
        torch.distributed.barrier()
    seen.clear()
    t0 = time.perf_counter()
    pipelined(steps)
    dt = reduce_max(time.perf_counter() - t0, world, dev)
    assert len(seen) == steps and len(set(seen)) == 1   # every step's accept length came back
    return {"value": round(world * steps / dt, 2), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "ms_per_step": round(1e3 * dt / steps, 4),
            "pipelined": "2 buffer sets: step i+1's input copies and step i-1's result copy overlap step i's compute",
            "serial": {"value": round(world * steps / dt_serial, 2),
                       "ms_per_step": round(1e3 * dt_serial / steps, 4)}}


def _config_text(name):
    return {
        "7b": "Qwen2.5-Coder-7B shapes (H 3584, 28/4 heads, d 128, V 152064, 28 layers), 1 sequence, "
              "ctx 4096 in 16-token pages, 64-node tree (48-token reuse chain + two 8-token branches), "
              "original code 3000 tokens",
        "batched": "8 sequences, ctx U[1k,16k], trees of 32-96 nodes, 7B shapes, 28 layers",
        "33b": "DeepSeek-Coder-33B shapes (H 7168, 56/8 heads, V 32256, 62 layers), ctx 32768, 128-node tree",
        "tiny": "1 sequence, ctx 512, 16-node tree, 8/2 heads, H 512, V 4096, 1 layer",
        "long": "long reuse draft: Qwen2.5-Coder-7B shapes (H 3584, 28/4 heads, V 152064, 28 layers), "
                "1 sequence, ctx 4096, a 2048-token linear draft copied from an 8000-token original code, "
                "verified in place (causal attention over ctx + 2048, greedy longest-prefix acceptance)",
    }[name]


# ----------------------------------------------------------------------------
# reference arm: the fp64 oracle as it stands, bounded sample per step
# ----------------------------------------------------------------------------

def run_reference(args, rank, world, budget_s=240.0):
    """The oracle as it stands, on the host cores.  When ``steps`` whole oracle
    steps (``oracle.verify_step``: every layer, the whole vocabulary) fit in
    about ``budget_s`` seconds, every timed step is one whole step and value =
    1 / its mean time.  Otherwise (7b and larger, long drafts) each timed step is a
    bounded sample of the step, sized so that the timed steps take about
    ``budget_s`` in all: ``ms_per_step`` is then the sample's own measured time
    and ``value`` the full step extrapolated from it (``extrapolated``: true,
    with the scale factors).  Warm-up steps run a minimal sample (the oracle has
    nothing to compile or cache)."""
    import oracle as O
    if rank != 0:
        return None
    w = W.build(args.config, device="cpu")
    # calibration: a minimal sample, scaled to a full step
    full_est, _, _ = oracle_step_time(w, attn_nodes=1, lm_rows=min(w.vocab, 256))
    for _ in range(max(0, args.warmup)):
        oracle_step_time(w, attn_nodes=1, lm_rows=min(w.vocab, 256))
    k = max(1, args.steps)
    chain = w.max_T > 128
    # (the minimal sample's estimate can be low by an order of magnitude for a
    # whole step -- the full-vocabulary fp64 LM head is memory-bound -- hence
    # the margin of 10)
    whole = not chain and 10.0 * k * full_est <= budget_s
    walls, fulls, sample = [], [], ""
    if whole:
        for _ in range(k):
            t0 = time.perf_counter()
            O.verify_step(w)
            walls.append(time.perf_counter() - t0)
        t_step = ms_wall = float(np.mean(walls))
        sample = (f"{w.name}: whole oracle steps (match, tree, attention of every node of all {w.layers} "
                  f"layers, LM head + near-tie sets over all {w.vocab} rows, acceptance, compaction of "
                  f"all layers)")
    else:
        nodes, rows = oracle_sample_size(w, max(0.02, budget_s / k))
        for _ in range(k):
            t0 = time.perf_counter()
            full, spent, sample = oracle_step_time(w, attn_nodes=nodes, lm_rows=rows)
            walls.append(time.perf_counter() - t0)
            fulls.append(full)
        t_step, ms_wall = float(np.mean(fulls)), float(np.mean(walls))
    v = round(1.0 / t_step, 6)
    out = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * ms_wall, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded)", "config": dict(W.describe(w), workload=args.config + ": " +
                                                     _config_text(args.config)),
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                         "sample": sample + " (per timed step)"},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "extrapolated": not whole,
    }
    if not whole:
        out["scale"] = {"attention": round(w.layers * w.total_nodes / nodes, 3),
                        "lm_head": round(w.vocab / rows, 3), "compaction": w.layers}
        out["full_step_ms_estimate"] = round(1e3 * t_step, 3)
        out["note"] = ("each timed step is the sample described; ms_per_step is its measured time, value "
                       "the full step extrapolated from it by the scale factors")
    return out


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        out = run_reference(args, rank, world)
        if out is not None:
            print(json.dumps(out), flush=True)
        return
    if args.profile:
        sys.exit(run_profile(args, local_rank))
    if args.config == "sweep":
        sys.exit("the sweep has no verification step to time: its kernels are measured in every run's "
                 "row_kernels, and --profile --config sweep launches them for ncu")
    if world > 1:
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    out = run_ours(args, rank, world, local_rank)
    if args.config == "7b" and not args.no_configs and world == 1:
        # the larger configurations, each timed after the headline in this process
        import gc
        gc.collect()
        torch.cuda.empty_cache()
        dev = torch.device("cuda", local_rank)
        stream = torch.cuda.Stream(device=dev)
        cfgs = {}
        for name, n in (("33b", 40), ("batched", 100)):
            try:
                cfgs[name] = time_config(name, args, rank, dev, stream, n)
            except Exception as e:  # a failed side measurement never hides the headline
                cfgs[name] = {"error": f"{type(e).__name__}: {e}"[:300]}
            gc.collect()
            torch.cuda.empty_cache()
        out["configs"] = cfgs
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
