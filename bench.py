#!/usr/bin/env python
"""Benchmark of the ReSS hot path: one sparsified global-attention layer of a 3D ViT.

One step = ress_forward over one layer of synthetic inputs resident in HBM: block scoring
and the initial selection, R restoration rounds, the kept-block lists, and the
block-sparse attention.  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload vggt_v32] [--sweep] [--variants]

N > 1 runs as independent replicas (one per GPU, launched by torchrun): the method has no
exchange step, so there is no collective on the data path.  --impl reference times the
CPU oracle (float64 numpy) on a bounded sample of the same workload, extrapolated.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "ReSS layer ms & kept-FLOP TFLOP/s at 32 views/90% sparsity; select overhead %"


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="vggt_v32")
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true", help="64-view sparsity x rounds sweep lines")
    ap.add_argument("--q-block", type=int, default=64, choices=[64, 128],
                    help="query block size: 64 (the configs' grid) or 128 (the paper's grid)")
    ap.add_argument("--variants", action="store_true",
                    help="drift of the ablation variants (probability, random, maximised) lines")
    ap.add_argument("--cdf", type=float, default=0.9,
                    help="threshold tau of the CDF-threshold variant in --variants")
    ap.add_argument("--forward-only", action="store_true",
                    help="only the warm-up and the timed forwards (a short line; for profiling)")
    return ap.parse_args(argv)


def workload(a):
    import synth
    return synth.WORKLOADS[a.workload]


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p.get("bf16_tflops_sustained"), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# ----------------------------------------------------------------------------------------
# work accounting
# ----------------------------------------------------------------------------------------
def kept_flops(row_ptr, col_idx, N, H, nb, q_block=64):
    """4 * 64 * sum over rows of (valid query tokens) x (valid keys of the kept blocks); rows
    are query blocks of q_block tokens, columns 64-token key blocks."""
    tok = np.minimum(64, N - 64 * np.arange(nb)).astype(np.int64)
    nq = -(-N // q_block)
    qtok = np.minimum(q_block, N - q_block * np.arange(nq)).astype(np.int64)
    lens = np.diff(row_ptr.astype(np.int64))
    keys = np.add.reduceat(tok[col_idx[:row_ptr[-1]]], row_ptr[:-1].astype(np.int64)) if col_idx.size else 0
    keys = np.where(lens > 0, keys, 0)
    q = np.tile(qtok, H)
    return 4.0 * 64.0 * float((q * keys).sum())


def selection_bytes(N, H, nb, ld, rounds, csr_entries, nq=None):
    """Algorithmic bytes of scoring + restoration, a fixed formula whatever the kernels move:
    read Q, K, V once and write P and q (score); per round read P and q and read/write the
    drop masks (one bit per pair); write the CSR (col_idx and row_ptr).  Rows are the nq
    query blocks (nb by default), columns the nb key blocks."""
    nq = nb if nq is None else nq
    mat = H * nq * nb * 4
    score = 3 * N * H * 64 * 2 + 2 * mat
    per_round = 2 * mat + 2 * H * nq * nb // 8
    return score + rounds * per_round + 4 * csr_entries + 4 * (H * nq + 1)


# ----------------------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.uuid = uuid
        self.rows = []
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) == 9:
                self.rows.append(parts)

    def __exit__(self, *a):
        if self.proc:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=2)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = [r for r in self.rows if not self.uuid or self.uuid in r[0]] or self.rows
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        reasons = set()
        for r in rows:
            for name, v in zip(("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"), r[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": num(rows[0][2]), "reasons": sorted(reasons),
                "power_w_max": max((num(r[3]) or 0.0) for r in rows), "samples": len(rows)}


# ----------------------------------------------------------------------------------------
# CPU oracle timing (bounded sample, extrapolated)
# ----------------------------------------------------------------------------------------
_ORACLE = {}  # per worker process: the workload's inputs, built once by _oracle_init


def _oracle_init(name):
    """Worker start-up: rebuild the seeded inputs locally (no large arrays cross processes)."""
    import oracle as O
    import synth
    wl = synth.WORKLOADS[name]
    bits = synth.make_inputs(wl)
    X = [synth.bf16_to_f32(bits[k]) for k in ("Q", "K", "V")]
    _ORACLE.update(wl=wl, X=X, pooled=O.pool(*X, wl.n_special),
                   W=synth.bf16_to_f32(bits["W_o"]).astype(np.float64))


def _oracle_ready(_):
    time.sleep(0.05)
    return os.getpid()


def _oracle_rows(rows):
    import oracle as O
    wl = _ORACLE["wl"]
    t = time.perf_counter()
    O.ress_select(_ORACLE["pooled"], _ORACLE["W"], wl.budgets(), wl.rounds, wl.rho, rows=rows)
    return time.perf_counter() - t


def _oracle_attn(args):
    kept, rows = args
    import oracle as O
    t = time.perf_counter()
    O.block_sparse_attention(*_ORACLE["X"], kept, rows)
    return time.perf_counter() - t


def job_totals(dist, ms, units, device="cpu"):
    """Whole-job figures of N replicas: (the slowest rank's ms, the units all ranks processed).

    `dist` is torch.distributed with an initialised process group, or None for one process.
    The rate a line reports is units / ms of this pair, so every rank must call it."""
    if dist is None:
        return float(ms), float(units)
    import torch
    t_max = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    t_sum = torch.tensor([float(units)], dtype=torch.float64, device=device)
    dist.all_reduce(t_max, op=dist.ReduceOp.MAX)
    dist.all_reduce(t_sum, op=dist.ReduceOp.SUM)
    return float(t_max.item()), float(t_sum.item())


def attn_traffic():
    """DRAM bytes per k_attn launch from the committed ncu summary, while the kernel sources
    still hash to the value recorded there (None otherwise, or without a summary)."""
    import hashlib
    import re
    h = hashlib.sha256()
    for f in ("k_attn.cu", "sm100_ptx.cuh", "ress_internal.cuh"):
        with open(os.path.join(ROOT, "paper_2609_35593_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    try:
        with open(os.path.join(ROOT, "profiles", "k_attn_vggt_v32.md")) as fh:
            text = fh.read()
    except OSError:
        return None
    m_src = re.search(r"source sha256: ([0-9a-f]{64})", text)
    m_b = re.search(r"DRAM bytes per launch: (\d+)", text)
    if m_src and m_b and m_src.group(1) == h.hexdigest():
        return int(m_b.group(1))
    return None


def make_pool(workers, name):
    """`workers` spawned processes, each holding the workload built by _oracle_init."""
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    os.environ.setdefault("MKL_NUM_THREADS", "1")
    import multiprocessing as mp
    pool = mp.get_context("spawn").Pool(workers, initializer=_oracle_init, initargs=(name,))
    seen = set()
    while len(seen) < workers:  # every worker has finished its start-up
        seen.update(pool.map(_oracle_ready, range(2 * workers), chunksize=1))
    return pool


def oracle_layer_seconds(wl, X, kept, pool, workers, budget_s, rng):
    """Extrapolated seconds of the oracle for the whole layer, measured on a sample.

    Pooling is timed on a slice of about an eighth of the tokens and scaled by the token
    count (it is linear in N); selection and attention on row samples, sized to about half
    of `budget_s` each, spread over the worker processes and extrapolated by rows
    (selection) and kept FLOPs (attention)."""
    import oracle as O
    n_slice = max(64, (wl.n_tokens // 8) // 64 * 64)
    t0 = time.perf_counter()
    O.pool(*(x[:n_slice] for x in X), min(wl.n_special, n_slice))
    t_pool = (time.perf_counter() - t0) * wl.n_tokens / n_slice
    H, nb, nc = wl.heads, wl.n_blocks, wl.n_candidates
    sparse_rows = [(h, i) for h in range(H) for i in range(nc)]
    # calibrate one row, then size the sample to about half of the budget per stage
    t1 = pool.apply(_oracle_rows, ([sparse_rows[int(rng.integers(len(sparse_rows)))]],))
    n_sel = int(min(len(sparse_rows), max(workers, 0.5 * budget_s * workers / max(t1, 1e-4))))
    pick = rng.choice(len(sparse_rows), n_sel, replace=False)
    srows = [sparse_rows[k] for k in pick]
    t0 = time.perf_counter()
    pool.map(_oracle_rows, [srows[k::workers] for k in range(workers) if srows[k::workers]], chunksize=1)
    t_sel = (time.perf_counter() - t0) * len(sparse_rows) / n_sel
    # attention: sample rows (sparse and dense) and scale by kept FLOPs
    all_rows = [(h, i) for h in range(H) for i in range(nb)]
    tok = np.minimum(64, wl.n_tokens - 64 * np.arange(nb))
    def row_flops(r):
        return 4 * 64 * tok[r[1]] * tok[kept[r]].sum()
    total = sum(row_flops(r) for r in all_rows)
    r0 = all_rows[int(rng.integers(len(all_rows)))]
    t1 = pool.apply(_oracle_attn, (({r0: kept[r0]}, [r0]),))
    per_flop = t1 / max(row_flops(r0), 1)
    n_att = int(min(len(all_rows), max(workers, 0.5 * budget_s * workers / max(per_flop * total / len(all_rows), 1e-4))))
    pick = rng.choice(len(all_rows), n_att, replace=False)
    arows = [all_rows[k] for k in pick]
    f_sample = sum(row_flops(r) for r in arows)
    chunks = [arows[k::workers] for k in range(workers) if arows[k::workers]]
    t0 = time.perf_counter()
    pool.map(_oracle_attn, [({r: kept[r] for r in ch}, ch) for ch in chunks], chunksize=1)
    t_att = (time.perf_counter() - t0) * total / max(f_sample, 1)
    sample = (f"pooling of {n_slice} of {wl.n_tokens} tokens; ReSS selection on {n_sel} of "
              f"{len(sparse_rows)} candidate rows; token attention on {n_att} of {len(all_rows)} "
              f"rows; extrapolated linearly by tokens (pooling), rows (selection) and kept FLOPs "
              f"(attention); {workers} worker processes, 1 BLAS thread each")
    return t_pool + t_sel + t_att, dict(pool_s=t_pool, select_s=t_sel, attn_s=t_att), sample


def arm_config(wl, q_block, world):
    """The workload description both arms print (the driver compares the two lines)."""
    return {"workload": wl.name, "views": wl.views, "heads": wl.heads, "tokens": wl.n_tokens,
            "head_dim": 64, "block": 64, "q_block": q_block, "sparsity": wl.sparsity,
            "rounds": wl.rounds, "rho": wl.rho, "c_h": int(wl.budgets()[0]),
            "parallelism": f"replicas{world}", "l2": l2_note(wl)}


def l2_note(wl):
    """How the timed steps meet the L2 rule: inputs larger than the 129 MB L2, or not."""
    mb = 3 * wl.n_tokens * wl.heads * 64 * 2 / 1e6
    if mb > 129.0:
        return f"inputs larger than L2 ({mb:.0f} MB Q/K/V), no flush"
    return f"inputs smaller than L2 ({mb:.0f} MB Q/K/V), no flush"


# ----------------------------------------------------------------------------------------
# reference arm: the oracle as the timed implementation
# ----------------------------------------------------------------------------------------
def run_reference(a, wl):
    import synth
    import oracle as O
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    workers = os.cpu_count() or 1
    pool = make_pool(workers, wl.name)
    bits = synth.make_inputs(wl)
    X = [synth.bf16_to_f32(bits[k]) for k in ("Q", "K", "V")]
    # kept lists from the oracle's own selection on a row sample would differ per row; the
    # attention cost depends only on the list lengths, which the budget fixes
    nb, nc, H = wl.n_blocks, wl.n_candidates, wl.heads
    c = int(wl.budgets()[0])
    rng = np.random.default_rng(0)
    kept = {}
    for h in range(H):
        for i in range(nb):
            kept[(h, i)] = np.arange(nb) if i >= nc else np.sort(np.concatenate(
                [rng.choice(nc, c, replace=False), np.arange(nc, nb)]))
    N = wl.n_tokens
    tok = np.minimum(64, N - 64 * np.arange(nb))
    flops = sum(4 * 64 * tok[i] * tok[kept[(h, i)]].sum() for (h, i) in kept)
    # about 150 s of oracle work for the whole run, whatever K and W are
    per_step = max(0.2, min(8.0, 150.0 / max(a.steps + a.warmup, 1)))
    times = []
    for s in range(a.warmup + a.steps):
        t, parts, sample = oracle_layer_seconds(wl, X, kept, pool, workers, per_step,
                                                np.random.default_rng(s))
        if s >= a.warmup:
            times.append(t)
    del X
    t = float(np.mean(times))
    val = flops / t / 1e12
    line = {"metric": METRIC, "value": val, "unit": "TFLOP/s", "impl": "reference",
            "n_gpus": a.gpus, "steps": a.steps, "warmup": a.warmup, "ms_per_step": t * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            # the oracle's selection and attention follow 64-token query blocks
            "config": arm_config(wl, 64, int(os.environ.get("WORLD_SIZE", "1"))),
            "layer_ms": t * 1e3, "stage_s": parts,
            "cpu_baseline": {"value": val, "unit": "TFLOP/s", "cores": workers, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    pool.terminate()


# ----------------------------------------------------------------------------------------
# our arm
# ----------------------------------------------------------------------------------------
def run_ours(a, wl):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pool = None
    workers = os.cpu_count() or 1
    # the oracle's row sampling follows the 64-token grid; no CPU baseline on the 128 grid
    if rank == 0 and world == 1 and not a.no_cpu_baseline and not a.forward_only and a.q_block == 64:
        pool = make_pool(workers, wl.name)  # spawned processes, started before the first CUDA call
    import torch
    import synth
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    import paper_2609_35593_gb300 as ress

    bits = synth.make_inputs(wl)
    dev = lambda b: torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).cuda()
    Q, K, V, W = (dev(bits[k]) for k in ("Q", "K", "V", "W_o"))
    c_h = wl.budgets()
    N, H = wl.n_tokens, wl.heads
    d = ress.dims(N, H, wl.n_special, wl.d_model, a.q_block)
    buf = ress.Buffers(d, c_h)
    nb, nq, nqc = buf.nb, buf.nq, ress.num_query_candidates(d)
    ress.prepare_wo(d, W, buf.F)  # model-load time (Eq. 8), outside the step
    stream = torch.cuda.current_stream()

    def step():
        ress.forward(d, Q, K, V, buf.F, c_h, wl.rounds, wl.rho, buf.ws, buf.row_ptr, buf.col_idx,
                     buf.O, buf.J_best)

    for _ in range(max(a.warmup, 3)):
        step()
    ress.status(buf.ws)
    torch.cuda.synchronize()

    props = torch.cuda.get_device_properties(local)
    uuid = str(getattr(props, "uuid", "") or "")
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(uuid) as clk:
        n0 = ress.kernel_launches()
        ev0.record(stream)
        for _ in range(a.steps):
            step()
        ev1.record(stream)
        launches = ress.kernel_launches() - n0
        torch.cuda.synchronize()
    if dist:
        dist.barrier()
    ms = ev0.elapsed_time(ev1) / a.steps
    ress.status(buf.ws)
    if a.forward_only:
        if rank == 0:
            print(json.dumps({"forward_only": True, "workload": wl.name, "q_block": a.q_block,
                              "ms_per_step": ms, "steps": a.steps, "warmup": a.warmup,
                              "gpu_launches": launches}), flush=True)
        if dist:
            dist.destroy_process_group()
        return

    # ---- stage breakdown (same work, events between the three calls) ---------------
    nst = max(20, min(200, a.steps))
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(nst)]
    for k in range(nst):
        e = evs[k]
        e[0].record(stream)
        ress.score(d, Q, K, V, buf.F, c_h, buf.ws)
        e[1].record(stream)
        ress.restore(d, c_h, wl.rounds, wl.rho, buf.ws, buf.row_ptr, buf.col_idx, buf.J_best)
        e[2].record(stream)
        ress.sparse_attn(d, Q, K, V, buf.row_ptr, buf.col_idx, buf.O, buf.ws)
        e[3].record(stream)
    torch.cuda.synchronize()
    st = np.array([[e[i].elapsed_time(e[i + 1]) for i in range(3)] for e in evs])
    score_ms, restore_ms, attn_ms = (float(x) for x in np.median(st, axis=0))

    # ---- the rounds against the fp32 roofline: a round's time is restore(R) - restore(0)
    #      over R; its arithmetic is the gain products, 2 H |P|_rows |P| 64 fp32 flop -----
    csr_t = []
    for k in range(nst):
        ress.score(d, Q, K, V, buf.F, c_h, buf.ws)
        e = evs[k]
        e[0].record(stream)
        ress.restore(d, c_h, 0, wl.rho, buf.ws, buf.row_ptr, buf.col_idx, buf.J_best)
        e[1].record(stream)
    torch.cuda.synchronize()
    csr_ms = float(np.median([e[0].elapsed_time(e[1]) for e in evs]))
    ress.score(d, Q, K, V, buf.F, c_h, buf.ws)  # back to the R-round state read below
    ress.restore(d, c_h, wl.rounds, wl.rho, buf.ws, buf.row_ptr, buf.col_idx, buf.J_best)
    torch.cuda.synchronize()
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    round_flop = 2.0 * H * ress.num_query_candidates(d) * ress.num_candidates(d) * 64

    rp = buf.row_ptr.cpu().numpy()
    ci = buf.col_idx.cpu().numpy()
    flops = kept_flops(rp, ci, N, H, nb, a.q_block)
    hbm, bf16, bf16_sus, peak_kind = peaks()
    # the forward's attention stage: the layer less its score and restore stages (it holds
    # the pairing of the query blocks, the items' union lists and the attention kernel)
    attn_fwd_ms = max(ms - score_ms - restore_ms, 1e-9)
    # union efficiency of the forward's attention items (kept tiles per 64-row half tile of
    # the union walked), and of adjacent query-block pairs over the same kept lists
    ress.forward(d, Q, K, V, buf.F, c_h, wl.rounds, wl.rho, buf.ws, buf.row_ptr, buf.col_idx,
                 buf.O, buf.J_best)
    torch.cuda.synchronize()
    rpi = 1 if a.q_block == 128 else 2
    n_items = -(-nq // rpi)
    plen = buf.ws_view("plen", torch.int32).cpu().numpy()[:H * n_items].astype(np.int64)
    row_len = np.diff(rp.astype(np.int64))
    kept_half_tiles = int(row_len.sum()) * (2 // rpi)
    adj = 0
    for h in range(H):
        for u in range(n_items):
            rows = [h * nq + rpi * u + k for k in range(rpi) if rpi * u + k < nq]
            adj += len(set().union(*[set(ci[rp[r]:rp[r + 1]].tolist()) for r in rows]))
    items = {"union_efficiency": kept_half_tiles / 2.0 / float(plen.sum()),
             "adjacent_union_efficiency": kept_half_tiles / 2.0 / float(adj),
             "union_entries": int(plen.sum())}

    # ---- dense run of the same attention kernel (no block dropped) -------------------
    dense = None
    if wl.name == "vggt_v32" and a.q_block == 64:
        rpd = torch.arange(0, H * nb * nb + 1, nb, dtype=torch.int32, device="cuda")
        cid = torch.arange(nb, dtype=torch.int32, device="cuda").repeat(H * nb)
        Od = torch.empty_like(buf.O)
        for _ in range(3):
            ress.sparse_attn(d, Q, K, V, rpd, cid, Od, buf.ws)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        nd = 10
        e0.record(stream)
        for _ in range(nd):
            ress.sparse_attn(d, Q, K, V, rpd, cid, Od, buf.ws)
        e1.record(stream)
        torch.cuda.synchronize()
        dms = e0.elapsed_time(e1) / nd
        dfl = kept_flops(rpd.cpu().numpy(), cid.cpu().numpy(), N, H, nb)
        dense = {"attn_ms": dms, "tflops": dfl / dms / 1e9, "frac_of_bf16_peak": dfl / dms / 1e9 / bf16,
                 "speedup_of_sparse_layer": dms / ms}
        # token-level drift of the sparse output against the dense one (Sec. 3's reference)
        drift = torch.empty(nb, dtype=torch.float32, device="cuda")
        ress.token_drift(d, buf.O, Od, W, drift, buf.ws)
        e0.record(stream)
        for _ in range(nd):
            ress.token_drift(d, buf.O, Od, W, drift, buf.ws)
        e1.record(stream)
        torch.cuda.synchronize()
        tms = e0.elapsed_time(e1) / nd
        tdr = drift.cpu().numpy().astype(np.float64)
        ncb = ress.num_candidates(d)
        dense["token_drift"] = {"sum_candidate_blocks": float(tdr[:ncb].sum()),
                                "sum_all_blocks": float(tdr.sum()), "ms": tms,
                                "tflops": 2 * 2.0 * N * d.d_model * H * 64 / tms / 1e9}
        ress.status(buf.ws)
        del Od, rpd, cid

    # ---- the paper's own grid: 128-token query blocks over 64-token key blocks ------
    paper_grid = None
    if wl.name == "vggt_v32" and a.q_block == 64:
        d2 = ress.dims(N, H, wl.n_special, wl.d_model, 128)
        buf2 = ress.Buffers(d2, c_h)
        ress.prepare_wo(d2, W, buf2.F)

        def step2():
            ress.forward(d2, Q, K, V, buf2.F, c_h, wl.rounds, wl.rho, buf2.ws, buf2.row_ptr,
                         buf2.col_idx, buf2.O, buf2.J_best)
        for _ in range(3):
            step2()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n2 = max(20, min(100, a.steps))
        e0.record(stream)
        for _ in range(n2):
            step2()
        e1.record(stream)
        torch.cuda.synchronize()
        lms2 = e0.elapsed_time(e1) / n2
        ev2 = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n2)]
        for e in ev2:
            e[0].record(stream)
            ress.score(d2, Q, K, V, buf2.F, c_h, buf2.ws)
            e[1].record(stream)
            ress.restore(d2, c_h, wl.rounds, wl.rho, buf2.ws, buf2.row_ptr, buf2.col_idx, buf2.J_best)
            e[2].record(stream)
            ress.sparse_attn(d2, Q, K, V, buf2.row_ptr, buf2.col_idx, buf2.O, buf2.ws)
            e[3].record(stream)
        torch.cuda.synchronize()
        st2 = np.median(np.array([[e[i].elapsed_time(e[i + 1]) for i in range(3)] for e in ev2]), axis=0)
        ress.status(buf2.ws)
        fl2 = kept_flops(buf2.row_ptr.cpu().numpy(), buf2.col_idx.cpu().numpy(), N, H, nb, 128)
        nq2 = ress.num_query_blocks(d2)
        Jb2 = buf2.J_best.cpu().numpy().reshape(H, nq2)[:, :ress.num_query_candidates(d2)]
        paper_grid = {"q_block": 128, "k_block": 64, "layer_ms": lms2,
                      "value": fl2 / lms2 / 1e9, "unit": "TFLOP/s", "kept_tflop": fl2 / 1e12,
                      "stage_ms": {"score": float(st2[0]), "restore": float(st2[1]),
                                   "attn": float(st2[2])},
                      "select_overhead_pct": 100.0 * float(st2[0] + st2[1]) / lms2,
                      "attn_tflops": fl2 / float(st2[2]) / 1e9,
                      "attn_frac_of_bf16_peak": fl2 / float(st2[2]) / 1e9 / bf16,
                      "sum_J_best": float(Jb2.astype(np.float64).sum())}
        del buf2

    # ---- the sublayer's residual update y = x + O W_o^T (tensor-core GEMM) ----------
    xres = torch.randn(N, d.d_model, dtype=torch.bfloat16, device="cuda",
                       generator=torch.Generator(device="cuda").manual_seed(0))
    yres = torch.empty_like(xres)
    for _ in range(3):
        ress.out_proj(d, buf.O, W, xres, yres, buf.ws)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    no = 20
    e0.record(stream)
    for _ in range(no):
        ress.out_proj(d, buf.O, W, xres, yres, buf.ws)
    e1.record(stream)
    torch.cuda.synchronize()
    oms = e0.elapsed_time(e1) / no
    ofl = 2.0 * N * d.d_model * H * 64
    obytes = 2.0 * (N * H * 64 + d.d_model * H * 64 + 2 * N * d.d_model)
    out_proj = {"ms": oms, "tflops": ofl / oms / 1e9, "frac_of_bf16_peak": ofl / oms / 1e9 / bf16,
                "gbs": obytes / oms / 1e6, "flop": ofl, "bytes": obytes}
    ress.status(buf.ws)
    del xres, yres

    # ---- end to end through the public API with host buffers -------------------------
    # ress_forward_host per step: the copies of the step's Q, K, V in, the forward, the copy
    # of O out, all on one stream.  Steps alternate between two streams, each with its own
    # device buffers, workspace and CSR arrays, so one step's copies overlap the other's
    # compute (the inputs of every step come from pinned host memory, every O goes back).
    hQ, hK, hV = (t.cpu().pin_memory() for t in (Q, K, V))
    sets = []
    for k in range(2):
        bk = buf if k == 0 else ress.Buffers(d, c_h)
        if k:
            bk.F.copy_(buf.F)
        sets.append({"buf": bk, "stream": torch.cuda.Stream(),
                     "dev": [torch.empty_like(t) for t in (Q, K, V, buf.O)],
                     "hO": torch.empty(buf.O.shape, dtype=torch.bfloat16).pin_memory()})
    torch.cuda.synchronize()

    def e2e_step(k):
        st = sets[k % 2]
        bk, (dQ, dK, dV, dO) = st["buf"], st["dev"]
        ress.forward_host(d, hQ, hK, hV, st["hO"], dQ, dK, dV, dO, bk.F, c_h, wl.rounds, wl.rho,
                          bk.ws, bk.row_ptr, bk.col_idx, bk.J_best, stream=st["stream"])

    ne = max(10, min(50, a.steps))
    for k in range(4):
        e2e_step(k)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for st in sets:
        st["stream"].wait_event(e0)
    for k in range(ne):
        e2e_step(k)
    for st in sets:
        done = torch.cuda.Event()
        done.record(st["stream"])
        stream.wait_event(done)
    e1 = torch.cuda.Event(enable_timing=True)
    e1.record(stream)
    torch.cuda.synchronize()
    ems = e0.elapsed_time(e1) / ne
    for st in sets:
        ress.status(st["buf"].ws)
    assert torch.equal(sets[0]["hO"].view(torch.int16), buf.O.cpu().view(torch.int16))
    del sets
    h2d = 3 * N * H * 64 * 2
    d2h = N * H * 64 * 2

    # ---- realised drift and sparsity ---------------------------------------------------
    Jb = buf.J_best.cpu().numpy().astype(np.float64)
    J0 = buf.ws_view("J0", torch.float32).cpu().numpy()[:H * nq].astype(np.float64)
    cand_rows = np.tile(np.arange(nq) < nqc, H)
    kept_pairs = int(np.diff(rp.astype(np.int64)).sum())

    sel_bytes = selection_bytes(N, H, nb, buf.layout.ld, wl.rounds, ci.size, nq)
    sel_ms = score_ms + restore_ms
    dev = "cuda" if dist and dist.get_backend() == "nccl" else "cpu"
    ms_job, flops_job = job_totals(dist, ms, flops, dev)      # device-timed step
    ems_job, eflops_job = job_totals(dist, ems, flops, dev)   # end to end, host buffers
    line = {
        "metric": METRIC, "value": flops_job / ms_job / 1e9, "unit": "TFLOP/s", "n_gpus": world,
        "steps": a.steps, "warmup": a.warmup, "ms_per_step": ms_job, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded VGGT-shaped Q/K/V and W_o)",
        "config": arm_config(wl, a.q_block, world),
        "layer_ms": ms_job,
        # attn: ress_sparse_attn on the same CSR (adjacent query blocks share a tile);
        # attn_forward: the forward's own attention stage (paired query blocks)
        "stage_ms": {"score": score_ms, "restore": restore_ms, "attn": attn_ms,
                     "attn_forward": attn_fwd_ms},
        "select_overhead_pct": 100.0 * sel_ms / ms,
        "attn_tflops": flops / attn_fwd_ms / 1e9,
        "attn_items": items,
        "selection": {"algorithmic_bytes": sel_bytes, "gbs": sel_bytes / sel_ms / 1e6,
                      "frac_of_hbm": sel_bytes / sel_ms / 1e6 / hbm, "hbm_peak_gbs": hbm,
                      "frac_of_nominal_8tbs": sel_bytes / sel_ms / 1e6 / 8000.0},
        "kept_tflop": flops / 1e12, "realized_pair_sparsity": 1.0 - kept_pairs / (H * nq * nb),
        "drift": {"sum_J_best": float(Jb[cand_rows].sum()), "sum_J0": float(J0[cand_rows].sum())},
        "dense": dense,
        "paper_grid": paper_grid,
        "out_proj": out_proj,
        "roofline": {"bound": "tensor", "kernel": "k_attn (ress_forward's attention stage)",
                     "achieved": flops / attn_fwd_ms / 1e9, "peak": bf16, "unit": "TFLOP/s",
                     "frac": flops / attn_fwd_ms / 1e9 / bf16,
                     "traffic": attn_traffic() if wl.name == "vggt_v32" and a.q_block == 64 else None,
                     "peak_kind": f"{peak_kind} bf16 burst"},
        # kernels the library enqueued inside the timed region (its own launch counter)
        "gpu_launches": launches,
        "e2e": {"value": eflops_job / ems_job / 1e9, "unit": "TFLOP/s", "ms_per_step": ems_job,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "clocks": clk.summary(),
    }
    if wl.rounds > 0:
        # fp32 SIMT peak: 128 FMA lanes per SM at the SM clock seen under load (2070 MHz max)
        mhz = line["clocks"].get("sm_max_mhz") or 2070.0
        fp32_peak = props.multi_processor_count * 128 * 2 * mhz * 1e6 / 1e12
        round_ms = max(restore_ms - csr_ms, 1e-9) / wl.rounds
        line["rounds"] = {
            "ms_per_round": round_ms, "csr_ms": csr_ms,
            "fp32_gain_flop_per_round": round_flop,
            "gain_tflops_over_round": round_flop / round_ms / 1e9,
            "fp32_simt_peak_tflops": fp32_peak,
            "frac_of_fp32_simt": round_flop / round_ms / 1e9 / fp32_peak,
            "note": "a round = the gain products (tensor cores, three-term bf16) plus the per-row "
                    "selection and update; its time bounds the gain arithmetic rate from below"}

    if pool is not None:
        kept = {(h, i): ci[rp[h * nb + i]:rp[h * nb + i + 1]] for h in range(H) for i in range(nb)}
        X = [synth.bf16_to_f32(bits[k]) for k in ("Q", "K", "V")]
        t, parts, sample = oracle_layer_seconds(wl, X, kept, pool, workers, a.cpu_budget,
                                                np.random.default_rng(0))
        line["cpu_baseline"] = {"value": flops / t / 1e12, "unit": "TFLOP/s", "cores": workers,
                                "kind": "oracle", "sample": sample, "layer_s": t, "stage_s": parts}
        pool.terminate()
    if rank == 0:
        print(json.dumps(line), flush=True)

    if a.sweep and rank == 0:
        sweep(a)
    if a.variants and rank == 0:
        variants(a, wl)
    if dist:
        dist.destroy_process_group()


def sweep(a):
    """64 views: sparsity x rounds, realised drift, selection and attention time per point."""
    import torch
    import synth
    import paper_2609_35593_gb300 as ress
    base = synth.WORKLOADS["vggt_v64"]
    bits = synth.make_inputs(base)
    dev = lambda b: torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).cuda()
    Q, K, V, W = (dev(bits[k]) for k in ("Q", "K", "V", "W_o"))
    for s, R in synth.SWEEP_V64:
        wl = base.with_(sparsity=s, rounds=R)
        c_h = wl.budgets()
        d = ress.dims(wl.n_tokens, wl.heads, wl.n_special, wl.d_model)
        buf = ress.Buffers(d, c_h)
        ress.prepare_wo(d, W, buf.F)
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        res = []
        for k in range(6):
            evs[0].record()
            ress.score(d, Q, K, V, buf.F, c_h, buf.ws)
            evs[1].record()
            ress.restore(d, c_h, R, wl.rho, buf.ws, buf.row_ptr, buf.col_idx, buf.J_best)
            evs[2].record()
            ress.sparse_attn(d, Q, K, V, buf.row_ptr, buf.col_idx, buf.O, buf.ws)
            evs[3].record()
            torch.cuda.synchronize()
            if k >= 2:
                res.append([evs[i].elapsed_time(evs[i + 1]) for i in range(3)])
        ress.status(buf.ws)
        m = np.median(np.array(res), axis=0)
        nb = buf.nb
        Jb = buf.J_best.cpu().numpy().reshape(wl.heads, nb)[:, :wl.n_candidates]
        print(json.dumps({"sweep": "vggt_v64", "sparsity": s, "rounds": R, "c_h": int(c_h[0]),
                          "sum_J_best": float(Jb.astype(np.float64).sum()),
                          "select_ms": float(m[0] + m[1]), "attn_ms": float(m[2])}), flush=True)
        del buf


def variants(a, wl):
    """The drift side of Fig. 8 on the synthetic layer: for ReSS and each ablation variant,
    the pooled objective sum_J(D_best) over candidate rows and the token-level drift of its
    sparse output against the dense output (ress_token_drift), at the workload's budget."""
    import torch
    import synth
    import paper_2609_35593_gb300 as ress
    bits = synth.make_inputs(wl)
    dev = lambda b: torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).cuda()
    Q, K, V, W = (dev(bits[k]) for k in ("Q", "K", "V", "W_o"))
    c_h = wl.budgets()
    d = ress.dims(wl.n_tokens, wl.heads, wl.n_special, wl.d_model)
    buf = ress.Buffers(d, c_h, variant=ress.variant(cdf=1.0))  # room for whole rows
    ress.prepare_wo(d, W, buf.F)
    H, nb, nc = wl.heads, buf.nb, wl.n_candidates
    rpd = torch.arange(0, H * nb * nb + 1, nb, dtype=torch.int32, device="cuda")
    cid = torch.arange(nb, dtype=torch.int32, device="cuda").repeat(H * nb)
    Od = torch.empty_like(buf.O)
    ress.sparse_attn(d, Q, K, V, rpd, cid, Od, buf.ws)
    drift = torch.empty(nb, dtype=torch.float32, device="cuda")
    cases = [("ress", "drift", "none", wl.rounds, 0.0),
             ("probability", "probability", "none", 0, 0.0),
             ("probability_cdf", "probability", "none", 0, a.cdf),  # top-k plus the CDF rule
             ("random", "random", "none", 0, 0.0), ("maximize_swap", "drift", "swap", wl.rounds, 0.0),
             ("maximize_full", "drift", "full", wl.rounds, 0.0)]
    for name, key, mx, R, cdf in cases:
        v = ress.variant(key, mx, seed=1, cdf=cdf)
        ress.score(d, Q, K, V, buf.F, c_h, buf.ws, variant=v)
        ress.restore(d, c_h, R, wl.rho, buf.ws, buf.row_ptr, buf.col_idx, buf.J_best, variant=v)
        ress.sparse_attn(d, Q, K, V, buf.row_ptr, buf.col_idx, buf.O, buf.ws)
        ress.token_drift(d, buf.O, Od, W, drift, buf.ws)
        ress.status(buf.ws)
        Jb = buf.J_best.cpu().numpy().reshape(H, nb)[:, :nc].astype(np.float64)
        kept = int(buf.row_ptr[-1].item())  # CSR entries: every query row's kept key blocks
        print(json.dumps({"variants": wl.name, "variant": name, "key": key, "maximize": mx,
                          "rounds": R, "cdf": cdf, "c_h": int(c_h[0]),
                          "kept_block_fraction": kept / float(H * nb * nb),
                          "sum_J_best": float(Jb.sum()),
                          "token_drift": float(drift.cpu().numpy().astype(np.float64).sum())}),
              flush=True)


def main():
    a = parse()
    wl = workload(a)
    if a.impl == "reference":
        run_reference(a, wl)
    else:
        run_ours(a, wl)


if __name__ == "__main__":
    main()
