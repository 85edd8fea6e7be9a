"""RoleSub hot-path benchmark: compress + attend on synthetic OpenVLA-OFT-7B
shaped inputs, timed on the GPU with CUDA events.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c1|c2|c3|c4]
                  [--impl ours|reference]

One step = rolesub_compress + rolesub_attend over every layer and episode of
the workload (all steps of the path). Prints ONE JSON line on rank 0.

Metric: action-query tokens per second per layer for compress + attend,
value = (query tokens x layers x ranks) / max-over-ranks time. Per-step
inputs are larger than L2 for c2-c4; for c1 the L2 is flushed (a 512 MB
write) between timed steps, outside the timed region.

--impl reference times the fp64 CPU oracle (the plain restatement of the
paper's method) on the host cores, on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "action-query attend+compress tokens/s per layer; HBM GB/s fraction of peak"
UNIT = "query tokens/s/layer"
FLUSH_BYTES = 512 << 20
E2E_CHUNK = 4   # layers per chunk of the end-to-end pipeline


# ---------------------------------------------------------------------------
# workload and accounting
# ---------------------------------------------------------------------------

def make_workload(name, rank=0, layers=None):
    from paper_2608_18410_gb300 import synth
    import dataclasses
    if name == "c2":
        wl = synth.c2(128, 4)
    else:
        wl = synth.WORKLOADS[name]()
    if layers:
        # fewer layers of the same workload: only for small profiling runs,
        # never a bench line (the headline always runs the full stack)
        wl = wl.with_layers(layers)
    if rank:
        wl = dataclasses.replace(wl, seed=wl.seed + 1000 * rank)
    return wl


def attend_bytes(wl):
    """Algorithmic bytes of one rolesub_attend over the workload.

    Per (layer, episode): q and o (Nq*d each), full keys (Nc*d), packed kept
    groups (sum_j k_j*H*d_s), their indices (sum_j k_j bytes); R_h once per
    layer (H*d_h^2). Elements are b bytes (2 for bf16, 4 for fp32).
    """
    b = 2 if wl.dtype == "bf16" else 4
    d, H, ds = wl.d, wl.H, wl.dh // wl.G
    per_layer = H * wl.dh * wl.dh * b
    for ep in wl.episodes:
        ks = sum(n * k for n, k in zip(ep.n_tok(), ep.k(wl.G)))
        per_layer += 2 * ep.n_query * d * b + ep.n_cache * d * b + ks * H * ds * b + ks
    return per_layer * wl.L


def compress_bytes(wl):
    """Algorithmic bytes of one rolesub_compress over the workload.

    Per layer: h of routed and language rows, v of stored rows, R, all
    router weights (W_re, W1, W2, fp32 biases), packed values and indices
    written.
    """
    b = 2 if wl.dtype == "bf16" else 4
    d, H, ds, G = wl.d, wl.H, wl.dh // wl.G, wl.G
    per_layer = H * wl.dh * wl.dh * b + (wl.C * d + wl.F * (2 * d + wl.C) + G * wl.F) * b
    per_layer += 4 * (wl.C + wl.F + G)
    for ep in wl.episodes:
        for kind, (n, k) in enumerate(zip(ep.n_tok(), ep.k(G))):
            routed = 0 < k < G
            if routed or kind == 1:
                per_layer += n * d * b
            if k > 0:
                per_layer += n * d * b + n * k * H * ds * b + n * k
    return per_layer * wl.L


def compress_additive_bytes(wl, C):
    """Algorithmic bytes of one rolesub_compress_additive over the workload.

    As compress_bytes, with the additive router's weights (W_re [C][d],
    W_v and W_l [S][d], W_role [S][C], fp32 biases) instead of the
    concatenation router's.
    """
    b = 2 if wl.dtype == "bf16" else 4
    d, H, ds, G = wl.d, wl.H, wl.dh // wl.G, wl.G
    per_layer = H * wl.dh * wl.dh * b + (C * d + 2 * G * d + G * C) * b + 4 * (C + 2 * G)
    for ep in wl.episodes:
        for kind, (n, k) in enumerate(zip(ep.n_tok(), ep.k(G))):
            if 0 < k < G or kind == 1:
                per_layer += n * d * b
            if k > 0:
                per_layer += n * d * b + n * k * H * ds * b + n * k
    return per_layer * wl.L


def attend_flops(wl):
    d, H, ds = wl.d, wl.H, wl.dh // wl.G
    f = 0
    for ep in wl.episodes:
        ks = sum(n * k for n, k in zip(ep.n_tok(), ep.k(wl.G)))
        f += 2 * ep.n_query * ep.n_cache * d + 2 * ep.n_query * H * ks * ds + 2 * ep.n_query * H * wl.dh ** 2
    return f * wl.L


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"],
                "bf16_tflops_sustained": j.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def load_traffic(kernel, workload):
    """DRAM bytes per launch from a committed ncu summary, if it is current.

    profiles/traffic.txt lines: kernel workload source_sha256[:16] dram_bytes,
    the hash taken over csrc/<kernel>.cuh when it exists, else <kernel>.cu
    """
    import hashlib
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    # the file that holds the kernel's code (the attention kernel is a header
    # shared by its fixed-k and budget translation units)
    csrc = os.path.join(ROOT, "paper_2608_18410_gb300", "csrc")
    src = os.path.join(csrc, kernel + ".cuh")
    if not os.path.exists(src):
        src = os.path.join(csrc, kernel + ".cu")
    if not os.path.exists(src):
        return None
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    for line in open(path):
        parts = line.split("#")[0].split()
        if len(parts) == 4 and parts[0] == kernel and parts[1] == workload and parts[2] == sha:
            return float(parts[3])
    return None


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1].split()[0]))
                mx.append(float(f[2].split()[0]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# distributed helpers (one process per GPU; timing reduce only)
# ---------------------------------------------------------------------------

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x, ws):
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling(total_ms_local, steps, query_tokens_per_step, ws):
    """Whole-job throughput over ranks that each process their own batch:
    the slowest rank's time bounds the job; every rank's tokens count."""
    total_ms = max_over_ranks(total_ms_local, ws)
    ms_per_step = total_ms / steps
    return ms_per_step, query_tokens_per_step * ws / (ms_per_step / 1e3)


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------------------
# CPU baseline: the oracle on a bounded sample
# ---------------------------------------------------------------------------

def oracle_sample(wl, inp, budget_s=12.0, max_items=None):
    """Times the fp64 oracle (compress + attend) on (layer, episode) items of
    the workload until about budget_s seconds; returns the measurement."""
    import oracle
    from paper_2608_18410_gb300 import synth
    G, H, dh = wl.G, wl.H, wl.dh
    order = [(l, e) for l in range(wl.L) for e in range(wl.E)]
    rng = np.random.default_rng(12345)
    rng.shuffle(order)
    glob_rows = np.concatenate([[0], np.cumsum([ep.n_cache for ep in wl.episodes])])
    glob_q = np.concatenate([[0], np.cumsum([ep.n_query for ep in wl.episodes])])
    items, qtok, t_total = 0, 0, 0.0
    for (l, e) in order:
        ep = wl.episodes[e]
        spec = oracle.Spec(H, dh, G, wl.C, wl.F, np.array(ep.n_tok())[None], np.array(ep.k(G))[None],
                           [ep.n_query])
        r0, r1 = int(glob_rows[e]), int(glob_rows[e + 1])
        q0, q1 = int(glob_q[e]), int(glob_q[e + 1])
        W = lambda n: synth.widen(inp[n][l], wl.dtype)
        h = synth.widen(inp["h"][l, r0:r1], wl.dtype)
        v = synth.widen(inp["v"][l, r0:r1], wl.dtype)
        q = synth.widen(inp["q"][l, q0:q1], wl.dtype)
        K = synth.widen(inp["K"][l, r0:r1], wl.dtype)
        R = W("R")
        args = (R, W("W_re"), inp["b_re"][l].astype(np.float64), W("W1"), inp["b1"][l].astype(np.float64),
                W("W2"), inp["b2"][l].astype(np.float64), wl.alpha_role, wl.alpha_lang)
        t0 = time.perf_counter()
        c = oracle.compress_layer(spec, h, v, *args, want_z=False)
        oracle.attend_layer(spec, q, K, c["packed"], c["idx"], R)
        t_total += time.perf_counter() - t0
        items += 1
        qtok += ep.n_query
        if t_total >= budget_s or (max_items and items >= max_items):
            break
    return {"value": qtok / t_total, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{items} (layer, episode) item(s) of {wl.name} ({qtok} query tokens x 1 layer each), "
                      f"fp64 compress+attend, {t_total:.1f} s, 1 thread"}


def _oracle_worker(job):
    """One host process of the all-cores oracle timing: regenerates its
    (layer, episode) items from the seeded recipe and times the fp64 oracle
    on them until its budget is spent. Returns (items, query tokens, s)."""
    name, layers, wid, order, budget_s = job
    import oracle
    from paper_2608_18410_gb300 import synth
    wl = make_workload(name, 0, layers)
    G, H, dh = wl.G, wl.H, wl.dh
    wcache = {}
    items, qtok, t_total = 0, 0, 0.0
    for (l, e) in order:
        ep = wl.episodes[e]
        if l not in wcache:
            wcache.clear()
            wcache[l] = synth.gen_layer_weights(wl, l)
        w = wcache[l]
        a = synth.gen_episode_acts(wl, l, e)
        spec = oracle.Spec(H, dh, G, wl.C, wl.F, np.array(ep.n_tok())[None], np.array(ep.k(G))[None],
                           [ep.n_query])
        W = lambda n: synth.widen(w[n], wl.dtype)
        X = lambda n: synth.widen(a[n], wl.dtype)
        R = W("R")
        args = (R, W("W_re"), w["b_re"].astype(np.float64), W("W1"), w["b1"].astype(np.float64),
                W("W2"), w["b2"].astype(np.float64), wl.alpha_role, wl.alpha_lang)
        h, v, q, K = X("h"), X("v"), X("q"), X("K")
        t0 = time.perf_counter()
        c = oracle.compress_layer(spec, h, v, *args, want_z=False)
        oracle.attend_layer(spec, q, K, c["packed"], c["idx"], R)
        t_total += time.perf_counter() - t0
        items += 1
        qtok += ep.n_query
        if t_total >= budget_s:
            break
    return items, qtok, t_total


def oracle_sample_all_cores(wl, key, layers, budget_s=10.0, pool=None, cores=None, seed=12345):
    """The fp64 oracle, as it stands, in one spawned process per host core,
    each timing its own share of shuffled (layer, episode) items for about
    budget_s seconds at the same time; throughput = query tokens of all
    processes / the longest process's oracle time."""
    import multiprocessing as mp
    cores = cores or os.cpu_count() or 1
    order = [(l, e) for l in range(wl.L) for e in range(wl.E)]
    rng = np.random.default_rng(seed)
    rng.shuffle(order)
    # each process's random share, grouped by layer so that it draws each
    # layer's weights once
    jobs = [(key, layers, w, sorted((tuple(map(int, x)) for x in order[w::cores]), key=lambda t: t[0]), budget_s)
            for w in range(cores)]
    if pool is None:
        with mp.get_context("spawn").Pool(cores) as p:
            res = p.map(_oracle_worker, jobs)
    else:
        res = pool.map(_oracle_worker, jobs)
    items = sum(r[0] for r in res)
    qtok = sum(r[1] for r in res)
    wall = max(r[2] for r in res)
    return {"value": qtok / wall, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{items} (layer, episode) item(s) of {wl.name} ({qtok} query tokens x 1 layer each), "
                      f"fp64 compress+attend, {cores} processes for {wall:.1f} s each"}


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    import multiprocessing as mp
    wl = make_workload(args.workload, 0, args.layers)
    # about a minute of oracle work over the steps (plus input generation)
    per_step_budget = max(0.5, min(15.0, 60.0 / max(1, args.steps + args.warmup)))
    cores = os.cpu_count() or 1
    vals = []
    meas = None
    with mp.get_context("spawn").Pool(cores) as pool:
        for i in range(args.warmup):
            oracle_sample_all_cores(wl, args.workload, args.layers, budget_s=0.5, pool=pool, cores=cores, seed=i)
        for i in range(args.steps):
            meas = oracle_sample_all_cores(wl, args.workload, args.layers, budget_s=per_step_budget, pool=pool,
                                           cores=cores, seed=1000 + i)
            vals.append(meas["value"])
    value = statistics.median(vals)
    meas["value"] = value
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": None,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(wl, l2_policy(wl)),
            "cpu_baseline": meas,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def l2_policy(wl):
    """How the timed steps keep L2 from serving inputs: workloads whose
    per-step inputs exceed twice the 129 MB L2 need nothing, smaller ones are
    flushed between steps."""
    big = wl.rows * wl.d * 2 * 3 * wl.L > 2 * (129 << 20)
    return "inputs larger than L2" if big else "flushed between steps (512 MB write)"


def workload_config(wl, flush):
    eps = wl.episodes
    cfg = {"workload": wl.name, "describe": wl.describe, "layers": wl.L, "episodes": wl.E,
           "heads": wl.H, "head_dim": wl.dh, "groups": wl.G, "role_dim": wl.C, "router_hidden": wl.F,
           "cache_tokens_per_layer": wl.rows, "query_tokens_per_layer": wl.q_rows,
           "routed_tokens_per_layer": sum(n for ep in eps for n, k in zip(ep.n_tok(), ep.k(wl.G)) if 0 < k < wl.G),
           "global_batch": wl.E, "parallelism": "replicas: independent episodes per GPU"}
    if flush is not None:
        cfg["l2"] = flush
    return cfg


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

def run_ours(args):
    import torch
    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())
    from paper_2608_18410_gb300 import build as pb
    if rank == 0:
        pb.build()
    barrier(ws)
    from paper_2608_18410_gb300 import rolesub, synth

    wl = make_workload(args.workload, rank, args.layers)
    inp = synth.gen_inputs(wl)
    rs = rolesub.RoleSub(wl.L, wl.H, wl.dh, wl.G, wl.C, wl.F, wl.dtype, wl.n_tok_array(), wl.k_array(),
                         wl.n_query_array(), device=dev)

    def to_dev(x):
        t = torch.from_numpy(x.view(np.int16) if x.dtype == np.uint16 else x)
        t = t.to(dev)
        return t.view(torch.bfloat16) if x.dtype == np.uint16 else t
    d = {k: to_dev(v) for k, v in inp.items()}
    packed, idx = rs.new_outputs()
    o = torch.empty((wl.L, max(wl.q_rows, 1), wl.d), dtype=rs.tdtype, device=dev)
    stream = torch.cuda.current_stream()
    big = l2_policy(wl) == "inputs larger than L2"
    flush_buf = None if big else torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def compress():
        rs.compress(d["h"], d["v"], d["R"], d["W_re"], d["b_re"], d["W1"], d["b1"], d["W2"], d["b2"],
                    wl.alpha_role, wl.alpha_lang, packed=packed, idx=idx)

    def attend():
        rs.attend(d["q"], d["K"], packed, idx, d["R"], o=o)

    for _ in range(max(args.warmup, 3)):
        compress()
        attend()
    torch.cuda.synchronize()
    code, _ = rs.device_status()
    assert code == 0, f"device status {code}"

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    barrier(ws)
    torch.cuda.synchronize()
    launches0 = rolesub.rolesub_launch_count()
    with ClockSampler(torch.cuda.current_device()) as clk:
        for i in range(args.steps):
            if flush_buf is not None:
                flush_buf.fill_(i & 0xFF)
            ev[i][0].record(stream)
            compress()
            ev[i][1].record(stream)
            attend()
            ev[i][2].record(stream)
        torch.cuda.synchronize()
    launches = rolesub.rolesub_launch_count() - launches0
    barrier(ws)
    t_comp = [a.elapsed_time(b) for a, b, c in ev]
    t_att = [b.elapsed_time(c) for a, b, c in ev]
    t_step = [x + y for x, y in zip(t_comp, t_att)]
    qtok = wl.q_rows * wl.L
    ms_per_step, value = weak_scaling(sum(t_step), args.steps, qtok, ws)

    # ---- the additive routing score (Sec. 3.4) in place of the concatenation
    # router, same cache, C = 6 role components; timed on its own, after the
    # step --------------------------------------------------------------------
    import dataclasses
    C_ADD = 6
    wl_add = dataclasses.replace(wl, C=C_ADD)
    rs_add = rolesub.RoleSub(wl.L, wl.H, wl.dh, wl.G, C_ADD, wl.F, wl.dtype, wl.n_tok_array(), wl.k_array(),
                             wl.n_query_array(), device=dev)
    add = {k: to_dev(v) for k, v in synth.gen_additive_weights(wl_add).items()}
    W_re_add = d["W_re"][:, :C_ADD].contiguous()
    b_re_add = d["b_re"][:, :C_ADD].contiguous()

    def compress_additive():
        rs_add.compress_additive(d["h"], d["v"], d["R"], W_re_add, b_re_add, add["W_v"], add["b_v"],
                                 add["W_role"], add["W_l"], add["b_l"], wl.alpha_role, wl.alpha_lang,
                                 packed=packed, idx=idx)

    for _ in range(3):
        compress_additive()
    torch.cuda.synchronize()
    ev_add = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps)]
    for i in range(args.steps):
        if flush_buf is not None:
            flush_buf.fill_(i & 0xFF)
        ev_add[i][0].record(stream)
        compress_additive()
        ev_add[i][1].record(stream)
    torch.cuda.synchronize()
    code, _ = rs_add.device_status()
    assert code == 0, f"device status {code}"
    add_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_add)

    # ---- per-token budgets (Sec. 3.5): compress_budget + attend_budget on
    # the same cache (segment budgets B_m = K_m n), timed on their own -------
    u_pri = torch.from_numpy(synth.gen_priority(wl_add)).to(dev)
    k_tok = torch.empty((wl.L, max(wl.rows, 1)), dtype=torch.uint8, device=dev)

    def compress_budget():
        rs_add.compress_budget(d["h"], d["v"], d["R"], W_re_add, b_re_add, add["W_v"], add["b_v"], add["W_role"],
                               add["W_l"], add["b_l"], u_pri, wl.alpha_role, wl.alpha_lang, packed=packed,
                               idx=idx, k_tok=k_tok)

    def attend_budget():
        rs_add.attend_budget(d["q"], d["K"], packed, idx, k_tok, d["R"], o=o)

    for _ in range(3):
        compress_budget()
        attend_budget()
    torch.cuda.synchronize()
    ev_bud = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
               torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for i in range(args.steps):
        if flush_buf is not None:
            flush_buf.fill_(i & 0xFF)
        ev_bud[i][0].record(stream)
        compress_budget()
        ev_bud[i][1].record(stream)
        attend_budget()
        ev_bud[i][2].record(stream)
    torch.cuda.synchronize()
    code, _ = rs_add.device_status()
    assert code == 0, f"device status {code}"
    bud_c_ms = statistics.mean(a.elapsed_time(b) for a, b, c in ev_bud)
    bud_a_ms = statistics.mean(b.elapsed_time(c) for a, b, c in ev_bud)

    # ---- token-level reduction (Sec. 3.1) ahead of the cache: 64 episodes x
    # 2 camera views x 256 visual tokens, hidden d, ratio 1/16 (32 of 512) ---
    sel_scores = torch.randn(64, 2, 256, device=dev)
    sel_x = torch.randn(64, 2, 256, wl.d, device=dev).to(rs.tdtype)
    sel_k = rolesub.rolesub_select_count(256, 0.0625)
    sel_idx = torch.empty((64, 2, sel_k), dtype=torch.int32, device=dev)
    sel_out = torch.empty((64, 2, sel_k, wl.d), dtype=rs.tdtype, device=dev)
    for _ in range(3):
        rolesub.rolesub_select_tokens(sel_scores, sel_x, 0.0625, sel_idx, sel_out)
    torch.cuda.synchronize()
    # the kept rows (17 MB) would stay in L2 between calls: flush before each
    sel_flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    ev_sel = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps)]
    for i in range(args.steps):
        sel_flush.fill_(i & 0xFF)
        ev_sel[i][0].record(stream)
        rolesub.rolesub_select_tokens(sel_scores, sel_x, 0.0625, sel_idx, sel_out)
        ev_sel[i][1].record(stream)
    torch.cuda.synchronize()
    sel_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_sel)
    del sel_flush
    sel_bytes = 64 * 2 * (256 * 4 + sel_k * 4 + 2 * sel_k * wl.d * sel_out.element_size())
    del sel_x

    # ---- the dense-rotation geometry (one d x d R per layer): compress_dense
    # + attend_dense on the same cache, timed on their own ------------------
    R_dense = to_dev(synth.gen_dense_rotation(wl))
    rs.compress_dense(d["h"], d["v"], R_dense, d["W_re"], d["b_re"], d["W1"], d["b1"], d["W2"], d["b2"],
                      wl.alpha_role, wl.alpha_lang, packed=packed, idx=idx)
    rs.attend_dense(d["q"], d["K"], packed, idx, R_dense, o=o)
    torch.cuda.synchronize()
    ev_den = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
               torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for i in range(args.steps):
        ev_den[i][0].record(stream)
        rs.compress_dense(d["h"], d["v"], R_dense, d["W_re"], d["b_re"], d["W1"], d["b1"], d["W2"], d["b2"],
                          wl.alpha_role, wl.alpha_lang, packed=packed, idx=idx)
        ev_den[i][1].record(stream)
        rs.attend_dense(d["q"], d["K"], packed, idx, R_dense, o=o)
        ev_den[i][2].record(stream)
    torch.cuda.synchronize()
    code, _ = rs.dense_device_status()
    assert code == 0, f"device status {code}"
    den_c_ms = statistics.mean(a.elapsed_time(b) for a, b, c in ev_den)
    den_a_ms = statistics.mean(b.elapsed_time(c) for a, b, c in ev_den)
    del R_dense
    rs._dws = None

    # ---- one OpenVLA-OFT layer (c1), a launch-latency-bound step: eager
    # calls and the same step replayed from a CUDA graph, L2 flushed --------
    wl1 = synth.c1()
    inp1 = synth.gen_inputs(wl1)
    rs1 = rolesub.RoleSub(wl1.L, wl1.H, wl1.dh, wl1.G, wl1.C, wl1.F, wl1.dtype, wl1.n_tok_array(),
                          wl1.k_array(), wl1.n_query_array(), device=dev)
    d1 = {k: to_dev(v) for k, v in inp1.items()}
    p1, i1 = rs1.new_outputs()
    o1 = torch.empty((wl1.L, wl1.q_rows, wl1.d), dtype=rs1.tdtype, device=dev)
    lat_flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def step1():
        rs1.compress(d1["h"], d1["v"], d1["R"], d1["W_re"], d1["b_re"], d1["W1"], d1["b1"], d1["W2"], d1["b2"],
                     wl1.alpha_role, wl1.alpha_lang, packed=p1, idx=i1)
        rs1.attend(d1["q"], d1["K"], p1, i1, d1["R"], o=o1)

    gstream = torch.cuda.Stream()
    gstream.wait_stream(stream)
    with torch.cuda.stream(gstream):
        for _ in range(3):
            step1()
    stream.wait_stream(gstream)
    torch.cuda.synchronize()
    graph1 = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph1):
        step1()

    def time_latency(fn):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        for i in range(args.steps):
            lat_flush.fill_(i & 0xFF)
            evs[i][0].record(stream)
            fn()
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    lat_eager = time_latency(step1)
    lat_graph = time_latency(graph1.replay)
    del graph1

    # ---- one robot-control step: a single episode through all 32 layers,
    # eager calls, L2 flushed before each step: c2's point of 128 visual
    # tokens keeping 4 of 16 groups + 48 language tokens, and c3's
    # aggressive joint compression (64 visual at 2 of 16, 48 language at 4
    # of 16, router near-ties) -----------------------------------------------
    def single_episode_ms(wl_s):
        inp_s = synth.gen_inputs(wl_s)
        rs_s = rolesub.RoleSub(wl_s.L, wl_s.H, wl_s.dh, wl_s.G, wl_s.C, wl_s.F, wl_s.dtype, wl_s.n_tok_array(),
                               wl_s.k_array(), wl_s.n_query_array(), device=dev)
        d_s = {k: to_dev(v) for k, v in inp_s.items()}
        p_s, i_s = rs_s.new_outputs()
        o_s = torch.empty((wl_s.L, wl_s.q_rows, wl_s.d), dtype=rs_s.tdtype, device=dev)

        def step_s():
            rs_s.compress(d_s["h"], d_s["v"], d_s["R"], d_s["W_re"], d_s["b_re"], d_s["W1"], d_s["b1"], d_s["W2"],
                          d_s["b2"], wl_s.alpha_role, wl_s.alpha_lang, packed=p_s, idx=i_s)
            rs_s.attend(d_s["q"], d_s["K"], p_s, i_s, d_s["R"], o=o_s)

        for _ in range(3):
            step_s()
        torch.cuda.synchronize()
        ms = time_latency(step_s)
        code, _ = rs_s.device_status()
        assert code == 0, f"device status {code}"
        return ms

    wl2, wl3 = synth.c2(128, 4), synth.c3()
    ctl_ms = single_episode_ms(wl2)
    c3_ms = single_episode_ms(wl3)
    del lat_flush

    # ---- end to end through the public API from pinned host buffers. The
    # layers go in chunks of E2E_CHUNK: a chunk's activations are copied in
    # on one stream, compress + attend run on the launching stream, and its
    # output is copied out on a third, so that copies in, compute and copies
    # out of neighbouring chunks overlap (the host link bounds the step).
    # Every step copies all of its inputs in and all of o out. -------------
    act = ("h", "v", "K", "q")
    host = {}
    for k in act:
        x = inp[k]
        t = torch.from_numpy(x.view(np.int16) if x.dtype == np.uint16 else x).pin_memory()
        host[k] = t
    o_host = torch.empty(o.shape, dtype=torch.int16 if o.dtype == torch.bfloat16 else o.dtype).pin_memory()
    h2d = sum(host[k].numel() * host[k].element_size() for k in act)
    d2h = o_host.numel() * o_host.element_size()
    dv = {k: (d[k].view(torch.int16) if d[k].dtype == torch.bfloat16 else d[k]) for k in act}
    ov = o.view(torch.int16) if o.dtype == torch.bfloat16 else o
    chunks = [(l0, min(wl.L, l0 + E2E_CHUNK)) for l0 in range(0, wl.L, E2E_CHUNK)]
    rs_chunk = {}
    for l0, l1 in chunks:
        if l1 - l0 not in rs_chunk:
            rs_chunk[l1 - l0] = rolesub.RoleSub(l1 - l0, wl.H, wl.dh, wl.G, wl.C, wl.F, wl.dtype, wl.n_tok_array(),
                                                wl.k_array(), wl.n_query_array(), device=dev)
    outs = [rs_chunk[l1 - l0].new_outputs() for l0, l1 in chunks]   # a chunk's own packed cache and indices
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in chunks]
    ev_done = [torch.cuda.Event() for _ in chunks]
    ev_out = [torch.cuda.Event() for _ in chunks]
    e2e_state = {"steps": 0}

    def e2e_step():
        later = e2e_state["steps"] > 0
        for c, (l0, l1) in enumerate(chunks):
            if later:
                s_in.wait_event(ev_done[c])    # the previous step's compute has read this chunk's inputs
            with torch.cuda.stream(s_in):
                for k in act:
                    dv[k][l0:l1].copy_(host[k][l0:l1], non_blocking=True)
                ev_in[c].record(s_in)
            stream.wait_event(ev_in[c])
            if later:
                stream.wait_event(ev_out[c])   # the previous step's o of this chunk has been copied out
            r = rs_chunk[l1 - l0]
            pk, ix = outs[c]
            r.compress(d["h"][l0:l1], d["v"][l0:l1], d["R"][l0:l1], d["W_re"][l0:l1], d["b_re"][l0:l1],
                       d["W1"][l0:l1], d["b1"][l0:l1], d["W2"][l0:l1], d["b2"][l0:l1], wl.alpha_role,
                       wl.alpha_lang, packed=pk, idx=ix, stream=stream)
            r.attend(d["q"][l0:l1], d["K"][l0:l1], pk, ix, d["R"][l0:l1], o=o[l0:l1], stream=stream)
            ev_done[c].record(stream)
            s_out.wait_event(ev_done[c])
            with torch.cuda.stream(s_out):
                o_host[l0:l1].copy_(ov[l0:l1], non_blocking=True)
                ev_out[c].record(s_out)
        e2e_state["steps"] += 1

    compress()                   # o of the whole-workload calls, to check the chunked steps against
    attend()
    o_whole = o.clone()
    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize()
    e2e_same = bool(torch.equal(o, o_whole))
    del o_whole
    for r in rs_chunk.values():
        code, _ = r.device_status()
        assert code == 0, f"device status {code}"
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e2e_steps = max(1, min(args.steps, 20))
    barrier(ws)
    e0.record(stream)
    s_in.wait_stream(stream)     # nothing of the timed steps starts before e0
    for _ in range(e2e_steps):
        e2e_step()
    stream.wait_stream(s_out)    # e1 after the last output copy
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), ws) / e2e_steps
    e2e_value = qtok * ws / (e2e_ms / 1e3)

    # ---- roofline of the dominant kernel --------------------------------
    peaks = load_peaks()
    att_ms = statistics.mean(t_att)
    comp_ms = statistics.mean(t_comp)
    ab = attend_bytes(wl)
    cb = compress_bytes(wl)
    att_gbs = ab / (att_ms / 1e3) / 1e9
    roof = {"kernel": "k_attend_tc (timed as the whole rolesub_attend call: the k_row_store pre-pass "
                      "of a few us, then the attention kernel)", "bound": "hbm",
            "achieved": att_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": att_gbs / peaks["hbm_gbs"], "peak_source": peaks["source"] + " hbm_gbs (copy)",
            "algorithmic_bytes_per_launch": ab, "avg_launch_ms": att_ms,
            "traffic": load_traffic("attend_tc", wl.name),
            "frac_of_8TBs": att_gbs / 8000.0,
            "tensor_tflops": attend_flops(wl) / (att_ms / 1e3) / 1e12}
    comp = {"ms": comp_ms, "algorithmic_bytes": cb, "GB/s": cb / (comp_ms / 1e3) / 1e9,
            "frac": cb / (comp_ms / 1e3) / 1e9 / peaks["hbm_gbs"]}
    cab = compress_additive_bytes(wl, C_ADD)
    comp_add = {"ms": add_ms, "role_dim": C_ADD, "algorithmic_bytes": cab, "GB/s": cab / (add_ms / 1e3) / 1e9,
                "frac": cab / (add_ms / 1e3) / 1e9 / peaks["hbm_gbs"]}
    # only kept groups are rotated: z_s = R_s^T v (compress) and v~ = sum over
    # kept s of R_s z_s (attend), 2 g d flop per kept (row, group) pair each
    kept_pairs = int((wl.n_tok_array().astype(np.int64) * wl.k_array()).sum()) * wl.L
    kept_flop = 2.0 * (wl.d // wl.G) * wl.d * kept_pairs
    dense = {"compress_ms": den_c_ms, "attend_ms": den_a_ms,
             "kept_pairs": kept_pairs,
             "rotation_tflop_kept": kept_flop / 1e12,
             "compress_tflops_kept": kept_flop / (den_c_ms / 1e3) / 1e12,
             "attend_tflops_kept": kept_flop / (den_a_ms / 1e3) / 1e12,
             "all_groups_tflop": 2.0 * wl.rows * wl.d * wl.d * wl.L / 1e12,
             "query_tokens_per_s_per_layer": qtok / ((den_c_ms + den_a_ms) / 1e3),
             "r": "one d x d orthonormal R per layer (kron of two 64 x 64 Haar factors)"}
    latency = {"workload": wl1.name, "l2": "flushed before each step", "eager_ms": lat_eager,
               "graph_ms": lat_graph, "query_tokens_per_s_per_layer_graph": wl1.q_rows / (lat_graph / 1e3)}
    control = {"workload": wl2.name, "describe": wl2.describe, "layers": wl2.L,
               "l2": "flushed before each step", "ms_per_step": ctl_ms,
               "query_tokens_per_s_per_layer": wl2.q_rows * wl2.L / (ctl_ms / 1e3)}
    step_c3 = {"workload": wl3.name, "describe": wl3.describe, "layers": wl3.L,
               "l2": "flushed before each step", "ms_per_step": c3_ms,
               "query_tokens_per_s_per_layer": wl3.q_rows * wl3.L / (c3_ms / 1e3)}
    select = {"episodes": 64, "views": 2, "tokens_per_view": 256, "kept_per_view": sel_k, "ms": sel_ms,
              "l2": "flushed before each call",
              "algorithmic_bytes": sel_bytes, "GB/s": sel_bytes / (sel_ms / 1e3) / 1e9}
    budget = {"role_dim": C_ADD, "compress_ms": bud_c_ms, "compress_GB/s": cab / (bud_c_ms / 1e3) / 1e9,
              "attend_ms": bud_a_ms, "attend_GB/s": ab / (bud_a_ms / 1e3) / 1e9,
              "attend_frac": ab / (bud_a_ms / 1e3) / 1e9 / peaks["hbm_gbs"],
              "query_tokens_per_s_per_layer": qtok / ((bud_c_ms + bud_a_ms) / 1e3)}

    clocks = clk.summary()
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
            "config": workload_config(wl, l2_policy(wl)),
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": e2e_ms,
                    "pipeline": f"{len(chunks)} chunks of {E2E_CHUNK} layers: copies in, compute, copies out "
                                "on three streams",
                    "o_equals_whole_workload_call": e2e_same},
            "gpu_launches": launches,
            "roofline": roof, "compress": comp, "compress_additive": comp_add, "budget": budget,
            "select_tokens": select, "latency_one_layer": latency, "control_step_c2": control, "step_c3": step_c3, "dense_rotation": dense,
            "clocks": {"sm_mhz": clocks["sm_mhz"], "sm_max_mhz": clocks["sm_max_mhz"],
                       "reasons": clocks["reasons"], "samples": clocks["samples"]}}
    if ws == 1 and rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = oracle_sample_all_cores(wl, args.workload, args.layers, budget_s=args.cpu_budget)
        line["cpu_baseline"]["single_thread"] = oracle_sample(wl, inp, budget_s=args.cpu_budget)
    if rank == 0:
        print(json.dumps(line))
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=os.environ.get("ROLESUB_BENCH_WORKLOAD", "c4"),
                    choices=["c1", "c2", "c3", "c4"])
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--layers", type=int, default=0,
                    help="run only this many layers of the workload (small profiling captures)")
    args = ap.parse_args(argv)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
