"""Benchmark: MAR-B-shaped 64-step decode with LazyMAR's caches on one GB300.

One benchmark step is one whole decode of a batch: 64 decoding steps of a
MAR-B-shaped transformer (24 blocks, width 768, 12 heads, 64 buffer + 256
image tokens) over 32 class-conditional + 32 unconditional rows, following the
periodic cache-reuse-refreshment schedule (full steps for k < 4 and every 9
steps after, cached steps recomputing 50 of 320 tokens per row in between, the
condition cache reused on every other cached step). Inputs (latents and masks
of all 64 steps, labels) are synthetic and seeded, resident in HBM before the
timed region; weights are random-init bf16 of the MAR-B shapes.

Prints one JSON line (rank 0): images/s of the whole job, decoding steps/s, the
full-recompute decode on the same GPU, per-kernel-class device time from CUDA
events recorded around each launch on its stream, the GEMM roofline against
the measured bf16 peak, an end-to-end figure through the C ABI with host
buffers, SM clocks sampled during the timed region, and the CPU oracle timed on
a bounded sample of the same workload.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Multi-GPU (torchrun, one process per GPU): cond/uncond pairs are independent,
so every rank decodes its own batch (weak scaling, no data-path collective);
the timed region is bracketed by barriers and the maximum over ranks is used.
"""
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

import synth  # noqa: E402

METRIC = "MAR-B-shaped 256-token decode: steps/sec and images/sec at 1 GB300; tensor-pipe % of peak"
GAMMA = 3.0
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


NAMES = {"mar_b": "MAR-B", "mar_l": "MAR-L", "mar_h": "MAR-H", "hires": "MAR-L high-resolution", "tiny": "tiny"}


def workload(cfg, select="least_similar"):
    n = synth.n_compute(cfg)
    return {
        "workload": "%s-shaped %d-step LazyMAR decode (%d blocks, width %d, %d heads, %d+%d tokens)" % (
            NAMES.get(cfg["name"], cfg["name"]), cfg["steps"], cfg["depth"], cfg["width"], cfg["heads"],
            cfg["n_buffer"], cfg["n_img"]),
        "batch_pairs": cfg["batch"], "rows": 2 * cfg["batch"], "tokens": cfg["T"],
        "recompute": "%d/%d tokens per row" % (n, cfg["T"]),
        "schedule": "full for k<%d and every %d steps; %s" % (
            cfg["k0"], cfg["tau"], "no condition cache" if cfg["tau_cfg"] == 0 else
            "cond cache reused on cached steps with (k-k0) %% %d != 0" % cfg["tau_cfg"]),
        "decoding_steps": cfg["steps"],
        "selection": select,
        "cached_qkv_operands": "e4m3" if cfg.get("qkv_e4m3") else "bf16",
        "l2": "no flush: the per-step working set (%.2f GB weights + %.2f GB K/V cache) exceeds the 129 MB L2" % (
            12 * cfg["depth"] * cfg["width"] ** 2 * 2 / 1e9,
            2 * (cfg["depth"] - cfg["sel_layers"]) * 2 * cfg["batch"] * cfg["T"] * cfg["width"] * 2 / 1e9),
    }


def schedule(cfg, plan_fn):
    return [plan_fn(k, cfg["k0"], cfg["tau"], cfg["tau_cfg"], True) for k in range(cfg["steps"])]


SELECT_RULES = {"least_similar": 0, "most_similar": 1, "random": 2, "observation": 0}


def selection_inputs(cfg, masks, rule_name, seed_offset):
    """Per-step selection inputs of the Table 3 strategies for [2B, T] rows (a
    cond-reuse step uses the first B): random keys (strategy III, seeded) or
    observation-based priorities (1 for the image tokens decoded at the
    previous step and at this step, Sec. 3.2.1); None where unused."""
    steps, B, n_img = masks.shape
    T, nb = cfg["T"], cfg["n_buffer"]
    if rule_name == "random":
        rng = np.random.default_rng(4 + seed_offset)
        return None, rng.integers(0, 1 << 32, size=(steps, 2 * B, T), dtype=np.uint64).astype(np.uint32)
    if rule_name != "observation":
        return None, None
    prio = np.zeros((steps, 2 * B, T), np.uint8)
    for k in range(steps):
        prev = masks[k - 1] if k > 0 else np.ones_like(masks[0])
        nxt = masks[k + 1] if k + 1 < steps else np.zeros_like(masks[0])
        hot = ((prev != 0) & (masks[k] == 0)) | ((masks[k] != 0) & (nxt == 0))
        prio[k, :B, nb:] = hot
        prio[k, B:, nb:] = hot
    return prio, None


def rank_seed_offset(rank):
    """Seed offset of a rank's inputs: every rank decodes its own batch of pairs
    (weak scaling; pairs are independent, so no data-path collective)."""
    return rank * 101


def max_over_ranks(values, device):
    """Element-wise maximum over all ranks (the slowest rank's timing)."""
    import torch
    import torch.distributed as dist
    if not dist.is_initialized() or dist.get_world_size() == 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t]


def job_images_per_s(world, batch, decodes, ms):
    """Whole-job throughput: `world` ranks each decode `batch` pairs `decodes`
    times within `ms` (the maximum over ranks)."""
    return world * batch * decodes / (ms / 1000.0)


def decode_inputs(cfg, seed_offset):
    """Latents and masks of every decoding step for one batch (numpy)."""
    order = synth.make_order(cfg, seed=2 + seed_offset)
    table = synth.make_latent_table(cfg, seed=3 + seed_offset)
    labels = synth.make_labels(cfg, seed=1 + seed_offset)
    m = synth.mask_counts(cfg["steps"], cfg["n_img"])
    lats, masks = [], []
    for k in range(cfg["steps"]):
        n_dec = cfg["n_img"] - (m[k - 1] if k > 0 else cfg["n_img"])
        lat, mask = synth.step_state(cfg, order, table, n_dec)
        lats.append(lat)
        masks.append(mask)
    return np.stack(lats), np.stack(masks), labels


# --------------------------------------------------------------------------
# Clocks sampled during the timed region
# --------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap"]

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.t.join(timeout=5)

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------------------
# CPU oracle baseline (bounded sample)
# --------------------------------------------------------------------------

def oracle_sample(cfg, plan):
    """Times the oracle on one cond/uncond pair: a full step, a cached step with
    both pathways and a condition-cache reuse step; scales to images/s with the
    schedule's step counts."""
    import oracle as O
    c1 = dict(cfg, batch=1)
    W = synth.make_weights(c1)
    lat, mask, labels = decode_inputs(c1, 0)
    N = synth.n_compute(cfg)
    cache = O.Cache(c1, 1)
    t0 = time.perf_counter()
    O.full_step(c1, W, cache, lat[10], mask[10], labels, GAMMA)
    t1 = time.perf_counter()
    O.cached_step(c1, W, cache, lat[11], mask[11], labels, N, False, GAMMA)
    t2 = time.perf_counter()
    O.cached_step(c1, W, cache, lat[12], mask[12], labels, N, True, GAMMA)
    t3 = time.perf_counter()
    n_full = sum(1 for f, r in plan if f)
    n_reuse = sum(1 for f, r in plan if not f and r)
    n_both = len(plan) - n_full - n_reuse
    sec_per_image = n_full * (t1 - t0) + n_both * (t2 - t1) + n_reuse * (t3 - t2)
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS") or os.environ.get("OMP_NUM_THREADS") or os.cpu_count())
    return {
        "value": 1.0 / sec_per_image, "unit": "images/s", "cores": cores, "kind": "oracle",
        "sample": "one cond/uncond pair: 1 full + 1 cached + 1 cond-reuse step (%.1f s of fp64 numpy), scaled by "
                  "the 64-step schedule (%d full, %d cached, %d cond-reuse)" % (t3 - t0, n_full, n_both, n_reuse),
        "sample_s": t3 - t0,
    }


def run_reference(args, cfg, plan):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    for _ in range(args.warmup):
        oracle_sample(cfg, plan)
    vals, secs = [], []
    cb = None
    for _ in range(args.steps):
        cb = oracle_sample(cfg, plan)
        vals.append(cb["value"])
        secs.append(cb["sample_s"])
    value = statistics.median(vals)
    cb = dict(cb, value=value)
    cb.pop("sample_s", None)
    # each step is one bounded sample (three decoding steps of one pair);
    # images/s is extrapolated from it by the schedule's step counts and B
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "images/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * statistics.mean(secs),
            "step": "one sample: 1 full + 1 cached + 1 cond-reuse decoding step of one cond/uncond pair",
            "value_extrapolated": "images/s = 1 / (schedule-weighted sample seconds); one sample stands for one "
                                  "image's 64-step decode (pairs are independent)",
            "timed_s": sum(secs), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": workload(cfg, args.select),
            "cpu_baseline": cb, "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0,
                                        "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------
# GPU arm
# --------------------------------------------------------------------------

def run_ours(args, cfg):
    import torch
    import torch.distributed as dist

    from paper_2503_12450_gb300 import build as libbuild
    from paper_2503_12450_gb300 import lazymar as lm

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    if rank == 0:
        libbuild.build()
    if world > 1:
        dist.barrier()
    lm.lib()
    plan = schedule(cfg, lm.lazymar_plan_step)

    B, N, steps = cfg["batch"], synth.n_compute(cfg), cfg["steps"]
    W = synth.make_weights(cfg)
    h = lm.lazymar_create(dict(cfg, max_batch=B, select_rule=SELECT_RULES[args.select]), W)
    lat_np, mask_np, labels_np = decode_inputs(cfg, rank_seed_offset(rank))
    lat = torch.from_numpy(lat_np).cuda()
    mask = torch.from_numpy(mask_np).cuda()
    labels = torch.from_numpy(labels_np).cuda()
    prio_np, keys_np = selection_inputs(cfg, mask_np, args.select, rank_seed_offset(rank))
    prio = None if prio_np is None else torch.from_numpy(prio_np).cuda()
    keys = None if keys_np is None else torch.from_numpy(keys_np.view(np.int32)).cuda()
    guided = torch.empty((B, cfg["n_img"], cfg["width"]), dtype=torch.bfloat16, device="cuda")
    zbuf = torch.empty((2 * B, cfg["n_img"], cfg["width"]), device="cuda",
                       dtype=torch.bfloat16 if cfg["dtype"] == "bf16" else torch.float32)
    stream = torch.cuda.current_stream()
    dev_in = {"lat": lat, "mask": mask, "labels": labels, "guided": guided, "prio": prio, "keys": keys}

    def decode(full_only=False, host=None, step_events=None, head_step=None, after_step=None):
        for k in range(steps):
            full, reuse = plan[k]
            src = host if host is not None else dev_in
            l_k, m_k, lab, g = src["lat"][k], src["mask"][k], src["labels"], src["guided"]
            p_k = None if src["prio"] is None else src["prio"][k]
            r_k = None if src["keys"] is None else src["keys"][k]
            if step_events is not None:
                step_events[k][0].record(stream)
            z = None if head_step is None else zbuf
            if full or full_only:
                lm.lazymar_full_step(h, l_k, m_k, lab, B, GAMMA, z, g, stream)
            else:
                lm.lazymar_cached_step(h, l_k, m_k, lab, B, N, reuse, GAMMA, None, None, z, g, stream,
                                       select_priority=p_k, select_keys=r_k)
            if head_step is not None:
                head_step(k)
            if after_step is not None:
                after_step(k)
            if step_events is not None:
                step_events[k][1].record(stream)
        if host is not None:
            stream.synchronize()  # the caller reads the last step's guided output

    def timed(fn, k_steps):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0 = time.perf_counter()
        e0.record(stream)
        for _ in range(k_steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        ms = e0.elapsed_time(e1)
        if world > 1:
            ms, wall_ms = max_over_ranks([ms, wall * 1000.0], "cuda")
            wall = wall_ms / 1000.0
            dist.barrier()
        return ms, wall

    for _ in range(args.warmup):
        decode()
    lm.lazymar_sync(h, stream)

    # 1) the headline: device-resident inputs, CUDA events around K decodes
    lm.lazymar_reset_stats(h)
    with ClockSampler(local) as clocks:
        ms, wall = timed(decode, args.steps)
    st = lm.lazymar_get_stats(h)
    launches = sum(v["launches"] for v in st.values())
    lm.lazymar_sync(h, stream)
    ms_per_step = ms / args.steps
    images_per_s = job_images_per_s(world, B, args.steps, ms)

    # 2a) step times by kind: the same graph-replayed decode with events
    # between steps only
    step_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    kind_ms = {"full": [], "cached": [], "cached_reuse": []}
    for _ in range(max(1, min(args.steps, 3))):
        decode(step_events=step_ev)
        torch.cuda.synchronize()
        for k in range(steps):
            full, reuse = plan[k]
            kind = "full" if full else ("cached_reuse" if reuse else "cached")
            kind_ms[kind].append(step_ev[k][0].elapsed_time(step_ev[k][1]))

    # 2b) per-kernel device time: events around every launch (separate pass;
    # the library captures each step body with its events into a CUDA graph,
    # so the times exclude the host's launch submission)
    lm.lazymar_reset_stats(h)
    lm.lazymar_set_profiling(h, True)
    # GEMM flops and event time per step kind (statistics read after every step)
    kind_gemm = {k: [0.0, 0.0] for k in kind_ms}
    last = [lm.lazymar_get_stats(h)["gemm"]]

    def after_step(k):
        g = lm.lazymar_get_stats(h)["gemm"]
        full, reuse = plan[k]
        kind = "full" if full else ("cached_reuse" if reuse else "cached")
        kind_gemm[kind][0] += g["flops"] - last[0]["flops"]
        kind_gemm[kind][1] += g["ms"] - last[0]["ms"]
        last[0] = g

    decode(after_step=after_step)             # captures the profiled graphs
    torch.cuda.synchronize()
    lm.lazymar_reset_stats(h)
    kind_gemm = {k: [0.0, 0.0] for k in kind_ms}
    last[0] = lm.lazymar_get_stats(h)["gemm"]
    for _ in range(max(1, min(args.steps, 3))):
        decode(after_step=after_step)
        torch.cuda.synchronize()
    prof = lm.lazymar_get_stats(h)
    lm.lazymar_set_profiling(h, False)
    lm.lazymar_sync(h, stream)

    # 3) full recompute on the same GPU (every decoding step a full step)
    for _ in range(1):
        decode(full_only=True)
    ms_full, _ = timed(lambda: decode(full_only=True), args.steps)
    full_images_per_s = job_images_per_s(world, B, args.steps, ms_full)

    # 4) end to end through the C ABI with host buffers (pinned), copies inside
    host = {"lat": lat.cpu().pin_memory(), "mask": mask.cpu().pin_memory(), "labels": labels.cpu().pin_memory(),
            "guided": torch.empty(tuple(guided.shape), dtype=torch.bfloat16).pin_memory(),
            "prio": None if prio is None else prio.cpu().pin_memory(),
            "keys": None if keys is None else keys.cpu().pin_memory()}
    decode(host=host)
    ms_e2e, _ = timed(lambda: decode(host=host), args.steps)
    e2e_images_per_s = job_images_per_s(world, B, args.steps, ms_e2e)
    # selection inputs are copied on cached steps only, for the rows they run
    cached_rows = sum(0 if f else (B if r else 2 * B) for f, r in plan)
    sel_bytes = cached_rows * cfg["T"] * ((1 if prio is not None else 0) + (4 if keys is not None else 0))
    h2d = steps * (lat[0].numel() * 4 + mask[0].numel() + labels.numel() * 4) + sel_bytes
    d2h = steps * guided.numel() * 2
    lm.lazymar_sync(h, stream)

    # 5) the whole MAR sampling step: after every decoding step the diffusion
    # head draws the latents of the tokens that step decodes (100 denoising
    # steps, guidance on the noise prediction)
    with_head = None
    if not args.no_head:
        with_head = run_head_phase(args, cfg, lm, torch, mask_np, rank, stream, decode, timed, world, zbuf)
    lm.lazymar_sync(h, stream)

    if rank != 0:
        h.close()
        dist.destroy_process_group()
        return

    pk, src = peaks()
    peak_tf = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
    g = prof["gemm"]
    gemm_tflops = g["flops"] / (g["ms"] / 1000.0) / 1e12 if g["ms"] > 0 else None
    total_ms = sum(v["ms"] for v in prof.values())
    kernels = {}
    for name, v in prof.items():
        if v["timed_launches"] == 0:
            continue
        kernels[name] = {"launches": v["timed_launches"], "ms": round(v["ms"], 3),
                         "share": round(v["ms"] / total_ms, 4) if total_ms else None,
                         "tflops": round(v["flops"] / (v["ms"] / 1e3) / 1e12, 2) if v["flops"] and v["ms"] else None,
                         "gbs": round(v["bytes"] / (v["ms"] / 1e3) / 1e9, 1) if v["ms"] else None}
    peak_burst = pk["bf16_tflops"]

    def gemm_rate(flops, ms):
        if ms <= 0:
            return None
        tf = flops / (ms / 1e3) / 1e12
        return {"tflops": round(tf, 1), "frac_of_sustained": round(tf / peak_tf, 4),
                "frac_of_burst": round(tf / peak_burst, 4)}

    gemm_by_kind = {k: gemm_rate(*v) for k, v in kind_gemm.items() if v[1] > 0}
    cf = kind_gemm["cached"][0] + kind_gemm["cached_reuse"][0]
    cm = kind_gemm["cached"][1] + kind_gemm["cached_reuse"][1]
    gemm_by_kind["cached_steps_all"] = gemm_rate(cf, cm)
    traffic, traffic_source = None, None
    tpath = os.path.join(ROOT, "profiles", "gemm_traffic.json")  # captured on the MAR-B decode
    if cfg["name"] == "mar_b" and os.path.exists(tpath):
        with open(tpath) as f:
            tj = json.load(f)
        traffic = tj.get("bytes_per_launch")
        traffic_source = tj.get("source")
    line = {
        "metric": METRIC, "value": images_per_s, "unit": "images/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded latents/masks, random-init MAR-B weights)",
        "config": workload(cfg, args.select),
        "decoding_steps_per_s": world * steps * args.steps / (ms / 1000.0),
        "step_ms": {k: round(statistics.mean(v), 3) for k, v in kind_ms.items() if v},
        "full_recompute": {"value": full_images_per_s, "unit": "images/s", "ms_per_step": ms_full / args.steps,
                           "speedup": images_per_s / full_images_per_s},
        "roofline": {"bound": "tensor", "kernel": "gemm_bf16_tc (tcgen05)", "achieved": gemm_tflops,
                     "peak": peak_tf, "unit": "TFLOP/s",
                     "frac": (gemm_tflops / peak_tf) if gemm_tflops else None,
                     "peak_source": "%s bf16 sustained" % src, "traffic": traffic,
                     "traffic_source": traffic_source,
                     "timing": "CUDA events around every GEMM launch, each step body replayed from a CUDA graph"},
        "kernels": kernels,
        "gemm_by_step_kind": gemm_by_kind,
        "e2e": {"value": e2e_images_per_s, "unit": "images/s", "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h)},
        "gpu_launches": int(launches),
        "clocks": clocks.summary(),
        "with_head": with_head,
        "wall_s": wall,
    }
    if not args.no_cpu_baseline and world == 1:
        line["cpu_baseline"] = oracle_sample(cfg, plan)
        line["cpu_baseline"].pop("sample_s", None)
    print(json.dumps(line), flush=True)
    h.close()
    if world > 1:
        dist.destroy_process_group()


def profile_case(args, cfg):
    """One launch of each kernel of a layer at the configuration's shapes, for a
    profiler: `gemm_layers` runs QKV, out-proj, fc1 and fc2 on all rows x T
    tokens, on the recomputed rows x N tokens and on the half of them a
    condition-reuse step runs; `attention_layers` runs the
    recomputed-token and the full-layer attention; `head` runs one eager
    diffusion-head sampling call (100 steps) for 4 new tokens per pair;
    `steps` runs one full and one cached step eagerly; `launch_floor` times the
    recomputed-token GEMMs and a minimal kernel inside CUDA graphs, back to
    back and with an event pair around every launch."""
    import torch
    from paper_2503_12450_gb300 import lazymar as lm
    lm.lib()
    torch.manual_seed(0)
    rows, T, D, H = 2 * cfg["batch"], cfg["T"], cfg["width"], cfg["heads"]
    N = synth.n_compute(cfg)
    dev = "cuda"
    if args.profile_case == "gemm_layers":
        # M: full blocks of both pathways, of the condition pathway alone, and
        # the recomputed tokens of both / of the condition pathway
        for M in (rows * T, rows * T // 2, rows * N, rows * N // 2):
            for n, k, epi in [(3 * D, D, lm.LAZYMAR_EPI_QKV), (D, D, lm.LAZYMAR_EPI_RESIDUAL),
                              (4 * D, D, lm.LAZYMAR_EPI_GELU), (D, 4 * D, lm.LAZYMAR_EPI_RESIDUAL)]:
                a = torch.randn(M, k, device=dev).bfloat16()
                w = (torch.randn(n, k, device=dev) * 0.05).bfloat16()
                b = torch.randn(n, device=dev).bfloat16()
                if epi == lm.LAZYMAR_EPI_QKV:
                    q = torch.empty(M, D, device=dev, dtype=torch.bfloat16)
                    kk, vv = torch.empty_like(q), torch.empty_like(q)
                    lm.lazymar_linear(lm.LAZYMAR_BF16, epi, a, w, b, M, n, k, q, D, kk, vv, None)
                elif epi == lm.LAZYMAR_EPI_RESIDUAL:
                    o = torch.zeros(M, n, device=dev)
                    lm.lazymar_linear(lm.LAZYMAR_BF16, epi, a, w, b, M, n, k, o, n)
                else:
                    o = torch.empty(M, n, device=dev, dtype=torch.bfloat16)
                    lm.lazymar_linear(lm.LAZYMAR_BF16, epi, a, w, b, M, n, k, o, n)
                torch.cuda.synchronize()
    elif args.profile_case == "launch_floor":
        # Per-launch device time of the recomputed-token GEMMs (both pathways,
        # M = rows x N; condition reuse, M = rows x N / 2) and of a minimal
        # kernel, each launched 20 times inside a CUDA graph: back to back (as
        # in the decode, consecutive launches overlap through programmatic
        # dependent launch) and with a CUDA event pair around every launch (how
        # the benchmark's per-kernel profile times them)
        R = 20

        def timed_graph(call):
            call()
            torch.cuda.synchronize()
            g1 = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g1, capture_error_mode="relaxed"):
                for _ in range(R):
                    call()
            evs = [(torch.cuda.Event(enable_timing=True, external=True),
                    torch.cuda.Event(enable_timing=True, external=True)) for _ in range(R)]
            g2 = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g2, capture_error_mode="relaxed"):
                for x, y in evs:
                    x.record()
                    call()
                    y.record()
            for _ in range(3):
                g1.replay()
                g2.replay()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            g1.replay()
            e1.record()
            torch.cuda.synchronize()
            back = e0.elapsed_time(e1) / R * 1e3
            g2.replay()
            torch.cuda.synchronize()
            return back, sum(x.elapsed_time(y) for x, y in evs) / R * 1e3

        out = {}
        zc = torch.randn(8, device=dev).bfloat16()
        zu, dl, gg = torch.randn_like(zc), torch.empty_like(zc), torch.empty_like(zc)
        b, e = timed_graph(lambda: lm.lazymar_cfg_combine(lm.LAZYMAR_BF16, lm.LAZYMAR_CFG_REFRESH, zc, zu, dl, GAMMA, 8,
                                                           None, gg))
        out["minimal kernel (guidance on 8 elements)"] = {"back_to_back_us": round(b, 2), "events_us": round(e, 2)}
        for M in (rows * N, rows * N // 2):
            for name, n, k, epi in [("qkv", 3 * D, D, lm.LAZYMAR_EPI_QKV), ("out", D, D, lm.LAZYMAR_EPI_RESIDUAL),
                                    ("fc1", 4 * D, D, lm.LAZYMAR_EPI_GELU), ("fc2", D, 4 * D, lm.LAZYMAR_EPI_RESIDUAL)]:
                a = torch.randn(M, k, device=dev).bfloat16()
                w = (torch.randn(n, k, device=dev) * 0.05).bfloat16()
                bias = torch.randn(n, device=dev).bfloat16()
                if epi == lm.LAZYMAR_EPI_QKV:
                    q = torch.empty(M, D, device=dev, dtype=torch.bfloat16)
                    kk, vv = torch.empty_like(q), torch.empty_like(q)
                    call = lambda: lm.lazymar_linear(lm.LAZYMAR_BF16, epi, a, w, bias, M, n, k, q, D, kk, vv, None)
                elif epi == lm.LAZYMAR_EPI_RESIDUAL:
                    o = torch.zeros(M, n, device=dev)
                    call = lambda: lm.lazymar_linear(lm.LAZYMAR_BF16, epi, a, w, bias, M, n, k, o, n)
                else:
                    o = torch.empty(M, n, device=dev, dtype=torch.bfloat16)
                    call = lambda: lm.lazymar_linear(lm.LAZYMAR_BF16, epi, a, w, bias, M, n, k, o, n)
                b, e = timed_graph(call)
                fl = 2.0 * M * n * k
                out["%s M=%d" % (name, M)] = {"back_to_back_us": round(b, 2), "events_us": round(e, 2),
                                              "tflops_back_to_back": round(fl / b / 1e6, 1),
                                              "tflops_events": round(fl / e / 1e6, 1)}
        print(json.dumps(out, indent=1), flush=True)
    elif args.profile_case == "steps":
        # one full and one cached step (both pathways) of the configuration,
        # every kernel launched eagerly
        B = cfg["batch"]
        W = synth.make_weights(cfg)
        h = lm.lazymar_create(dict(cfg, max_batch=B), W)
        lm.lazymar_set_graphs(h, False)
        lat, mask, labels = decode_inputs(cfg, 0)
        lat, mask, labels = (torch.from_numpy(x).cuda() for x in (lat, mask, labels))
        g = torch.empty((B, cfg["n_img"], D), device=dev, dtype=torch.bfloat16)
        lm.lazymar_full_step(h, lat[10], mask[10], labels, B, GAMMA, None, g)
        lm.lazymar_cached_step(h, lat[11], mask[11], labels, B, N, False, GAMMA, None, None, None, g)
        lm.lazymar_sync(h)
        h.close()
    elif args.profile_case == "head":
        B, n_img, td = cfg["batch"], cfg["n_img"], cfg["token_dim"]
        hc = synth.head_config(HEAD_FOR[cfg["name"]])
        n_new = 4
        hd = lm.lazymar_head_create(hc, D, td, synth.make_head_weights(hc, D, td), max_tokens=B * n_new)
        z = torch.randn(2 * B, n_img, D, device=dev).bfloat16()
        pos = torch.stack([torch.randperm(n_img, device=dev)[:n_new] for _ in range(B)]).int()
        noise = torch.randn(hc["n_steps"], B * n_new, td, device=dev)
        x = torch.empty(B * n_new, td, device=dev)
        lm.lazymar_head_sample(hd, z, B, n_img, pos, n_new, noise, GAMMA, 1.0, x)
        lm.lazymar_head_sync(hd)
        hd.close()
    else:
        for nq in (N, T):
            q = torch.randn(rows * nq, D, device=dev).bfloat16()
            k = torch.randn(rows * T, D, device=dev).bfloat16()
            v = torch.randn_like(k)
            o = torch.empty_like(q)
            lm.lazymar_attention(lm.LAZYMAR_BF16, q, k, v, o, rows, nq, T, H, D // H)
            torch.cuda.synchronize()
    lm.lazymar_device_check()
    print(json.dumps({"profile_case": args.profile_case, "config": cfg["name"], "ok": True}), flush=True)


HEAD_FOR = {"tiny": "tiny", "mar_b": "mar_b", "mar_l": "mar_l", "mar_h": "mar_h", "hires": "mar_l"}


def decoded_positions(mask_np):
    """Per decoding step, the image positions each pair decodes at that step
    ([B, n_new]; masked at step k and known at step k + 1, all remaining ones at
    the last step). The cosine schedule decodes the same count in every pair."""
    steps = mask_np.shape[0]
    out = []
    for k in range(steps):
        new = mask_np[k].astype(bool) & (~mask_np[k + 1].astype(bool) if k + 1 < steps else True)
        counts = new.sum(axis=1)
        assert np.all(counts == counts[0]), "pairs decode different token counts"
        out.append(np.stack([np.flatnonzero(r) for r in new]).astype(np.int32) if counts[0] else None)
    return out


def run_head_phase(args, cfg, lm, torch, mask_np, rank, stream, decode, timed, world, zbuf):
    """Decodes with the diffusion head after every step; returns the report
    (images/s of whole MAR sampling, head time and launches), or None."""
    B, n_img, D, td = cfg["batch"], cfg["n_img"], cfg["width"], cfg["token_dim"]
    hc = synth.head_config(HEAD_FOR[cfg["name"]])
    pos = decoded_positions(mask_np)
    max_new = max(p.shape[1] for p in pos if p is not None)
    HW = synth.make_head_weights(hc, D, td, seed=4 + rank_seed_offset(rank))
    hd = lm.lazymar_head_create(hc, D, td, HW, max_tokens=B * max_new, z_dtype=cfg["dtype"])
    pos_d = [None if p is None else torch.from_numpy(p).cuda() for p in pos]
    noise_d = [None if p is None else torch.from_numpy(synth.make_head_noise(hc["n_steps"], B * p.shape[1], td,
                                                                              seed=100 + k + rank_seed_offset(rank))).cuda()
               for k, p in enumerate(pos)]
    x_d = [None if p is None else torch.empty((B * p.shape[1], td), device="cuda") for p in pos]

    def head_step(k):
        # zbuf holds step k's features of both pathways (the step's z output)
        if pos_d[k] is not None:
            lm.lazymar_head_sample(hd, zbuf, B, n_img, pos_d[k], pos_d[k].shape[1], noise_d[k], GAMMA, 1.0, x_d[k],
                                   stream)

    decode(head_step=head_step)          # eager runs of every token count
    decode(head_step=head_step)          # graph captures
    lm.lazymar_head_sync(hd, stream)
    n_dec = max(1, min(args.steps, 2))
    n0, f0 = lm.lazymar_head_counters(hd)
    ms, _ = timed(lambda: decode(head_step=head_step), n_dec)
    n1, f1 = lm.lazymar_head_counters(hd)
    lm.lazymar_head_sync(hd, stream)
    # the head alone, same calls
    def heads_only():
        for k in range(cfg["steps"]):
            head_step(k)
    ms_head, _ = timed(heads_only, n_dec)
    hd.close()
    return {"value": job_images_per_s(world, B, n_dec, ms), "unit": "images/s",
            "ms_per_decode": ms / n_dec, "head_ms_per_decode": ms_head / n_dec,
            "head_launches_per_decode": int((n1 - n0) // n_dec),
            "head_tflops": (f1 - f0) / n_dec / (ms_head / n_dec / 1e3) / 1e12,
            "head": {"width": hc["width"], "depth": hc["depth"], "n_steps": hc["n_steps"], "tokens_per_step": "B x n_new(k)",
                     "note": "latents drawn by the head go to an output buffer; the next step's inputs stay the seeded ones"}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="mar_b")
    ap.add_argument("--ratio", type=float, default=None, help="recompute ratio (default: the config's)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-head", action="store_true", help="skip the decode with the diffusion head")
    ap.add_argument("--qkv-e4m3", action="store_true",
                    help="Q/K/V projection of the cached blocks on 8-bit (E4M3) tensor cores")
    ap.add_argument("--select", default="least_similar", choices=sorted(SELECT_RULES),
                    help="token-selection strategy of the cached steps (Table 3; default: LazyMAR's)")
    ap.add_argument("--profile-case", choices=["gemm_layers", "attention_layers", "head", "steps", "launch_floor"],
                    default=None,
                    help="run each kernel of a layer once at the configuration's shapes (for ncu) and exit")
    args = ap.parse_args()
    cfg = synth.config(args.config)
    if args.ratio is not None:
        cfg["ratio"] = args.ratio
    cfg["qkv_e4m3"] = 1 if args.qkv_e4m3 else 0
    if args.profile_case:
        profile_case(args, cfg)
    elif args.impl == "reference":
        import oracle as O
        plan = [O.plan(k, cfg["k0"], cfg["tau"], cfg["tau_cfg"]) for k in range(cfg["steps"])]
        run_reference(args, cfg, plan)
    else:
        run_ours(args, cfg)


if __name__ == "__main__":
    main()
