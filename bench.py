"""Benchmark of the FeatFix cached sampling path on GB300.

One bench step = one whole cached sampling run (featfix_sample) of the
DiT-XL/2-shaped bf16 workload: 28 blocks, hidden 1152, 16 heads x 72,
MLP 4608, 32x32x4 latent with patch 2 (256 tokens), batch 8 doubled to 16 by
classifier-free guidance, 50 DDIM steps, order-2 Taylor draft, full refresh
every 5 steps, 8 fixed sites -- every row of the hot path (exact blocks,
drafts, paid checks with forwarding, final layer and sampler) runs each step.

Metric: denoising steps per second (50 per sampling run), whole job over all
ranks.  Inputs stay resident in HBM for ``value``; ``e2e`` repeats the
measurement through featfix_sample_host with pinned host buffers (labels in,
final latent out) inside the timed region.

Multi-GPU: replicas only (independent samples per GPU, no collective on the
data path); the barrier and max-over-ranks timing use torch.distributed.

``--impl reference`` times the CPU oracle on the host cores instead (a bounded
sample of the same workload, extrapolated by the plan's counts).
"""

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "cached-DiT denoise steps/s on 1 GB300; % of bf16 TC peak / HBM roofline"
UNIT = "denoise steps/s"
WORKLOAD = "dit_xl2"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default=WORKLOAD)
    p.add_argument("--mode", default="featfix", choices=["featfix", "verify", "exact_only", "vanilla"])
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--sweep", choices=["resolution"], default=None,
                   help="instead of the headline line: one line per FLUX resolution (512^2, 768^2, 1024^2) with "
                        "sampling rate and device memory")
    return p.parse_args()


def workload_config(wl):
    sh = wl.shape
    return {"workload": "%s: %d blocks, hidden %d, %d heads x %d, MLP %d, %d tokens, batch %d (model batch %d), "
                        "%d %s steps, order-%d draft, refresh every %d, %d sites"
                        % (sh.name, sh.n_layers, sh.hidden, sh.heads, sh.head_dim, sh.mlp, sh.tokens, sh.batch,
                           sh.batch_model, wl.steps, sh.sampler.upper(), wl.K, wl.refresh[1] - wl.refresh[0],
                           len(wl.sites)),
            "batch": sh.batch, "model_batch": sh.batch_model, "tokens": sh.tokens, "denoise_steps_per_sample": wl.steps,
            "draft_order": wl.K, "refresh_steps": len(wl.refresh), "sites": len(wl.sites),
            "weights": "random N(0,0.02), seeded",
            "l2": "no flush: inputs larger than L2 -- each sampling run streams %.2f GB of weights and %.2f GB of "
                  "refresh history through the 129 MB L2" % (weight_bytes(sh) / 1e9, history_bytes(wl) / 1e9)}


def weight_bytes(sh):
    from paper_2607_27842_gb300 import featfix as ff
    n = 0
    for _, dims in ff.weight_spec(sh):
        k = 1
        for d in dims:
            k *= d
        n += k
    return n * (2 if sh.dtype == "bf16" else 4)


def history_bytes(wl):
    sh = wl.shape
    return sh.n_layers * (wl.K + 1) * sh.batch_model * sh.tokens * sh.hidden * (2 if sh.dtype == "bf16" else 4)


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p.get("bf16_tflops_sustained", p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.rows = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.QUERY,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            f = [x.strip() for x in line.split(",")]
            if len(f) >= 9:
                self.rows.append(f)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        mhz = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in self.rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in self.rows for k in range(4) if r[5 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(mhz) if mhz else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.rows)}


# ----------------------------------------------------------------------------
# CPU oracle baseline (bounded sample, extrapolated)
# ----------------------------------------------------------------------------

def oracle_sample_time(wl, W64, cond64, budget_s=20.0):
    """Seconds of one whole sampling run of the oracle, extrapolated from
    timed pieces: one exact block, one drafted block, one paid check's
    discrepancy, the per-step conditioning/embedding/final layer/sampler."""
    import numpy as np
    import oracle
    sh = wl.shape
    L = sh.n_layers
    kind, keff = oracle.schedule.build_plan(wl.steps, L, wl.refresh, wl.K, wl.sites, "featfix")
    n_exact = sum(k != oracle.schedule.DRAFT for row in kind for k in row)
    n_draft = sum(k != oracle.schedule.EXACT for row in kind for k in row)   # sites form the draft too
    n_site = sum(k == oracle.schedule.SITE for row in kind for k in row)
    x = oracle.noise.initial_latent(1, sh).astype(np.float64)
    t0 = time.perf_counter()
    xm = np.concatenate([x, x]) if sh.cfg else x
    c = oracle.model.cond_vector(W64, 500.0, labels=cond64, batch=sh.batch_model)
    tok = oracle.model.embed_tokens(W64, sh, xm)
    out = oracle.model.final_layer(W64, sh, tok, c)
    x = oracle.sampler.step_update(sh, x, out, wl.steps, 0)
    t_step = time.perf_counter() - t0
    reps_e, t_exact = 0, 0.0
    while reps_e < 1 or (t_exact < budget_s * 0.6 and reps_e < 3):
        t0 = time.perf_counter()
        h = oracle.model.exact_block(W64, sh, reps_e % L, tok, c)
        t_exact += time.perf_counter() - t0
        reps_e += 1
    hist = [(5, h - tok), (0, (h - tok) * 0.5), (-5, (h - tok) * 0.25)]
    reps_d, t_draft = 0, 0.0
    while reps_d < 3:
        t0 = time.perf_counter()
        hd = oracle.draft.draft(tok, hist[:wl.K + 1], 7, wl.K)
        t_draft += time.perf_counter() - t0
        reps_d += 1
    t0 = time.perf_counter()
    oracle.featfix.rel_l1(hd, h)
    oracle.featfix.rel_l2(hd, h)
    t_log = time.perf_counter() - t0
    total = (wl.steps * t_step + n_exact * t_exact / reps_e + n_draft * t_draft / reps_d + n_site * t_log)
    sample = ("%d exact block(s), %d draft(s), 1 discrepancy, 1 embed+final+sampler step of the %s workload, timed "
              "and extrapolated by the plan's counts (%d exact, %d drafts, %d checks, %d steps)"
              % (reps_e, reps_d, sh.name, n_exact, n_draft, n_site, wl.steps))
    return total, sample


def cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        info = threadpool_info()
        if info:
            return max(i.get("num_threads", 1) for i in info)
    except Exception:
        pass
    return os.cpu_count() or 1


def oracle_inputs(wl, device="cpu"):
    from paper_2607_27842_gb300 import synthetic as syn
    w = syn.make_weights(wl.shape, seed=0, device=device)
    return syn.oracle_weights(w), syn.oracle_cond(wl.shape, syn.make_cond(wl.shape, seed=2))


def run_reference(args, wl, rank):
    if rank != 0:
        return
    W64, cond64 = oracle_inputs(wl)
    oracle_sample_time(wl, W64, cond64, budget_s=2.0)   # untimed: first-touch of the weights
    times = []
    sample = ""
    for _ in range(args.steps):
        t, sample = oracle_sample_time(wl, W64, cond64, budget_s=5.0)
        times.append(t)
    t = statistics.median(times)
    value = wl.steps / t
    cores = cpu_threads()
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(wl),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "note": "CPU oracle (float64 numpy) on the host cores, extrapolated per sampling run"}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------
# our arm
# ----------------------------------------------------------------------------

def slowest_rank(dist, durations, device):
    """Max over ranks of each timed duration: replicas run independently and
    the job ends with its slowest rank (no data is exchanged)."""
    if dist is None:
        return list(durations)
    import torch
    t = torch.tensor(list(durations), dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def job_rate(units_per_rank, world, seconds):
    """Whole-job throughput: the units every rank processed over the slowest
    rank's time (weak scaling: per-rank work fixed)."""
    return units_per_rank * world / seconds


def profile_traffic():
    """DRAM bytes per launch of the dominant kernel from the committed ncu
    summary, when it was taken on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", "gemm_tc_dit_xl2.md")
    src = b""
    for f in ("ff_gemm_tc.cu", "ff_tc.cuh", "ff_common.cuh"):
        with open(os.path.join(ROOT, "paper_2607_27842_gb300", "csrc", f), "rb") as fh:
            src += fh.read()
    digest = hashlib.sha256(src).hexdigest()[:16]
    try:
        txt = open(path).read()
    except Exception:
        return None
    tr, hsh = None, None
    for line in txt.splitlines():
        if line.startswith("traffic_bytes_per_launch:"):
            tr = float(line.split(":")[1])
        if line.startswith("kernel_source_sha256_16:"):
            hsh = line.split(":")[1].strip()
    return tr if hsh == digest else None


def run_sweep(args):
    """Latency and device memory of the FLUX-shaped cached sampler over image
    resolutions (the paper's resolution study): per resolution one JSON line
    with denoise steps/s, ms per sampling run, the bf16 weights, the
    library's own device memory (history ring, activations, workspaces) and
    the total device memory the run holds."""
    import torch
    from paper_2607_27842_gb300 import featfix as ff, synthetic as syn
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    for name, img in (("flux_512", 512), ("flux_768", 768), ("flux", 1024)):
        wl = syn.workload(name)
        sh = wl.shape
        torch.cuda.synchronize(dev)
        torch.cuda.empty_cache()
        free0 = torch.cuda.mem_get_info(dev)[0]
        weights = syn.make_weights(sh, seed=0, device=dev)
        cond = syn.make_cond(sh, seed=2, device=dev)
        lat = torch.empty(sh.latent_dims, dtype=torch.float32, device=dev)
        torch.cuda.synchronize(dev)
        free1 = torch.cuda.mem_get_info(dev)[0]
        ctx = ff.featfix_create(sh, weights, stream)
        ff.featfix_set_schedule(ctx, wl.steps, wl.refresh, wl.K, wl.sites, args.mode)
        for i in range(max(1, args.warmup)):
            ff.featfix_sample(ctx, 1000 + i, wl.steps, cond, lat)
        torch.cuda.synchronize(dev)
        free2 = torch.cuda.mem_get_info(dev)[0]
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for i in range(args.steps):
            ff.featfix_sample(ctx, 1 + i, wl.steps, cond, lat)
        ev1.record(stream)
        torch.cuda.synchronize(dev)
        ms = ev0.elapsed_time(ev1) / args.steps
        wbytes = sum(t.numel() * t.element_size() for t in weights.values())
        print(json.dumps({"sweep": "resolution", "workload": name, "image": "%dx%d" % (img, img),
                          "tokens": sh.tokens, "mode": args.mode, "value": wl.steps / (ms / 1e3), "unit": UNIT,
                          "ms_per_sample": ms, "weights_gb": wbytes / 1e9, "library_gb": (free1 - free2) / 1e9,
                          "device_gb": (free0 - free2) / 1e9, "steps": args.steps}), flush=True)
        ff.featfix_destroy(ctx)
        del weights, cond, lat


def main():
    args = parse()
    if args.sweep:
        run_sweep(args)
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    from paper_2607_27842_gb300 import synthetic as syn
    wl = syn.workload(args.workload)
    if args.impl == "reference":
        run_reference(args, wl, rank)
        return
    import torch
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    from paper_2607_27842_gb300 import featfix as ff

    sh = wl.shape
    weights = syn.make_weights(sh, seed=0, device=dev)
    cond = syn.make_cond(sh, seed=2 + 97 * rank, device=dev)
    lat = torch.empty(sh.latent_dims, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    ctx = ff.featfix_create(sh, weights, stream)
    ff.featfix_set_schedule(ctx, wl.steps, wl.refresh, wl.K, wl.sites, args.mode)

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for i in range(args.warmup):
        ff.featfix_sample(ctx, 1000 + i, wl.steps, cond, lat)
    barrier()

    # ---- timed region 1: the headline value, no instrumentation ----
    clocks = ClockSampler(local)
    clocks.start()
    l0 = ff.featfix_launch_count()
    barrier()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for i in range(args.steps):
        ff.featfix_sample(ctx, 1 + i, wl.steps, cond, lat)
    ev1.record(stream)
    barrier()
    clk = clocks.stop()
    launches = ff.featfix_launch_count() - l0
    ms = ev0.elapsed_time(ev1)
    logs, counters = ff.featfix_get_log(ctx)   # synchronises and checks the watchdog

    # ---- timed region 2: CUDA events around every launch of each kernel class ----
    timed_classes = ("gemm", "draft", "attention", "verify")
    for k in timed_classes:
        ff.featfix_kernel_timing(ctx, k, True)
    ff.featfix_sample(ctx, 999, wl.steps, cond, lat)      # untimed: rebuilds the graph with the event nodes
    for k in timed_classes:
        ff.featfix_kernel_timing(ctx, k, True)             # zero the counters (graph kept)
    barrier()
    for i in range(args.steps):
        ff.featfix_sample(ctx, 1 + i, wl.steps, cond, lat)
    barrier()
    kt = {k: ff.featfix_kernel_time(ctx, k) for k in timed_classes}
    for k in timed_classes:
        ff.featfix_kernel_timing(ctx, k, False)

    # ---- end to end through the host-buffer entry point ----
    cond_h = cond.cpu().pin_memory()
    out_h = torch.empty(sh.latent_dims, dtype=torch.float32).pin_memory()
    ff.featfix_sample_host(ctx, 7, wl.steps, cond_h, out_h)
    barrier()
    t0 = time.perf_counter()
    for i in range(args.steps):
        ff.featfix_sample_host(ctx, 11 + i, wl.steps, cond_h, out_h)
    barrier()
    e2e_s = time.perf_counter() - t0

    ms_max, e2e_max = slowest_rank(dist, [ms, e2e_s], dev)
    value = job_rate(args.steps * wl.steps, world, ms_max / 1e3)
    e2e = job_rate(args.steps * wl.steps, world, e2e_max)

    hbm, tf_burst, tf_sus, src = peaks()
    g_ms, g_n, g_work = kt["gemm"]
    achieved = (g_work / (g_ms / 1e3)) / 1e12 if g_ms > 0 else 0.0
    traffic = profile_traffic()
    d_ms, d_n, d_work = kt["draft"]
    draft_gbs = (d_work / (d_ms / 1e3)) / 1e9 if d_ms > 0 else 0.0
    a_ms, a_n, a_work = kt["attention"]
    v_ms, v_n, v_work = kt["verify"]
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_max / args.steps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic", "config": dict(workload_config(wl), mode=args.mode,
                                                            parallelism="replicas x%d" % world),
        "e2e": {"value": e2e, "unit": UNIT, "h2d_bytes_per_step": int(cond_h.numel() * cond_h.element_size()),
                "d2h_bytes_per_step": int(out_h.numel() * out_h.element_size())},
        "gpu_launches": int(launches),
        "roofline": {"bound": "tensor", "kernel": "k_gemm_tc (tcgen05, all linear layers of the path)",
                     "region": "second timed region of the same %d sampling runs with CUDA events on the context "
                               "stream around every launch of the kernel (inside the replayed graph)" % args.steps,
                     "achieved": achieved, "peak": tf_sus, "unit": "TFLOP/s", "frac": achieved / tf_sus,
                     "peak_kind": "bf16_tflops_sustained (%s)" % src, "traffic": traffic,
                     "launches": g_n, "ms_total": g_ms},
        "secondary": {
            "draft": {"bound": "hbm", "achieved": draft_gbs, "peak": hbm, "unit": "GB/s",
                      "frac": draft_gbs / hbm, "launches": d_n, "ms_total": d_ms},
            "attention": {"achieved_tflops": (a_work / (a_ms / 1e3)) / 1e12 if a_ms > 0 else 0.0,
                          "launches": a_n, "ms_total": a_ms},
            "verify": {"achieved_gbs": (v_work / (v_ms / 1e3)) / 1e9 if v_ms > 0 else 0.0, "launches": v_n,
                       "ms_total": v_ms},
            "counters": counters},
        "clocks": clk,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        try:
            W64 = syn.oracle_weights({k: v.cpu() for k, v in weights.items()})
            t, sample = oracle_sample_time(wl, W64, syn.oracle_cond(sh, cond.cpu()))
            line["cpu_baseline"] = {"value": wl.steps / t, "unit": UNIT, "cores": cpu_threads(), "kind": "oracle",
                                    "sample": sample}
        except Exception as e:  # reported, never fatal for the GPU number
            line["cpu_baseline"] = {"value": None, "unit": UNIT, "cores": cpu_threads(), "kind": "oracle",
                                    "sample": "failed: %s" % e}
    ff.featfix_destroy(ctx)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
