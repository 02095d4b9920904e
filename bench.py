"""Benchmark of the FeatFix cached sampling path on GB300.

One bench step = one whole cached sampling run (featfix_sample) of the
HunyuanVideo-1.5-shaped bf16 workload, the largest of the five: 54 dual-stream
MMDiT blocks, hidden 2048, 16 heads x 128, MLP 8192, 3-D rotary embedding,
9 x 30 x 53 video tokens + 256 text tokens (14566), batch 1, 50 Euler steps,
order-1 Taylor draft, full refresh every 5 steps, 12 fixed sites -- every row
of the hot path (exact blocks, drafts, paid checks with forwarding, final
layer and sampler) runs each step.  ``--workload dit_xl2`` (and flux, qwen)
bench the other shapes.

Metric: denoising steps per second (50 per sampling run), whole job over all
ranks.  Inputs stay resident in HBM for ``value``; ``e2e`` repeats the
measurement through featfix_sample_host with pinned host buffers
(conditioning in, final latent out) inside the timed region.

Rooflines: a second timed region of the same sampling runs brackets every
launch of each kernel class (tensor-core GEMM, attention, draft, paid check)
with CUDA events and divides its algorithmic work by the summed time;
``roofline`` is the class with the most time, ``rooflines`` all four.

Multi-GPU: replicas only (independent samples per GPU, no collective on the
data path); the barrier and max-over-ranks timing use torch.distributed.

Beside the cached rate the line carries the all-exact (vanilla) rate on the
same GPU (``vanilla``; ``--no-vanilla`` skips it) and the paper's own
latencies for the backbone the workload is shaped like (``paper``: context,
hardware not stated).

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
WORKLOAD = "hunyuan"
NOMINAL_TFLOPS = 2250.0    # GB300 dense bf16 datasheet figure
NOMINAL_GBS = 8000.0       # HBM3e, about 8 TB/s


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default=WORKLOAD)
    p.add_argument("--mode", default="featfix", choices=["featfix", "verify", "exact_only", "vanilla"])
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-vanilla", action="store_true",
                   help="skip the all-exact (vanilla) runs measured beside the cached rate")
    p.add_argument("--stepwise", action="store_true",
                   help="also time the same runs driven one featfix_step call per denoising step (no whole-run graph)")
    p.add_argument("--cpu-leg", type=int, default=0, help=argparse.SUPPRESS)   # internal: oracle timing process
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

FIT_ABOVE_FLOPS = 0.5e12   # exact blocks above this are timed on token-reduced copies


def token_reduced_shapes(sh):
    """Two copies of a shape with about 1/8 and 1/4 of its image tokens
    (fewer video frames, or fewer patch rows of an image); same weights."""
    from paper_2607_27842_gb300 import synthetic as syn
    if sh.lat_f > 0:
        f1 = max(sh.patch_t, (sh.lat_f // 8) // sh.patch_t * sh.patch_t)
        return [syn.reduced(sh, lat_f=f1), syn.reduced(sh, lat_f=2 * f1)]
    h1 = max(sh.patch, (sh.lat_h // 8) // sh.patch * sh.patch)
    return [syn.reduced(sh, lat_h=h1), syn.reduced(sh, lat_h=2 * h1)]


def oracle_sample_time(wl, W, cond64, budget_s=20.0):
    """Seconds of one whole sampling run of the oracle, extrapolated from
    timed pieces by the plan's counts: the per-step conditioning, embedding,
    final layer and sampler update; one exact block; one drafted block; one
    paid check's discrepancy.  An exact block of more than 0.5 TFLOP is timed
    on two copies of the workload with about 1/8 and 1/4 of its tokens and
    extrapolated as a*T + b*T^2 (the projections grow linearly, attention
    quadratically with the token count T)."""
    import numpy as np
    import oracle
    sh = wl.shape
    L = sh.n_layers
    kind, _ = oracle.schedule.build_plan(wl.steps, L, wl.refresh, wl.K, wl.sites, "featfix")
    n_exact = sum(k != oracle.schedule.DRAFT for row in kind for k in row)
    n_draft = sum(k != oracle.schedule.EXACT for row in kind for k in row)   # sites form the draft too
    n_site = sum(k == oracle.schedule.SITE for row in kind for k in row)
    txt = cond64 if sh.arch == "mmdit" else None
    labels = cond64 if sh.arch == "dit" else None
    x = oracle.noise.initial_latent(1, sh).astype(np.float64)
    t0 = time.perf_counter()
    xm = np.concatenate([x, x]) if sh.cfg else x
    c = oracle.model.cond_vector(W, 500.0, labels=labels, batch=sh.batch_model)
    tok = oracle.model.embed_tokens(W, sh, xm, txt=txt)
    out = oracle.model.final_layer(W, sh, tok, c)
    oracle.sampler.step_update(sh, x, out, wl.steps, 0)
    t_step = time.perf_counter() - t0

    pre = oracle.model.block_prefix(sh, 0)
    for name in [n for n in W.keys() if n.startswith(pre)]:
        W[name]                      # make the timed block's weights before timing it

    def exact_once(shape):
        u = np.ascontiguousarray(np.resize(tok, (sh.batch_model, shape.tokens, sh.hidden)))
        t1 = time.perf_counter()
        h = oracle.model.exact_block(W, shape, 0, u, c)
        return time.perf_counter() - t1, h

    if oracle.flops.block_flops(sh, 0) <= FIT_ABOVE_FLOPS:
        reps, t_sum = 0, 0.0
        while reps < 1 or (t_sum < budget_s * 0.6 and reps < 3):
            dt, h = exact_once(sh)
            t_sum += dt
            reps += 1
        t_exact = t_sum / reps
        inc = h - tok
        how = "%d exact block(s) at full size" % reps
    else:
        small = token_reduced_shapes(sh)
        (d1, _), (d2, _) = exact_once(small[0]), exact_once(small[1])
        T1, T2, T = small[0].tokens, small[1].tokens, sh.tokens
        b = (d2 / T2 - d1 / T1) / (T2 - T1)
        a = d1 / T1 - b * T1
        if b < 0:
            a, b = d2 / T2, 0.0
        t_exact = a * T + b * T * T
        inc = tok * 0.125
        how = ("2 exact blocks at %d and %d of the %d tokens, extrapolated as a*T + b*T^2 (%.2f s / %.2f s timed, "
               "%.1f s at full size)" % (T1, T2, T, d1, d2, t_exact))
    hist = [(5, inc), (0, inc * 0.5), (-5, inc * 0.25)]
    t_draft = 0.0
    for _ in range(2):
        t1 = time.perf_counter()
        hd = oracle.draft.draft(tok, hist[:wl.K + 1], 7, wl.K)
        t_draft += (time.perf_counter() - t1) / 2
    t1 = time.perf_counter()
    oracle.featfix.rel_l1(hd, tok)
    oracle.featfix.rel_l2(hd, tok)
    t_log = time.perf_counter() - t1
    total = wl.steps * t_step + n_exact * t_exact + n_draft * t_draft + n_site * t_log
    sample = ("%s, 2 drafts, 1 discrepancy and 1 conditioning+embed+final+sampler step of the %s workload, "
              "extrapolated by the plan's counts (%d exact blocks, %d drafts, %d checks, %d steps)"
              % (how, sh.name, n_exact, n_draft, n_site, wl.steps))
    return total, sample


def lazy_oracle_inputs(wl, source=None):
    """Float64 oracle weights made block by block on access (the large
    workloads' float64 weights do not fit host memory) and the conditioning."""
    from paper_2607_27842_gb300 import synthetic as syn
    W = syn.LazyOracleWeights(wl.shape, seed=0, source=source, prefetch=False)
    return W, syn.oracle_cond(wl.shape, syn.make_cond(wl.shape, seed=2))


def cpu_leg(args, wl):
    """Internal: time the oracle sample in this process (the thread count is
    fixed by the parent through the BLAS environment) and print one JSON line."""
    W, cond64 = lazy_oracle_inputs(wl)
    t, sample = oracle_sample_time(wl, W, cond64, budget_s=10.0)
    print(json.dumps({"seconds": t, "sample": sample, "threads": args.cpu_leg}), flush=True)


def start_cpu_leg(wl, threads):
    """The oracle timing as a separate interpreter (not forked from a process
    that holds a CUDA context) with its BLAS limited to `threads` threads."""
    env = dict(os.environ)
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = str(threads)
    env["CUDA_VISIBLE_DEVICES"] = ""
    return subprocess.Popen([sys.executable, os.path.abspath(__file__), "--workload", wl.shape.name,
                             "--cpu-leg", str(threads)], stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True,
                            env=env, cwd=ROOT)


def finish_cpu_leg(proc, wl, timeout_s=600):
    try:
        out, err = proc.communicate(timeout=timeout_s)
        rec = json.loads(out.strip().splitlines()[-1])
        return {"value": wl.steps / rec["seconds"], "unit": UNIT, "cores": rec["threads"], "kind": "oracle",
                "sample": rec["sample"]}
    except Exception as e:  # reported, never fatal for the GPU number
        proc.kill()
        return {"value": None, "unit": UNIT, "cores": None, "kind": "oracle", "sample": "failed: %s" % e}


def all_cores():
    return os.cpu_count() or 1


def host_cpu():
    """The host the oracle legs run on: logical CPUs and the CPU model."""
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                model = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    import platform
    return {"nproc": all_cores(), "cpu": model or platform.processor() or None, "machine": platform.machine()}


# The paper's own latencies for the backbone each workload is shaped like
# (real checkpoints, prompts and resolutions; hardware, precision and batch
# not stated): context beside the measured rates, not a target.
PAPER = {
    "flux": {"backbone": "FLUX.1-dev, DrawBench200", "source": "Table 1", "vanilla_s": 23.93,
             "featfix_s": [7.57, 4.76, 3.57], "speedup": [3.16, 5.03, 6.70]},
    "qwen": {"backbone": "Qwen-Image, DrawBench200", "source": "Table 4", "vanilla_s": 22.59,
             "featfix_s": [15.08, 10.40], "speedup": [1.50, 2.17]},
    "hunyuan": {"backbone": "HunyuanVideo-1.5, 65 frames", "source": "Table 3", "vanilla_s": 772.60,
                "featfix_s": [483.50, 415.10, 338.40], "speedup": [1.60, 1.86, 2.28]},
    "dit_xl2": {"backbone": "DiT-XL/2, ImageNet-256", "source": "Table 5", "vanilla_s": 1.52,
                "featfix_s": [0.45], "speedup": [3.38]},
}


def paper_context(wl):
    base = wl.shape.name.split("_")[0] if wl.shape.name not in PAPER else wl.shape.name
    rec = PAPER.get(base)
    return dict(rec, hardware="not stated") if rec else None


def run_reference(args, wl, rank):
    if rank != 0:
        return
    W, cond64 = lazy_oracle_inputs(wl)
    for _ in range(args.warmup):
        oracle_sample_time(wl, W, cond64, budget_s=2.0)
    times = []
    sample = ""
    for _ in range(args.steps):
        t, sample = oracle_sample_time(wl, W, cond64, budget_s=2.0)
        times.append(t)
    t = statistics.median(times)
    value = wl.steps / t
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": dict(workload_config(wl), mode=args.mode, parallelism="replicas x%d" % args.gpus),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": all_cores(), "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "note": "CPU oracle (float64 numpy) on the host cores; each step times a bounded sample of one "
                    "sampling run and extrapolates it"}
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


KERNELS = {   # kernel class -> (kernel, bound, the sources its profile summary was taken on)
    "gemm": ("k_gemm_tc / k_gemm_tc2 (tcgen05, all linear layers of the path)", "tensor",
             ("ff_gemm_tc.cu", "ff_tc.cuh", "ff_common.cuh")),
    "attention": ("k_attn_tc (tcgen05 flash attention)", "tensor", ("ff_attention_tc.cu", "ff_tc.cuh", "ff_common.cuh")),
    "draft": ("k_draft", "hbm", ("ff_elementwise.cu", "ff_common.cuh")),
    "verify": ("k_verify (paid check, forwarding)", "hbm", ("ff_elementwise.cu", "ff_common.cuh")),
}


def source_digest(files):
    src = b""
    for f in files:
        with open(os.path.join(ROOT, "paper_2607_27842_gb300", "csrc", f), "rb") as fh:
            src += fh.read()
    return hashlib.sha256(src).hexdigest()[:16]


def profile_traffic(kclass, workload):
    """DRAM bytes per launch of a kernel class on a workload from its committed
    ncu summary (profiles/<class>_<workload>.md), when that summary was taken
    on the current kernel sources (else None)."""
    path = os.path.join(ROOT, "profiles", "%s_%s.md" % (kclass, workload))
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
    return tr if hsh == source_digest(KERNELS[kclass][2]) else None


def roofline(kclass, kt, wl, steps):
    """Achieved rate of a kernel class over the second timed region against
    the measured peak (sustained bf16 for tensor work: the kernels run inside a
    seconds-long step) and against the nominal GB300 figures."""
    hbm, tf_burst, tf_sus, src = peaks()
    ms, n, work = kt[kclass]
    kernel, bound, _ = KERNELS[kclass]
    if bound == "tensor":
        ach = (work / (ms / 1e3)) / 1e12 if ms > 0 else 0.0
        r = {"bound": "tensor", "kernel": kernel, "achieved": ach, "peak": tf_sus, "unit": "TFLOP/s",
             "frac": ach / tf_sus, "peak_kind": "bf16_tflops_sustained (%s)" % src,
             "frac_of_burst_peak": ach / tf_burst, "peak_nominal": NOMINAL_TFLOPS,
             "frac_vs_nominal": ach / NOMINAL_TFLOPS}
    else:
        ach = (work / (ms / 1e3)) / 1e9 if ms > 0 else 0.0
        r = {"bound": "hbm", "kernel": kernel, "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm,
             "peak_kind": "hbm_gbs copy (%s)" % src, "peak_nominal": NOMINAL_GBS, "frac_vs_nominal": ach / NOMINAL_GBS}
    r.update({"traffic": profile_traffic(kclass, wl.shape.name), "launches": n, "ms_total": ms,
              "work_per_launch": work / n if n else 0.0,
              "work_unit": "FLOP (2*M*N*K, 4*B*H*N^2*d)" if bound == "tensor" else "bytes ((K_eff+3)*E*b, ...)",
              "region": "second timed region: the same %d sampling runs with CUDA events on the context stream "
                        "around every launch of the class (event nodes inside the replayed graph)" % steps})
    return r


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
    from paper_2607_27842_gb300 import synthetic as syn
    wl = syn.workload(args.workload)
    if args.cpu_leg:
        cpu_leg(args, wl)
        return
    if args.sweep:
        run_sweep(args)
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, wl, rank)
        return
    want_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    # the one-core oracle leg runs beside the GPU work (one host core of many)
    leg1 = start_cpu_leg(wl, 1) if want_cpu else None
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
    timed_classes = tuple(KERNELS)
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

    # ---- optional: the same runs driven one featfix_step call per denoising step ----
    step_ms = None
    if args.stepwise:
        x = torch.empty(sh.latent_dims, dtype=torch.float32, device=dev)
        for i in range(args.warmup):
            x.normal_()
            for t in range(wl.steps):
                ff.featfix_step(ctx, x, t, cond)
        barrier()
        ev2, ev3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev2.record(stream)
        for i in range(args.steps):
            x.normal_()
            for t in range(wl.steps):
                ff.featfix_step(ctx, x, t, cond)
        ev3.record(stream)
        barrier()
        step_ms = ev2.elapsed_time(ev3)

    # ---- the all-exact (vanilla) rate on the same GPU, weights and inputs ----
    vanilla = None
    if args.mode != "vanilla" and not args.no_vanilla and world == 1:
        try:
            nv = 2
            ff.featfix_set_schedule(ctx, wl.steps, wl.refresh, wl.K, wl.sites, "vanilla")
            ff.featfix_sample(ctx, 2000, wl.steps, cond, lat)   # untimed: builds the vanilla graph
            barrier()
            ev4, ev5 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            ev4.record(stream)
            for i in range(nv):
                ff.featfix_sample(ctx, 2001 + i, wl.steps, cond, lat)
            ev5.record(stream)
            barrier()
            v_rate = job_rate(nv * wl.steps, 1, ev4.elapsed_time(ev5) / 1e3)
            vanilla = {"value": v_rate, "unit": UNIT, "runs": nv, "cached_over_vanilla": None,
                       "how": "the same context rescheduled with every block exact at every step, one untimed "
                              "run, then %d runs timed with CUDA events" % nv}
        except Exception as e:  # reported, never fatal for the cached number
            vanilla = {"value": None, "unit": UNIT, "error": str(e)}

    ms_max, e2e_max = slowest_rank(dist, [ms, e2e_s], dev)
    value = job_rate(args.steps * wl.steps, world, ms_max / 1e3)
    e2e = job_rate(args.steps * wl.steps, world, e2e_max)

    rl = {k: roofline(k, kt, wl, args.steps) for k in timed_classes}
    dominant = max(("gemm", "attention"), key=lambda k: kt[k][0])
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_max / args.steps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if sh.dtype == "bf16" else "f32", "data": "synthetic",
        "config": dict(workload_config(wl), mode=args.mode, parallelism="replicas x%d" % world),
        "e2e": {"value": e2e, "unit": UNIT, "h2d_bytes_per_step": int(cond_h.numel() * cond_h.element_size()),
                "d2h_bytes_per_step": int(out_h.numel() * out_h.element_size())},
        "gpu_launches": int(launches),
        "roofline": dict(rl[dominant], kclass=dominant),
        "rooflines": rl,
        "counters": counters,
        "clocks": clk,
    }
    if vanilla is not None:
        if vanilla.get("value"):
            vanilla["cached_over_vanilla"] = value / vanilla["value"]
        line["vanilla"] = vanilla
    paper = paper_context(wl)
    if paper is not None:
        line["paper"] = paper
    if step_ms is not None:
        line["stepwise"] = {"value": job_rate(args.steps * wl.steps, 1, step_ms / 1e3), "unit": UNIT,
                            "how": "one featfix_step call per denoising step from the host (no whole-run CUDA "
                                   "graph), the same runs, CUDA events (latent re-initialised with normal_ per run)"}
    if want_cpu:
        one_core = finish_cpu_leg(leg1, wl)
        line["cpu_baseline"] = finish_cpu_leg(start_cpu_leg(wl, all_cores()), wl)
        line["cpu_baseline_1core"] = one_core
        line["cpu_baseline"]["host"] = host_cpu()
    ff.featfix_destroy(ctx)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
