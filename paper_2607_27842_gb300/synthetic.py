"""Seeded synthetic workloads shaped like the paper's backbones.

Holds none of the method's arithmetic: model shapes, schedules, site lists,
random-init weights N(0, 0.02) and conditioning inputs only.  Both the CUDA
path and the CPU oracle consume what this module produces.

The five workloads (stand-ins for the paper's DiT-XL/2 on ImageNet-256,
FLUX.1-dev and Qwen-Image on DrawBench and HunyuanVideo-1.5 on VBench,
whose checkpoints and datasets are not used):
  tiny     4-block class-conditional DiT, fp32, 8x8x4 latent, 10 Euler steps
  dit_xl2  DiT-XL/2 shape, bf16, 32x32x4 latent, batch 8 (16 with guidance), 50 DDIM steps
  flux     19 dual + 38 single MMDiT blocks, 4096 image + 512 text tokens, 50 Euler steps
  qwen     60 dual MMDiT blocks, 4096 image + 256 text tokens, guidance, 50 Euler steps
  hunyuan  54 dual MMDiT blocks, 9x30x53 video tokens + 256 text, 3-D rotary, 50 Euler steps
"""

import dataclasses

import numpy as np

from .featfix import weight_spec

WEIGHT_STD = 0.02


@dataclasses.dataclass(frozen=True)
class ModelShape:
    name: str
    arch: str            # "dit" | "mmdit"
    n_dual: int          # DiT blocks, or MMDiT two-stream blocks
    n_single: int
    hidden: int
    heads: int
    head_dim: int
    mlp: int
    in_ch: int
    out_ch: int
    patch: int
    patch_t: int
    lat_f: int           # 0 for images
    lat_h: int
    lat_w: int
    txt_tokens: int
    n_classes: int
    batch: int           # latent samples
    cfg: bool            # model batch = [cond ; uncond]
    cfg_scale: float
    rope_dims: int
    dtype: str           # "f32" | "bf16"
    sampler: str         # "euler" | "ddim"

    @property
    def n_layers(self):
        return self.n_dual + self.n_single

    @property
    def batch_model(self):
        return self.batch * (2 if self.cfg else 1)

    @property
    def img_tokens(self):
        gf = self.lat_f // self.patch_t if self.lat_f > 0 else 1
        return gf * (self.lat_h // self.patch) * (self.lat_w // self.patch)

    @property
    def tokens(self):
        return self.img_tokens + self.txt_tokens

    @property
    def latent_dims(self):
        f = (self.lat_f,) if self.lat_f > 0 else ()
        return (self.batch, self.in_ch) + f + (self.lat_h, self.lat_w)


@dataclasses.dataclass(frozen=True)
class Workload:
    shape: ModelShape
    steps: int
    K: int
    refresh: tuple
    sites: tuple         # (step, layer) pairs


def refresh_every(steps, interval):
    """Fixed-interval full refresh: steps 0, interval, 2 * interval, ..."""
    return tuple(range(0, steps, interval))


def diagonal_sites(steps, L, refresh, n_sites):
    """A fixed, spread-out site set: site j at layer floor((j + 1/2) L / n) and
    at the non-refresh step of rank floor((j + 1/2) |M| / n)."""
    rs = set(refresh)
    M = [i for i in range(steps) if i not in rs]
    out = []
    for j in range(n_sites):
        layer = (2 * j + 1) * L // (2 * n_sites)
        step = M[(2 * j + 1) * len(M) // (2 * n_sites)]
        out.append((step, layer))
    return tuple(out)


def _shape(**kw):
    base = dict(n_single=0, patch_t=1, lat_f=0, txt_tokens=0, n_classes=0, cfg=False, cfg_scale=4.0,
                rope_dims=0)
    base.update(kw)
    return ModelShape(**base)


SHAPES = {
    "tiny": _shape(name="tiny", arch="dit", n_dual=4, hidden=128, heads=4, head_dim=32, mlp=512, in_ch=4,
                   out_ch=4, patch=1, lat_h=8, lat_w=8, n_classes=10, batch=1, dtype="f32", sampler="euler"),
    "dit_xl2": _shape(name="dit_xl2", arch="dit", n_dual=28, hidden=1152, heads=16, head_dim=72, mlp=4608,
                      in_ch=4, out_ch=8, patch=2, lat_h=32, lat_w=32, n_classes=1000, batch=8, cfg=True,
                      dtype="bf16", sampler="ddim"),
    "flux": _shape(name="flux", arch="mmdit", n_dual=19, n_single=38, hidden=3072, heads=24, head_dim=128,
                   mlp=12288, in_ch=16, out_ch=16, patch=2, lat_h=128, lat_w=128, txt_tokens=512, batch=1,
                   rope_dims=2, dtype="bf16", sampler="euler"),
    "qwen": _shape(name="qwen", arch="mmdit", n_dual=60, hidden=3072, heads=24, head_dim=128, mlp=12288, in_ch=16,
                   out_ch=16, patch=2, lat_h=128, lat_w=128, txt_tokens=256, batch=1, cfg=True, rope_dims=2,
                   dtype="bf16", sampler="euler"),
    "hunyuan": _shape(name="hunyuan", arch="mmdit", n_dual=54, hidden=2048, heads=16, head_dim=128, mlp=8192,
                      in_ch=16, out_ch=16, patch=2, patch_t=1, lat_f=9, lat_h=60, lat_w=106, txt_tokens=256,
                      batch=1, rope_dims=3, dtype="bf16", sampler="euler"),
}


# Variants of the large workloads with fewer image tokens, each at full depth
# and width with its base workload's schedule:
#   flux_512 / flux_768  FLUX at 512^2 / 768^2 images (latent 64x64 / 96x96,
#                        1024 / 2304 image tokens): the resolution sweep, and
#                        flux_512 the FLUX parity workload
#   qwen_512             Qwen-Image at 512^2 (1024 image tokens + 256 text,
#                        guidance batch 2)
#   hunyuan_3f           HunyuanVideo with 3 of the 9 latent frames
#                        (3x30x53 = 4770 video tokens + 256 text)
# The parity workloads are the sizes at which a whole float64 oracle
# trajectory finishes in about an hour on eight host cores.
VARIANTS = {"flux_512": ("flux", dict(lat_h=64, lat_w=64)), "flux_768": ("flux", dict(lat_h=96, lat_w=96)),
            "qwen_512": ("qwen", dict(lat_h=64, lat_w=64)), "hunyuan_3f": ("hunyuan", dict(lat_f=3))}


def workload(name):
    """The schedule of each workload: draft order, refresh interval, sites."""
    if name in VARIANTS:
        base_name, over = VARIANTS[name]
        base = workload(base_name)
        return Workload(reduced(base.shape, name=name, **over), base.steps, base.K, base.refresh, base.sites)
    s = SHAPES[name]
    if name == "tiny":
        return Workload(s, 10, 1, (0, 3, 6, 9), ((4, 2), (7, 1)))
    cfg = {"dit_xl2": (50, 2, 5, 8), "flux": (50, 1, 6, 12), "qwen": (50, 2, 5, 16), "hunyuan": (50, 1, 5, 12)}
    steps, K, every, n_sites = cfg[name]
    ref = refresh_every(steps, every)
    return Workload(s, steps, K, ref, diagonal_sites(steps, s.n_layers, ref, n_sites))


def reduced(shape, **overrides):
    """A smaller variant of a shape (fewer blocks, smaller latent, ...)."""
    return dataclasses.replace(shape, **overrides)


# ----------------------------------------------------------------------------
# tensors (torch: CPU or CUDA)
# ----------------------------------------------------------------------------

def torch_dtype(shape):
    import torch
    return torch.float32 if shape.dtype == "f32" else torch.bfloat16


def make_weights(shape, seed=0, device="cpu", names=None, to=None):
    """Random-init weights: every tensor N(0, 0.02) from its own seeded
    generator (seed * 1000003 + index), stored in the model dtype.
    ``names`` restricts generation to a subset (same values).  ``to`` moves
    each tensor to that device as soon as it is made (CPU-generated values
    on a GPU without a host copy of the whole model).  On the CPU the
    tensors are made by several threads, each from its own generator, so
    the values do not depend on the thread count.

    CPU draws are made in float64 and rounded to float32, then to the model
    dtype: torch's float64 normal sampler gives the same values on x86 and
    Arm hosts, its float32 sampler (vectorised differently per
    instruction set) does not."""
    import concurrent.futures
    import os
    import torch
    want = None if names is None else set(names)
    jobs = [(idx, name, dims) for idx, (name, dims) in enumerate(weight_spec(shape))
            if want is None or name in want]

    def one(job):
        idx, name, dims = job
        g = torch.Generator(device=device)
        g.manual_seed(seed * 1000003 + idx)
        if str(device) == "cpu":
            t = (torch.randn(dims, generator=g, dtype=torch.float64) * WEIGHT_STD).to(torch.float32)
        else:
            t = torch.randn(dims, generator=g, device=device, dtype=torch.float32) * WEIGHT_STD
        t = t.to(torch_dtype(shape)).contiguous()
        return name, (t if to is None else t.to(to))

    if str(device) == "cpu" and len(jobs) > 1:
        with concurrent.futures.ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
            return dict(ex.map(one, jobs))
    return dict(one(j) for j in jobs)


def make_cond(shape, seed=2, device="cpu"):
    """DiT: int32 labels [B_model] (uniform classes; the guidance half uses the
    null class n_classes).  MMDiT: float32 text tokens [B_model, N_txt, C]
    from N(0, 1) (the guidance half from seed + 1000)."""
    import torch
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    if shape.arch == "dit":
        lab = torch.randint(0, shape.n_classes, (shape.batch,), generator=g, dtype=torch.int64)
        if shape.cfg:
            lab = torch.cat([lab, torch.full((shape.batch,), shape.n_classes, dtype=torch.int64)])
        return lab.to(torch.int32).to(device)
    # float64 draws rounded to float32 (the same values on x86 and Arm hosts)
    txt = torch.randn((shape.batch, shape.txt_tokens, shape.hidden), generator=g, dtype=torch.float64).float()
    if shape.cfg:
        g2 = torch.Generator(device="cpu")
        g2.manual_seed(seed + 1000)
        unc = torch.randn((shape.batch, shape.txt_tokens, shape.hidden), generator=g2, dtype=torch.float64).float()
        txt = torch.cat([txt, unc])
    return txt.contiguous().to(device)


def to_numpy64(t):
    """float64 numpy copy of a torch tensor (bf16 values are exact in fp64)."""
    import torch
    return t.detach().to("cpu", torch.float64).numpy()


def oracle_weights(weights):
    return {k: to_numpy64(v) for k, v in weights.items()}


def oracle_cond(shape, cond):
    if shape.arch == "dit":
        return np.asarray(cond.cpu().numpy(), dtype=np.int64)
    return to_numpy64(cond)


def block_group(name):
    """Weights are grouped per block ("blk3.", "dual3.", "single7.");
    the embedding / conditioning / final-layer tensors form group ""."""
    head = name.split(".", 1)[0]
    if head.startswith(("blk", "dual", "single")):
        return head + "."
    return ""


class LazyOracleWeights:
    """float64 numpy weights made on first access, for models whose float64
    weights do not fit host memory (the MMDiT workloads hold 5-20 G
    parameters).  The values are those of ``make_weights(shape, seed)`` on the
    CPU generator, or of the torch tensors in ``source`` when given.

    Kept in memory: the non-block tensors, the most recently used block in
    float64, and model-dtype copies of blocks while their total stays under
    ``cache_bytes``.  Using block l starts a background thread preparing
    block l + 1, since the oracle walks the blocks in order."""

    def __init__(self, shape, seed=0, source=None, cache_bytes=0, prefetch=True):
        import threading
        self.shape, self.seed, self.source = shape, seed, source
        self.cache_bytes = cache_bytes
        self.prefetch = prefetch
        self.spec = dict(weight_spec(shape))
        self.groups = {}
        for name in self.spec:
            self.groups.setdefault(block_group(name), []).append(name)
        self.order = [g for g in self.groups if g]
        self.lock = threading.Lock()
        self.low = {}          # group -> {name: model-dtype torch tensor}
        self.low_bytes = 0
        self.cur = {}          # group -> {name: float64 array}; the global group and at most two blocks
        self.pending = {}      # group -> thread preparing it
        self.cur[""] = self._make64("")

    def _make_low(self, group):
        names = self.groups[group]
        if self.source is not None:
            return {n: self.source[n].detach().cpu() for n in names}
        return make_weights(self.shape, seed=self.seed, names=names)

    def _make64(self, group):
        with self.lock:
            low = self.low.get(group)
        if low is None:
            low = self._make_low(group)
            size = sum(t.numel() * t.element_size() for t in low.values())
            with self.lock:
                if group and self.low_bytes + size <= self.cache_bytes:
                    self.low[group] = low
                    self.low_bytes += size
        return {n: to_numpy64(t) for n, t in low.items()}

    def _prepare(self, group):
        import threading
        out = {}
        def work():
            out.update(self._make64(group))
        th = threading.Thread(target=work)
        th.result = out
        th.start()
        self.pending[group] = th

    def _group(self, group):
        if group in self.cur:
            return self.cur[group]
        th = self.pending.pop(group, None)
        if th is not None:
            th.join()
            data = th.result
        else:
            data = self._make64(group)
        for g in [g for g in self.cur if g]:
            del self.cur[g]
        self.cur[group] = data
        if self.prefetch:
            nxt = self.order[(self.order.index(group) + 1) % len(self.order)]
            for g in [g for g in self.pending if g != nxt]:
                self.pending.pop(g).join()
            if nxt not in self.pending and nxt != group:
                self._prepare(nxt)
        return data

    def __getitem__(self, name):
        if name not in self.spec:
            raise KeyError(name)
        return self._group(block_group(name))[name]

    def __contains__(self, name):
        return name in self.spec

    def keys(self):
        return self.spec.keys()

    def __iter__(self):
        return iter(self.spec)

    def __len__(self):
        return len(self.spec)
