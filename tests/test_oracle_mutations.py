"""The oracle pins catch plausible mistakes: each case plants one mistake in a
temporary copy of ``oracle/`` (a dropped term, a wrong sign, index or
operand order, a swapped reading), runs the pins of
``tests/test_oracle_pins.py`` against the copy in a fresh interpreter, and
requires at least one of them to fail.  The unmodified copy passes.  The
mistakes live only in the temporary copy; nothing here touches a GPU."""

import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (file, text, replacement, pins to run (-k), what the mistake is)
MUTATIONS = [
    ("model.py", "return (x - mu) / np.sqrt(var + LN_EPS)", "return x / np.sqrt(var + LN_EPS)",
     "layer_norm", "LayerNorm without the mean"),
    ("model.py", "return x * (1.0 + scale[:, None, :]) + shift[:, None, :]",
     "return x * (1.0 + shift[:, None, :]) + scale[:, None, :]",
     "block", "shift and scale swapped"),
    ("model.py", "(x + 0.044715 * x ** 3)", "(x + 0.044715 * x ** 2)",
     "gelu", "GELU's cubic term squared"),
    ("model.py", "out[..., 1::2] = x1 * s + x2 * c", "out[..., 1::2] = -x1 * s + x2 * c",
     "rope", "rotary embedding with a sign error"),
    ("model.py", "scale = 1.0 / np.sqrt(d)", "scale = 1.0 / d",
     "attention", "attention scaled by 1/d"),
    ("model.py", "e = linear(silu(linear(s, W[\"t_fc1.w\"], W[\"t_fc1.b\"])), W[\"t_fc2.w\"], W[\"t_fc2.b\"])",
     "e = linear(linear(s, W[\"t_fc1.w\"], W[\"t_fc1.b\"]), W[\"t_fc2.w\"], W[\"t_fc2.b\"])",
     "cond_vector", "SiLU dropped from the time MLP"),
    ("model.py", "y = linear(modulate(layer_norm(tok), shift, scale), W[\"final.lin.w\"], W[\"final.lin.b\"])",
     "y = linear(modulate(tok, shift, scale), W[\"final.lin.w\"], W[\"final.lin.b\"])",
     "final_layer", "LayerNorm dropped from the final layer"),
    ("model.py", "return np.concatenate([np.asarray(txt, dtype=np.float64), img], axis=1)",
     "return np.concatenate([img, np.asarray(txt, dtype=np.float64)], axis=1)",
     "embed_tokens", "text tokens after the image tokens"),
    ("model.py", "u1 = u + g1[:, None, :] * linear(o, W[pre + \"proj.w\"], W[pre + \"proj.b\"])",
     "u1 = u + g2[:, None, :] * linear(o, W[pre + \"proj.w\"], W[pre + \"proj.b\"])",
     "dit_block", "the MLP gate on the attention branch"),
    ("model.py", "idx = np.indices(grid).reshape(len(grid), -1).T",
     "idx = np.indices(grid[::-1]).reshape(len(grid), -1).T[:, ::-1]",
     "image_positions or rope_table", "image positions in column-major order"),
    ("draft.py", "out = out + (t - s[0]) ** k / math.factorial(k) * Dk", "out = out + (t - s[0]) ** k * Dk",
     "draft or order", "factorial dropped from the Taylor series"),
    ("sampler.py", "return x + (sig[i + 1] - sig[i]) * v", "return x + (sig[i] - sig[i + 1]) * v",
     "euler", "Euler step with the wrong sign"),
    ("sampler.py", "return ou + scale * (oc - ou)", "return oc + scale * (oc - ou)",
     "guidance", "guidance around the conditional output"),
    ("sampler.py", "return euler_update(x, g[:, :shape.in_ch], steps, i)",
     "return euler_update(x, g[:, -shape.in_ch:], steps, i)",
     "step_update", "the velocity read from the wrong channels"),
    ("sampler.py", "return 1000.0 * euler_sigmas(steps)[i]", "return 1000.0 * euler_sigmas(steps)[i + 1]",
     "model_time", "the model time one step late"),
    ("schedule.py", "k_eff.append(min(K, r - 1))", "k_eff.append(min(K, r))",
     "plan or schedule", "draft order not limited by the refreshes seen"),
    ("model.py", "p /= p.sum(axis=-1, keepdims=True)", "p /= p.sum(axis=-2, keepdims=True)",
     "attention", "softmax normalised over the queries"),
    ("model.py", "return np.concatenate([np.cos(args), np.sin(args)])",
     "return np.concatenate([np.sin(args), np.cos(args)])",
     "sinusoid", "timestep features in [sin | cos] order"),
    ("model.py", "rows, cols = np.meshgrid(np.arange(gh), np.arange(gw), indexing=\"ij\")",
     "cols, rows = np.meshgrid(np.arange(gh), np.arange(gw), indexing=\"ij\")",
     "sincos", "position rows and columns swapped"),
    ("model.py", "qkv_t = linear(modulate(layer_norm(txt), mt[0], mt[1]), W[pre + \"txt_qkv.w\"], W[pre + \"txt_qkv.b\"])",
     "qkv_t = linear(modulate(layer_norm(txt), mi[0], mi[1]), W[pre + \"txt_qkv.w\"], W[pre + \"txt_qkv.b\"])",
     "dual_block", "the text stream modulated by the image stream's vectors"),
    ("model.py", "out = linear(np.concatenate([o, gelu_tanh(mlp)], axis=-1), W[pre + \"lin2.w\"], W[pre + \"lin2.b\"])",
     "out = linear(np.concatenate([gelu_tanh(mlp), o], axis=-1), W[pre + \"lin2.w\"], W[pre + \"lin2.b\"])",
     "single_block", "the single block's [attention | MLP] order reversed"),
    ("noise.py", "z = (z ^ (z >> np.uint64(27))) * M2", "z = (z ^ (z >> np.uint64(28))) * M2",
     "splitmix", "a SplitMix64 shift off by one"),
    ("schedule.py", "        if i in rs:\n            raise ScheduleError(\"site on a refresh step\")\n", "",
     "schedule_rules", "a site on a refresh step accepted"),
    ("draft.py", "table = [(table[j] - table[j + 1]) / (s[j] - s[j + m]) for j in range(n - m)]",
     "table = [(table[j] - table[j + 1]) / (s[j] - s[j + 1]) for j in range(n - m)]",
     "draft or order or taylor", "divided differences over the wrong node span"),
    ("draft.py", "D[k] = D[k] + math.factorial(k) * coef[k] * dd[m]", "D[k] = D[k] + coef[k] * dd[m]",
     "draft or order or taylor", "derivative estimates without k!"),
    ("featfix.py", "hist[l].insert(0, (i, h - u))", "hist[l].insert(0, (i, h))",
     "identity_blocks", "the block outputs forecast instead of their increments"),
    ("featfix.py", "                        h = hd\n", "                        h = hf\n",
     "verify", "the Verify arm forwarding the exact output"),
    ("featfix.py", "return float(np.abs(hd - hf).sum() / (np.abs(hf).sum() + EPS))",
     "return float(np.abs(hd - hf).sum() / (np.abs(hd).sum() + EPS))",
     "discrepancy", "Eq. 4 normalised by the draft"),
]


def _copy(tmp):
    """The pins and what they import: tests (with the golden texts), the
    oracle, and the input generator of the package."""
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(tmp, "oracle"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    os.makedirs(os.path.join(tmp, "tests", "golden"))
    for f in ("__init__.py", "conftest.py", "test_oracle_pins.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), os.path.join(tmp, "tests", f))
    for f in os.listdir(os.path.join(ROOT, "tests", "golden")):
        if f.endswith(".txt"):
            shutil.copy(os.path.join(ROOT, "tests", "golden", f), os.path.join(tmp, "tests", "golden", f))
    pkg = os.path.join(tmp, "paper_2607_27842_gb300")
    os.makedirs(pkg)
    # the pins need the seeded generators and the weight names of the binding
    # module (its library is never loaded)
    with open(os.path.join(pkg, "__init__.py"), "w") as f:
        f.write("")
    for f in ("synthetic.py", "featfix.py"):
        shutil.copy(os.path.join(ROOT, "paper_2607_27842_gb300", f), os.path.join(pkg, f))


def _run_pins(tmp, select):
    env = dict(os.environ, PYTHONDONTWRITEBYTECODE="1", OMP_NUM_THREADS="2", OPENBLAS_NUM_THREADS="2")
    cmd = [sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider", "-m", "not gpu",
           os.path.join("tests", "test_oracle_pins.py")]
    if select:
        cmd += ["-k", select]
    return subprocess.run(cmd, cwd=tmp, env=env, capture_output=True, text=True, timeout=600)


def _mutant_run(case, tmp):
    fname, old, new, select, what = case
    _copy(tmp)
    path = os.path.join(tmp, "oracle", fname)
    with open(path) as f:
        src = f.read()
    if src.count(old) != 1:
        return None, "the text to change must occur once in oracle/%s" % fname
    with open(path, "w") as f:
        f.write(src.replace(old, new))
    r = _run_pins(tmp, select)
    return r.returncode, r.stdout + r.stderr


@pytest.fixture(scope="module")
def runs(tmp_path_factory):
    """The unmodified copy and every mutant, run four at a time."""
    import concurrent.futures
    cases = [None] + MUTATIONS
    dirs = [str(tmp_path_factory.mktemp("oracle_copy")) for _ in cases]

    def one(k):
        if cases[k] is None:
            _copy(dirs[k])
            r = _run_pins(dirs[k], None)
            return r.returncode, r.stdout + r.stderr
        return _mutant_run(cases[k], dirs[k])

    with concurrent.futures.ThreadPoolExecutor(max_workers=4) as ex:
        res = list(ex.map(one, range(len(cases))))
    return {"pristine": res[0], **{m[4]: res[k + 1] for k, m in enumerate(MUTATIONS)}}


def test_unmodified_copy_passes(runs):
    rc, out = runs["pristine"]
    assert rc == 0, out[-6000:]


@pytest.mark.parametrize("what", [m[4] for m in MUTATIONS])
def test_planted_mistake_fails_a_pin(runs, what):
    rc, out = runs[what]
    assert rc is not None, out
    assert "no tests ran" not in out, out[-2000:]
    assert rc == 1, "%s: no pin failed\n%s" % (what, out[-3000:])
