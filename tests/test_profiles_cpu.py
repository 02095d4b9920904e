"""The committed ncu summaries: short text, every profiler command given in
full with the clocks left alone, and the traffic records the bench reads
well formed."""

import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROFILES = sorted(glob.glob(os.path.join(ROOT, "profiles", "*")))


def test_profiles_exist():
    assert PROFILES, "no ncu summaries committed"


@pytest.mark.parametrize("path", PROFILES, ids=[os.path.basename(p) for p in PROFILES])
def test_summary_is_short_text(path):
    assert os.path.splitext(path)[1] in (".md", ".txt")
    assert os.path.getsize(path) < 16 * 1024
    with open(path, "rb") as f:
        raw = f.read()
    raw.decode("utf-8")  # text, not a report file


def _ncu_commands(txt):
    """The ncu command lines of a summary, continuation lines joined."""
    cmds = []
    for block in re.findall(r"```\n(.*?)```", txt, flags=re.S):
        joined = block.replace("\\\n", " ")
        cmds += [line.strip() for line in joined.splitlines() if line.strip().startswith("ncu ")]
    return cmds


@pytest.mark.parametrize("path", PROFILES, ids=[os.path.basename(p) for p in PROFILES])
def test_commands_leave_clocks_alone(path):
    with open(path) as f:
        txt = f.read()
    cmds = _ncu_commands(txt)
    if not cmds:
        # a summary that reuses another capture names it
        assert re.search(r"capture of `profiles/\w+\.md`", txt), path
        return
    for c in cmds:
        assert "--clock-control none" in c, c
        # one kernel and a bounded launch count, or a single-metric launch list
        assert ("-k " in c and "-c " in c) or "--metrics gpu__time_duration.sum" in c, c


def test_traffic_records_parse():
    """Every summary the bench reads a traffic figure from carries both the
    per-launch bytes and the source digest it was taken on."""
    import bench
    from paper_2607_27842_gb300 import synthetic as syn
    seen = 0
    for kclass in bench.KERNELS:
        for wl in list(syn.SHAPES) + list(syn.VARIANTS):
            path = os.path.join(ROOT, "profiles", "%s_%s.md" % (kclass, wl))
            if not os.path.exists(path):
                continue
            with open(path) as f:
                lines = f.read().splitlines()
            tr = [l for l in lines if l.startswith("traffic_bytes_per_launch:")]
            dg = [l for l in lines if l.startswith("kernel_source_sha256_16:")]
            assert len(tr) == 1 and len(dg) == 1, path
            assert float(tr[0].split(":")[1]) > 0
            assert re.fullmatch(r"[0-9a-f]{16}", dg[0].split(":")[1].strip())
            seen += 1
    assert seen >= 2
