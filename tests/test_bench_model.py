"""CPU tests of bench.py's measurement model: the algorithmic bytes per
parameter of every kernel it times, and the rule that ties the committed ncu
traffic figures to the kernel source they were taken on."""
import os
import shutil
import sys

import pytest

from conftest import ROOT

sys.path.insert(0, ROOT)
import bench  # noqa: E402


# (optimizer, g bytes, copy bytes, variant) -> per-kernel bytes per parameter.
# Two-pass LAMB: pass 1 reads g, m, v, w and writes m, v; pass 2 reads m, v, w
# and writes w and the copy.  LARS has no v.  N-LAMB's pass 2 also reads g
# (the Nesterov term).  The skip mode moves the m, v writes to pass 2, which
# then re-reads g.
CASES = [
    ("lamb", 2, 2, "plain", [22, 18], 40, 28),     # BERT-large
    ("lamb", 4, 0, "plain", [24, 16], 40, 28),     # fp32 LAMB
    ("lars", 4, 0, "plain", [16, 12], 28, 20),     # fp32 LARS
    ("lamb", 2, 2, "skip_nonfinite", [14, 28], 40, 28),
    ("lars", 4, 0, "skip_nonfinite", [12, 20], 28, 20),
    ("nlamb", 2, 2, "plain", [22, 20], 42, 28),
    ("nnlamb", 4, 0, "plain", [24, 20], 44, 28),
    ("lamb", 2, 2, "grad_norm", [22, 18], 40, 28),
    ("lamb", 2, 2, "decoupled", [22, 18], 40, 28),
]


@pytest.mark.parametrize("opt,gb,cb,variant,per_kernel,two_pass,single",
                         CASES)
def test_kernel_byte_model(opt, gb, cb, variant, per_kernel, two_pass,
                           single):
    names, got = bench.kernel_model(opt, 1, gb, cb, variant)
    assert got == per_kernel and len(names) == 2
    assert bench.two_pass_bytes(opt, gb, cb) == two_pass
    assert bench.single_touch_bytes(opt, gb, cb) == single
    if variant in ("plain", "grad_norm", "decoupled"):
        assert sum(got) == two_pass
    if variant == "skip_nonfinite":   # one more read of g per step
        assert sum(got) == two_pass + gb


def test_onchip_model_counts_streamed_tensors_at_two_pass_bytes():
    names, got = bench.kernel_model("lamb", 3, 2, 2)
    assert len(names) == 1 and got == [28]
    # a quarter of the parameters streamed through the two-pass kernels
    names, got = bench.kernel_model("lamb", 3, 2, 2, "plain", 0.25)
    assert len(names) == 3 and got == [22 * 0.25, 18 * 0.25, 28 * 0.75]
    # the flagged variants run on the two-pass kernels of such a plan
    names, got = bench.kernel_model("lamb", 3, 2, 2, "grad_norm")
    assert len(names) == 2 and got == [22, 18]


def test_profiled_traffic_by_workload_label(tmp_path):
    f = tmp_path / "multi.md"
    h = bench.kernel_source_hash(bench.ONCHIP_SOURCES)
    f.write_text(f"kernel_source_sha256: {h}\n"
                 "traffic_bytes_per_launch[resnet50/lamb][0]: 6.613e8\n"
                 "traffic_bytes_per_launch[resnet50/lars][0]: 4.562e8\n")
    assert bench.profiled_traffic(str(f), 0, "resnet50/lars",
                                  bench.ONCHIP_SOURCES) == 4.562e8
    assert bench.profiled_traffic(str(f), 0, "mlp/lamb",
                                  bench.ONCHIP_SOURCES) is None
    # the two-pass sources give another hash
    assert bench.profiled_traffic(str(f), 0, "resnet50/lars") is None


def _tree_copy(tmp_path):
    dst = tmp_path / "paper_1904_00962_gb300" / "csrc"
    shutil.copytree(os.path.join(ROOT, "paper_1904_00962_gb300", "csrc"), dst,
                    ignore=shutil.ignore_patterns("*.o", "*.so"))
    return dst


def test_kernel_hash_ignores_comments_not_code(tmp_path, monkeypatch):
    base = bench.kernel_source_hash()
    csrc = _tree_copy(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.kernel_source_hash() == base
    f = csrc / "lamb_kernels.cu"
    src = f.read_text()
    f.write_text("// a new comment line\n/* and a block\n comment */\n" +
                 src.replace("\n", "\n  ", 5))
    assert bench.kernel_source_hash() == base
    f.write_text(src.replace("kUnroll2 = 4", "kUnroll2 = 2", 1))
    assert bench.kernel_source_hash() != base


def test_profiled_traffic_only_for_matching_source(tmp_path):
    good = tmp_path / "good.md"
    good.write_text(f"kernel_source_sha256: {bench.kernel_source_hash()}\n"
                    "traffic_bytes_per_launch[0]: 7.1586e9\n"
                    "traffic_bytes_per_launch[1]: 5.8486e9\n")
    assert bench.profiled_traffic(str(good), 0) == 7.1586e9
    assert bench.profiled_traffic(str(good), 1) == 5.8486e9
    assert bench.profiled_traffic(str(good), 2) is None
    stale = tmp_path / "stale.md"
    stale.write_text("kernel_source_sha256: 0123456789abcdef\n"
                     "traffic_bytes_per_launch[0]: 7.1586e9\n")
    assert bench.profiled_traffic(str(stale), 0) is None
    assert bench.profiled_traffic(str(tmp_path / "missing.md"), 0) is None


def test_committed_kernel_profile_has_the_parsed_fields():
    text = open(bench.KERNELS[1][2]).read()
    assert "kernel_source_sha256:" in text
    for i in range(2):
        assert f"traffic_bytes_per_launch[{i}]:" in text


def test_layout_hyper_takes_the_layouts_lars_settings_or_the_default():
    from paper_1904_00962_gb300 import binding as B
    from paper_1904_00962_gb300.workloads import get_layout
    rn = get_layout("resnet50")
    h, c = bench.layout_hyper(rn, "lars")
    assert h is rn.lars_hyper and c.trust_coef == pytest.approx(h.trust_coef)
    assert not (c.flags & B.LAMB_FLAG_BIAS_CORRECTION)
    mlp = get_layout("mlp")
    h, c = bench.layout_hyper(mlp, "lars")
    assert (h.lr, h.trust_coef, h.bias_correction) == (1.0, 1e-3, False)
    h, c = bench.layout_hyper(get_layout("bert_large"), "lamb", "decoupled")
    assert c.flags & B.LAMB_FLAG_BIAS_CORRECTION
    assert c.flags & B.LAMB_FLAG_DECOUPLED_DECAY
    assert c.flags & B.LAMB_FLAG_INCREMENT_STEP


def test_shard_timing_declines_under_several_ranks():
    """--shard-world is a one-process measurement: under torchrun every rank
    exits 0 and rank 0 prints an `unavailable` line, before any device use."""
    import json
    import subprocess
    env = dict(os.environ, RANK="0", LOCAL_RANK="0", WORLD_SIZE="2")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"),
                        "--shard-world", "2"], capture_output=True, text=True,
                       env=env, cwd=ROOT, timeout=300)
    assert r.returncode == 0, r.stderr
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert "unavailable" in line


def test_clock_record_keeps_the_timed_window_and_its_reasons(tmp_path,
                                                             monkeypatch):
    """bench.py's clock sampler, fed by a stand-in nvidia-smi: only samples
    inside the marked window count, the median SM clock and the maximum are
    taken from them, and a throttle reason is reported when any of those
    samples shows it active."""
    import datetime as dt
    import stat
    rows = [  # time, sm, max, power, active, hw, hw_thermal, sw_thermal, cap
        ("10:00:00.000", 1000, 2070, "Not Active", "Not Active"),   # before
        ("10:00:00.200", 2070, 2070, "Not Active", "Not Active"),
        ("10:00:00.300", 2050, 2070, "Not Active", "Active"),
        ("10:00:00.400", 2070, 2070, "Not Active", "Not Active"),
        ("10:00:00.900", 900, 2070, "Active", "Not Active"),       # after
    ]
    lines = [f"2026/12/02 {t}, {sm}, {mx}, 950.00, 0x0, {hw}, Not Active, "
             f"Not Active, {cap}" for t, sm, mx, hw, cap in rows]
    fake = tmp_path / "nvidia-smi"
    fake.write_text("#!/bin/sh\ncat <<'EOF_'\n" + "\n".join(lines) +
                    "\nEOF_\nexec sleep 30\n")
    fake.chmod(fake.stat().st_mode | stat.S_IEXEC)
    monkeypatch.setenv("PATH", f"{tmp_path}:{os.environ['PATH']}")
    cs = bench.ClockSampler()
    import time
    time.sleep(0.5)   # let the stand-in print
    cs.mark(dt.datetime(2026, 12, 2, 10, 0, 0, 100000),
            dt.datetime(2026, 12, 2, 10, 0, 0, 500000))
    rec = cs.stop()
    assert rec == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "samples": 3,
                   "reasons": ["sw_power_cap"]}
