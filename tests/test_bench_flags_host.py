"""bench.py's ablation flags (the paper's axes: alpha of Eq. 3, the window
ratios, the static budget, cluster size, the hierarchy's fanouts and kept
ratios, the sharing group size, the inputs' cross-layer correlation): they
change the workload the line measures, the line's config reports them, and
the single-thread oracle child receives them unchanged."""
import sys

import pytest

import bench
from paper_2501_06807_gb300 import synth


def _args(*argv):
    old = sys.argv
    sys.argv = ["bench.py", *argv]
    try:
        return bench.parse_args()
    finally:
        sys.argv = old


def test_no_flags_is_the_named_workload():
    a = _args("--workload", synth.C3.name)
    assert bench.workload_of(a) is synth.C3
    assert bench.override_argv(a) == []


def test_flags_replace_the_workload_fields():
    a = _args("--workload", synth.C5.name, "--alpha", "0.8", "--window-ppm", "150000", "--keep-ppm", "300000",
              "--fanouts", "4", "--level-keep-ppm", "100000,500000", "--share-every", "2", "--layer-rho-ppm", "900000")
    w = bench.workload_of(a)
    assert (w.alpha, w.window_ppm, w.keep_ppm, w.share_every, w.layer_rho_ppm) == (0.8, 150_000, 300_000, 2, 900_000)
    assert w.fanouts == (4,) and w.level_keep_ppm == (100_000, 500_000) and w.n_levels == 2
    assert (w.prompt_len, w.n_layers, w.seed) == (synth.C5.prompt_len, synth.C5.n_layers, synth.C5.seed)
    cfg = bench.workload_config(w, 8, "replicas1")
    assert cfg["alpha"] == 0.8 and cfg["fanouts"] == [4] and cfg["level_keep_ppm"] == [100_000, 500_000]
    # the child that times the oracle on one core rebuilds the same workload
    child = _args("--workload", synth.C5.name, *bench.override_argv(a))
    assert bench.workload_of(child) == w


def test_flat_hierarchy_and_mismatched_ratios():
    a = _args("--workload", synth.C3.name, "--fanouts", "", "--level-keep-ppm", "200000")
    w = bench.workload_of(a)
    assert w.fanouts == () and w.n_levels == 1
    with pytest.raises(SystemExit):
        bench.workload_of(_args("--workload", synth.C3.name, "--fanouts", "4,4"))  # three levels, two ratios
    with pytest.raises(SystemExit):
        bench.workload_of(_args("--workload", synth.C3.name, "--alpha", "1.5"))


def test_decode_form_flags():
    a = _args("--speculate", "0", "--fuse", "1")
    assert (a.speculate, a.fuse) == (0, 1)
    d = _args()
    assert (d.speculate, d.fuse, d.report) == (-1, -1, None)
