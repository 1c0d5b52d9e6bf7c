"""Host-side logic of bench.py and the binding's constants, without a GPU."""
import contextlib
import io
import json
import os
import re

import bench
from paper_2207_10731_gb300 import binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _parse(argv):
    # the same parser bench.main uses, without running anything
    import argparse
    captured = {}
    real = argparse.ArgumentParser.parse_args

    def grab(self, args=None, namespace=None):
        ns = real(self, args, namespace)
        captured["ns"] = ns
        raise SystemExit(0)

    argparse.ArgumentParser.parse_args = grab
    try:
        try:
            bench.main(argv)
        except SystemExit:
            pass
    finally:
        argparse.ArgumentParser.parse_args = real
    return captured["ns"]


def test_reference_arm_prints_one_contract_line():
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        rc = bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "2",
                         "--warmup", "3"])
    assert rc in (0, None)
    lines = [ln for ln in buf.getvalue().splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["value"] > 0 and d["steps"] == 2 and d["warmup"] == 3
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0


def test_shape_and_distribution_overrides():
    ns = _parse(["--Z", "16", "--G", "1", "--ids", "uniform"])
    assert bench._shape_overrides(ns) == {"Z": 16, "G": 1, "ids": ("uniform",)}
    ns = _parse([])
    assert bench._shape_overrides(ns) == {}


def test_binding_option_values_match_the_header():
    src = open(os.path.join(ROOT, "include", "pss.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    opts = dict((k, int(v)) for k, v in re.findall(r"\bPSS_OPT_([A-Z_0-9]+)\s*=\s*(\d+)", src))
    assert opts, "no options found in the header"
    for name, value in opts.items():
        assert getattr(binding, "OPT_" + name) == value, name


def test_traffic_hash_ignores_comments_and_the_host_only_file():
    assert bench._code_only("a = 1;  // note\n/* block\n comment */b = 2;\n\n") == "a = 1;\nb = 2;"
    assert "pss_api.cu" in bench._HOST_ONLY
    assert len(bench._kernel_sha()) == 16
