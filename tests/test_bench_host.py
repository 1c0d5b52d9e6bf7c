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


def test_info_struct_matches_the_header():
    # pss_info as the header declares it, field by field, against the binding's ctypes mirror
    src = open(os.path.join(ROOT, "include", "pss.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    body = re.search(r"typedef struct \{(.*?)\} pss_info;", src, flags=re.S).group(1)
    fields = []
    for ctype, names in re.findall(r"(int64_t|uint64_t|double)\s+([^;]+);", body):
        fields += [(n.strip(), ctype) for n in names.split(",")]
    want = {"int64_t": "c_long", "uint64_t": "c_ulong", "double": "c_double"}
    got = [(n, t.__name__) for n, t in binding.PSSInfo._fields_]
    assert [n for n, _ in got] == [n for n, _ in fields]
    for (n, t), (_, ct) in zip(got, fields):
        assert t in (want[ct], want[ct].replace("long", "longlong")), n


def test_enum_values_match_the_header():
    src = open(os.path.join(ROOT, "include", "pss.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    for prefix in ("PATH", "UPDATE", "SORT", "ACCUM"):
        vals = dict((k, int(v)) for k, v in re.findall(rf"\bPSS_{prefix}_([A-Z_0-9]+)\s*=\s*(\d+)", src))
        assert vals, prefix
        for name, value in vals.items():
            assert getattr(binding, f"{prefix}_{name}") == value, (prefix, name)


def test_workload_description_follows_the_batch_and_M():
    ns = _parse(["--workload", "sweep", "--M", str(1 << 28), "--B", "8192"])

    class W:
        B, M = 8192, 1 << 28
    desc = bench._workload_desc(ns, W)
    assert "batch 8192" in desc and f"M={1 << 28} fp32" in desc and "--M" not in desc
    ns = _parse(["--workload", "tb"])
    W.B, W.M = 65536, 2_500_000
    assert bench._workload_desc(ns, W) == bench.WORKLOAD_DESC["tb"]


def test_sort_description_names_the_grouping_that_ran():
    class H:
        def __init__(self, **info):
            self._info = dict(last_path=binding.PATH_SORTED, last_collision_rate=0.5, R=1 << 20)
            self._info.update(info)

        def info(self):
            return self._info
    ns = _parse([])
    assert bench._sort_desc(H(last_path=binding.PATH_ATOMIC), binding, ns) == {}
    assert "segment-local" in bench._sort_desc(H(last_collision_rate=-1.0), binding, ns)["sort"]
    d = bench._sort_desc(H(), binding, ns)
    assert d["sort"].startswith("counting") and d["collision_rate"] == 0.5
    assert bench._sort_desc(H(R=1 << 26), binding, ns)["sort"].startswith("radix")
    ns = _parse(["--deterministic"])
    assert bench._sort_desc(H(), binding, ns)["sort"].startswith("stable radix")
