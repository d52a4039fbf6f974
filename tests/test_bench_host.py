"""bench.py host logic without a GPU: the kernel-source hash that decides
whether the recorded ncu DRAM traffic belongs to the kernels being timed
ignores comments and whitespace-only lines but follows every code change, and
a record is reported only for the code and workload it was taken on."""
import importlib.util
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    argv = sys.argv
    sys.argv = ["bench.py"]
    try:
        spec.loader.exec_module(mod)
    finally:
        sys.argv = argv
    return mod


def test_code_only_strips_comments_not_code():
    b = _bench()
    src = 'int a = 1;  // one\n/* two\n   lines */\nconst char* s = "x // y /* z */";\n\n  char c = \'/\';\n'
    got = b._code_only(src)
    assert got == 'int a = 1;\nconst char* s = "x // y /* z */";\n  char c = \'/\';'
    # a comment edit leaves the code the same, a code edit does not
    assert b._code_only(src.replace("// one", "// uno")) == got
    assert b._code_only(src.replace("= 1", "= 2")) != got
    # escaped quotes inside a literal do not end it
    assert b._code_only('s = "a\\"b // c"; // d') == 's = "a\\"b // c";'


def test_recorded_traffic_lookup():
    """A record taken on the current kernel code is reported for its own
    workload only; a record of other code is not reported at all."""
    b = _bench()
    with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
        rec = json.load(f)
    sha = b.kernel_src_hash()
    for name, e in rec.items():
        want = e["dram_bytes_per_launch"] if e["src_sha"] == sha else None
        assert b.recorded_traffic(name, e["workload"]) == want
        assert b.recorded_traffic(name, "another_workload") is None
