"""bench.py host logic without a GPU: the kernel-source hash that decides
whether the recorded ncu DRAM traffic belongs to the kernels being timed
ignores comments and whitespace-only lines but follows every code change, and
a record is reported only for the code and workload it was taken on, and the
input checksums do not depend on how the sum is sliced."""
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


def test_input_checksums_are_chunk_independent():
    """The bench records a checksum of each generated bf16 tensor, summed in
    slices so that no full-size wider copy is made: any slice size gives the
    sum of the bit patterns as 16-bit integers."""
    import torch
    from paper_2505_11254_gb300.inputs import TINY_N2048, checksum, checksums, generate
    g = torch.Generator().manual_seed(0)
    x = torch.randn(10007, generator=g).to(torch.bfloat16)
    ref = int(x.view(torch.int16).to(torch.int64).sum())
    assert all(checksum(x, chunk=c) == ref for c in (1, 7, 4096, 1 << 26))
    q, k, v = generate(TINY_N2048)
    rec = checksums(q, k, v)
    assert rec["Q"] == checksum(q) and rec["K"] == checksum(k) and rec["V"] == checksum(v)
    assert generate(TINY_N2048)[0].equal(q), "seeded generation is repeatable"
