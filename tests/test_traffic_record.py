"""The ncu traffic record (profiles/ncu_traffic.json) and the code hash that
ties each entry to the kernel source it was captured on: comments and layout
do not count, code does."""
import hashlib
import importlib.util
import json
import os

import pytest

from conftest import ROOT


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


B = _bench()

SRC = '''// leading comment
#include "x.h"
__global__ void k(float *p) {   /* block
   comment */ p[0] = 1.0f;  // trailing
    const char *s = "a // not a comment /* nor this */";
    char q = '"';
}
'''


def test_code_text_drops_comments_keeps_strings():
    t = B.code_text(SRC)
    assert "leading" not in t and "trailing" not in t and "block" not in t
    assert '"a // not a comment /* nor this */"' in t
    assert "'\"'" in t
    assert t == ('#include "x.h" __global__ void k(float *p) { p[0] = 1.0f; '
                 'const char *s = "a // not a comment /* nor this */"; char q = \'"\'; }')


@pytest.mark.parametrize("edit", [
    lambda s: s.replace("// trailing", "// another remark"),
    lambda s: s.replace("/* block\n   comment */", "/* x */"),
    lambda s: s.replace("    const", "\tconst"),
    lambda s: s + "\n\n// appended note\n",
])
def test_code_text_ignores_comments_and_layout(edit):
    assert B.code_text(edit(SRC)) == B.code_text(SRC)


@pytest.mark.parametrize("edit", [
    lambda s: s.replace("1.0f", "2.0f"),
    lambda s: s.replace("p[0]", "p[1]"),
    lambda s: s.replace('"a // not', '"b // not'),
    lambda s: s.replace("/* block", "p[2] = 0; /* block"),
])
def test_code_text_sees_code_edits(edit):
    assert B.code_text(edit(SRC)) != B.code_text(SRC)


def test_record_entries_are_complete_and_consistent():
    with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
        rec = json.load(f)
    n = 0
    for kernel, per in rec.items():
        if kernel.startswith("_"):
            continue
        for workload, e in per.items():
            n += 1
            assert e["dram_bytes_per_launch"] == e["dram_read_bytes"] + e["dram_write_bytes"], (kernel, workload)
            assert os.path.exists(os.path.join(ROOT, e["source"])), e["source"]
            for key in ("source_sha256_16", "code_sha256_16"):
                assert len(e[key]) == 16 and int(e[key], 16) >= 0
            # where the file is still the captured one, its code hash must be the recorded one
            path = os.path.join(ROOT, e["source"])
            with open(path, "rb") as f:
                if hashlib.sha256(f.read()).hexdigest()[:16] == e["source_sha256_16"]:
                    assert B.code_hash(path) == e["code_sha256_16"], (kernel, workload)
    assert n >= 5
