"""The C ABI from a plain C (and C++) caller, without Python in between.

tests/c_consumer.c includes only include/kvtier.h and links libkvtier.so.
It is compiled as strict C99 and as C++17 (so the header's types and
extern "C" guards hold for both), run on a host-logic-only pool, and its
printed block ids are checked against the oracle's free-list contract:
Fisher-Yates over 0..n-1 seeded by splitmix64, allocations popped from the
end, blocks freed at a pause pushed back in logical order.
"""
import os
import shutil
import subprocess

import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
PKG = os.path.join(ROOT, "paper_2609_25782_gb300")


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__.build()
    return os.path.join(PKG, "libkvtier.so")


def compile_and_run(tmp_path, compiler, flags):
    exe = str(tmp_path / f"c_consumer_{compiler.replace('+', 'p')}")
    cmd = [compiler, *flags, "-Wall", "-Wextra", "-Werror", "-pedantic",
           os.path.join(HERE, "c_consumer.c"), "-I", os.path.join(ROOT, "include"),
           "-L", PKG, "-lkvtier", f"-Wl,-rpath,{PKG}", "-Wl,--allow-shlib-undefined", "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([exe], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr
    out = {}
    for line in r.stdout.splitlines():
        for part in line.split():
            k, _, v = part.partition("=")
            out[k] = v
    return out


def ids(s):
    return [int(x) for x in s.split(",")] if s else []


@pytest.mark.parametrize("compiler,flags", [("gcc", ["-std=c99", "-x", "c"]),
                                            ("g++", ["-std=c++17", "-x", "c++"])])
def test_c_caller(lib, tmp_path, compiler, flags):
    if shutil.which(compiler) is None:
        pytest.skip(f"{compiler} not installed")
    out = compile_and_run(tmp_path, compiler, flags)
    assert out["failures"] == "0"
    assert int(out["token_bytes"]) == 98304            # 96 KiB per token (48 layers)
    assert int(out["block_bytes"]) == 16 * 98304       # 1.5 MiB per 16-token block
    assert out["sids"] == "0,1"

    fl = oracle.FreeList(20, 7)
    row0 = [int(x) for x in fl.pop(3)]                 # 40 tokens: 3 blocks
    row1 = [int(x) for x in fl.pop(1)]                 # 16 tokens: 1 block
    assert ids(out["row0_after_append"]) == row0
    assert ids(out["row1_after_append"]) == row1
    row1 += [int(x) for x in fl.pop(1)]                # reserve: session 1's tail was full
    assert ids(out["row1_after_reserve"]) == row1
    assert out["tokens0"] == "41"
    fl.push(row0)                                      # pause frees in logical order
    assert ids(out["row0_after_resume"]) == [int(x) for x in fl.pop(3)]
    assert out["last_error_nonempty"] == "1"
    assert out["free_blocks"] == str(20 - 5) and out["used_blocks"] == "5"
    assert out["appends"] == "4" and out["pauses"] == "1" and out["resumes"] == "1"
