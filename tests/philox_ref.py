"""Independent Philox4x32-10 for the tests: torch's PhiloxRNGEngine.h.

A tiny C++ program (compiled once per session with g++) includes torch's
header and prints the four output words of one (key, counter) block.  The
engine's (seed, subsequence, offset) map to key = (seed lo, seed hi) and
counter = (offset lo, offset hi, subsequence lo, subsequence hi), so every
counter can be reached.  This is the library cross-check of the oracle's own
Philox; nothing here is copied from that header.
"""
import os
import subprocess
import tempfile

import numpy as np

_PROG = r"""
#include <ATen/core/PhiloxRNGEngine.h>
#include <cstdio>
#include <cstdlib>
int main() {
  unsigned long long seed, sub, off;
  while (std::scanf("%llu %llu %llu", &seed, &sub, &off) == 3) {
    at::Philox4_32 eng(seed, sub, off);
    unsigned a = eng(), b = eng(), c = eng(), d = eng();
    std::printf("%u %u %u %u\n", a, b, c, d);
  }
  return 0;
}
"""
_exe = None


def _torch_include():
    import torch
    return os.path.join(os.path.dirname(torch.__file__), "include")


def available() -> bool:
    return os.path.exists(os.path.join(_torch_include(), "ATen", "core", "PhiloxRNGEngine.h"))


def _build():
    global _exe
    if _exe is None:
        d = tempfile.mkdtemp(prefix="philox_ref_")
        src = os.path.join(d, "p.cpp")
        with open(src, "w") as f:
            f.write(_PROG)
        exe = os.path.join(d, "p")
        subprocess.run(["g++", "-std=c++17", "-O1", "-I", _torch_include(), src, "-o", exe],
                       check=True)
        _exe = exe
    return _exe


def blocks(seed: int, counters) -> np.ndarray:
    """Philox4x32-10 words [n, 4] for counters [n, 4] under one 64-bit seed."""
    ctr = np.asarray(counters, dtype=np.uint64).reshape(-1, 4)
    lines = []
    for c0, c1, c2, c3 in ctr:
        off = int(c0) | (int(c1) << 32)
        sub = int(c2) | (int(c3) << 32)
        lines.append(f"{seed} {sub} {off}")
    out = subprocess.run([_build()], input="\n".join(lines) + "\n", capture_output=True,
                         text=True, check=True).stdout.split()
    return np.array([int(x) for x in out], dtype=np.uint32).reshape(-1, 4)


def rademacher(seed: int, step: int, expert: int, probe: int, p0: int, count: int) -> np.ndarray:
    """z[p] = 1 - 2 * bit of block (p >> 7, probe, step, expert): word
    (p & 127) >> 5, bit (o >> 1) + 16 (o & 1) with o = p & 31."""
    p = np.arange(p0, p0 + count, dtype=np.int64)
    blk = np.unique(p >> 7)
    words = blocks(seed, [(int(b), probe, step & 0xFFFFFFFF, expert) for b in blk])
    row = {int(b): k for k, b in enumerate(blk)}
    k = p & 127
    w = np.array([words[row[int(b)], int(kk) >> 5] for b, kk in zip(p >> 7, k)], dtype=np.uint64)
    o = k & 31
    bit = (w >> ((o >> 1) + 16 * (o & 1)).astype(np.uint64)) & np.uint64(1)
    return (1 - 2 * bit.astype(np.int64)).astype(np.int8)
