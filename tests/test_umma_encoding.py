"""Host-side check of the tcgen05 encodings in csrc/umma.cuh (no GPU): the
shared-memory matrix descriptor, the kind::f16 instruction descriptor and the
128-byte swizzle are compiled for the host with g++ and compared with the
bit layout packed independently here, field by field."""

import os
import shutil
import subprocess
import tempfile

import pytest

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "paper_2607_02805_gb300", "csrc")

PROG = r"""
#define __host__
#define __device__
#define __forceinline__ inline
#include <cstdio>
#include "umma.cuh"
int main() {
  using namespace bds::umma;
  const unsigned addrs[] = {0x400u, 0x8000u, 0x1F000u, 0x3FFF0u};
  const unsigned lbos[] = {16u, 1024u, 16384u, 32768u};
  const unsigned sbos[] = {1024u, 2048u};
  for (unsigned a : addrs) for (unsigned l : lbos) for (unsigned s : sbos)
    std::printf("S %u %u %u %llu\n", a, l, s, (unsigned long long)sdesc(a, l, s));
  const unsigned ms[] = {64u, 128u}, ns[] = {64u, 128u, 256u};
  for (unsigned m : ms) for (unsigned n : ns) for (int amn = 0; amn < 2; ++amn) for (int bmn = 0; bmn < 2; ++bmn)
    std::printf("I %u %u %d %d %u\n", m, n, amn, bmn, idesc_bf16(m, n, amn, bmn));
  for (unsigned r = 0; r < 16; ++r) for (unsigned c = 0; c < 8; ++c) std::printf("W %u %u %u\n", r, c, sw128(r, c));
  return 0;
}
"""


def _run():
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not available")
    with tempfile.TemporaryDirectory() as d:
        src, exe = os.path.join(d, "enc.cpp"), os.path.join(d, "enc")
        open(src, "w").write(PROG)
        subprocess.run([gxx, "-std=c++17", "-I" + CSRC, src, "-o", exe], check=True)
        return subprocess.run([exe], check=True, capture_output=True, text=True).stdout.split("\n")


def test_smem_descriptor_fields():
    n = 0
    for line in _run():
        if not line.startswith("S "):
            continue
        a, l, s, v = (int(x) for x in line.split()[1:])
        assert v & 0x3FFF == (a >> 4) & 0x3FFF                # start address >> 4, bits 0-13
        assert (v >> 16) & 0x3FFF == (l >> 4) & 0x3FFF        # leading byte offset >> 4, bits 16-29
        assert (v >> 32) & 0x3FFF == (s >> 4) & 0x3FFF        # stride byte offset >> 4, bits 32-45
        assert (v >> 46) & 0x3 == 1                           # descriptor version
        assert (v >> 49) & 0x7 == 0                           # base offset (1024-byte aligned atoms)
        assert (v >> 61) & 0x7 == 2                           # 128-byte swizzle
        assert v & ((0x3 << 14) | (0x3 << 30) | (0x1 << 48) | (0xFF << 53)) == 0  # reserved bits clear
        n += 1
    assert n == 32


def test_instruction_descriptor_fields():
    n = 0
    for line in _run():
        if not line.startswith("I "):
            continue
        m, nn, amn, bmn, v = (int(x) for x in line.split()[1:])
        expect = (1 << 4) | (1 << 7) | (1 << 10) | (amn << 15) | (bmn << 16) | ((nn >> 3) << 17) | ((m >> 4) << 24)
        assert v == expect
        assert (v >> 4) & 3 == 1 and (v >> 7) & 7 == 1 and (v >> 10) & 7 == 1  # f32 accumulate, bf16 A and B
        assert (v >> 17) & 0x3F == nn >> 3 and (v >> 24) & 0x1F == m >> 4
        assert v & ((1 << 23) | (1 << 29) | 0xF | (1 << 6) | (3 << 13)) == 0   # sparsity, negate, reserved clear
        n += 1
    assert n == 24


def test_swizzle_is_a_permutation_within_each_row():
    rows = {}
    for line in _run():
        if line.startswith("W "):
            r, c, off = (int(x) for x in line.split()[1:])
            assert off // 128 == r and off % 16 == 0
            rows.setdefault(r, set()).add((off % 128) // 16)
            assert (off % 128) // 16 == c ^ (r % 8)
    assert all(v == set(range(8)) for v in rows.values()) and len(rows) == 16
