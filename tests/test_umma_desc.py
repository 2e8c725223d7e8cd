"""The tcgen05 descriptor encoders (csrc/umma_desc.h), field by field, on the host.

A wrong field in either descriptor makes the tensor cores read the wrong
shared memory or the wrong shape, so each field is checked here against the
bit layout of the PTX ISA's tables (instruction descriptor of kind::f16;
shared-memory matrix descriptor of tcgen05) before any kernel uses them. The
header is plain C++; a small host program prints the encodings.
"""
import shutil
import subprocess
from pathlib import Path

import pytest

CSRC = Path(__file__).resolve().parents[1] / "paper_2608_11742_gb300" / "csrc"

PROGRAM = r"""
#include <cstdio>
#include "umma_desc.h"
using namespace rps::umma;
int main() {
    const unsigned mn[][2] = {{128, 256}, {128, 128}, {64, 64}, {128, 16}};
    for (auto &p : mn) std::printf("I %u %u %u\n", p[0], p[1], instr_desc_bf16(p[0], p[1]));
    const unsigned addr[] = {0u, 1024u, 0x12340u, 0x37c00u};
    for (unsigned a : addr) {
        std::printf("S %u %llu\n", a, (unsigned long long)smem_desc_kmajor_sw128(a));
        for (unsigned k = 0; k < 4; ++k)
            std::printf("K %u %u %llu\n", a, k, (unsigned long long)advance_k16(smem_desc_kmajor_sw128(a), k));
    }
    std::printf("G %llu\n", (unsigned long long)smem_desc(0x2000u, 0x80u, 0x400u, kSwizzleNone));
    return 0;
}
"""


def bits(x, lo, hi):
    """Field [lo, hi) of x."""
    return (x >> lo) & ((1 << (hi - lo)) - 1)


@pytest.fixture(scope="module")
def encodings(tmp_path_factory):
    gxx = shutil.which("g++")
    if not gxx:
        pytest.skip("no host C++ compiler")
    d = tmp_path_factory.mktemp("umma")
    src, exe = d / "desc.cpp", d / "desc"
    src.write_text(PROGRAM)
    subprocess.run([gxx, "-std=c++17", "-O0", f"-I{CSRC}", str(src), "-o", str(exe)], check=True)
    return subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines()


def test_instruction_descriptor_fields(encodings):
    rows = [l.split() for l in encodings if l.startswith("I ")]
    assert len(rows) == 4
    for _, m, n, v in rows:
        m, n, v = int(m), int(n), int(v)
        assert bits(v, 0, 2) == 0 and bits(v, 2, 3) == 0 and bits(v, 3, 4) == 0   # dense, no saturation
        assert bits(v, 4, 6) == 1                                                  # D: f32
        assert bits(v, 6, 7) == 0
        assert bits(v, 7, 10) == 1 and bits(v, 10, 13) == 1                        # A, B: bf16
        assert bits(v, 13, 14) == 0 and bits(v, 14, 15) == 0                       # no negation
        assert bits(v, 15, 16) == 0 and bits(v, 16, 17) == 0                       # A, B K-major
        assert bits(v, 17, 23) == n >> 3                                           # N / 8
        assert bits(v, 23, 24) == 0
        assert bits(v, 24, 29) == m >> 4                                           # M / 16
        assert bits(v, 29, 32) == 0
    m128n256 = int(rows[0][3])
    assert m128n256 == (1 << 4) | (1 << 7) | (1 << 10) | (32 << 17) | (8 << 24)


def test_shared_memory_descriptor_fields(encodings):
    rows = [l.split() for l in encodings if l.startswith("S ")]
    assert len(rows) == 4
    for _, a, v in rows:
        a, v = int(a), int(v)
        assert bits(v, 0, 14) == (a >> 4) & 0x3FFF      # start address / 16
        assert bits(v, 14, 16) == 0
        assert bits(v, 16, 30) == 1                     # leading offset: 16 bytes (unused by swizzled K-major)
        assert bits(v, 30, 32) == 0
        assert bits(v, 32, 46) == 1024 >> 4             # stride offset: 8-row groups 1024 bytes apart
        assert bits(v, 46, 48) == 1                     # descriptor version of tcgen05
        assert bits(v, 48, 49) == 0
        assert bits(v, 49, 52) == 0                     # base offset: atoms on 1024-byte boundaries
        assert bits(v, 52, 53) == 0                     # relative leading offset
        assert bits(v, 53, 61) == 0
        assert bits(v, 61, 64) == 2                     # 128-byte swizzle


def test_k_slices_advance_32_bytes_inside_the_address_field(encodings):
    for _, a, k, v in (l.split() for l in encodings if l.startswith("K ")):
        a, k, v = int(a), int(k), int(v)
        assert bits(v, 0, 14) == ((a + 32 * k) >> 4)
        assert v >> 14 == int([l for l in encodings if l.startswith(f"S {a} ")][0].split()[2]) >> 14


def test_general_encoder_places_each_offset(encodings):
    v = int([l for l in encodings if l.startswith("G ")][0].split()[1])
    assert bits(v, 0, 14) == 0x2000 >> 4
    assert bits(v, 16, 30) == 0x80 >> 4
    assert bits(v, 32, 46) == 0x400 >> 4
    assert bits(v, 61, 64) == 0 and bits(v, 46, 48) == 1
