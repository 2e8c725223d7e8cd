"""Compile the CPU oracle (test infrastructure) into ``oracle/liboracle.so``.

``-ffp-contract=off`` keeps every multiply and add separately rounded, so the
oracle gives the same bits on x86-64 and on aarch64 (where GCC would otherwise
fuse them into FMAs).
"""
from __future__ import annotations

import os
import subprocess
from pathlib import Path

HERE = Path(__file__).resolve().parent
SOURCE = HERE / "rps_oracle.c"
LIBRARY = HERE / "liboracle.so"
CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]


def build_oracle(out: Path = LIBRARY, src: Path = SOURCE, extra=()) -> Path:
    out = Path(out)
    tmp = out.with_name(out.name + f".tmp{os.getpid()}")
    cmd = ["gcc", *CFLAGS, *extra, "-o", str(tmp), str(src), "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def oracle_up_to_date() -> bool:
    return LIBRARY.exists() and LIBRARY.stat().st_mtime >= SOURCE.stat().st_mtime


if __name__ == "__main__":
    print(build_oracle())
