"""Build the CUDA libraries in-tree: ``librps.so`` (the scoring path) and
``librps_synth.so`` (the seeded logit generator), for sm_103a only.

Translation units compile in parallel; nothing is installed outside the package.
Set ``RPS_PTXAS_VERBOSE=1`` to print register / spill / shared-memory usage.
"""
from __future__ import annotations

import os
import subprocess
import sys
from pathlib import Path

PKG = Path(__file__).resolve().parent
ROOT = PKG.parent
CSRC = PKG / "csrc"
INCLUDE = ROOT / "include"
BUILD = PKG / "_build"
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-ffp-contract=off",
                f"-I{INCLUDE}", f"-I{CSRC}"]

LIBS = {
    "librps.so": ["abi.cu", "rowstats.cu", "decide.cu", "decode.cu", "gather.cu", "static_scratch.cu", "lmhead.cu", "attention.cu"],
    "librps_synth.so": ["synth.cu"],
}
HEADERS = [INCLUDE / "rps.h", INCLUDE / "rps_synth.h", CSRC / "rps_internal.cuh", CSRC / "umma_desc.h"]


def _stale(target: Path, sources) -> bool:
    if not target.exists():
        return True
    t = target.stat().st_mtime
    return any(Path(s).stat().st_mtime > t for s in sources)


def build(force: bool = False, verbose: bool = False) -> dict:
    """Compile every library that is missing or older than its sources."""
    BUILD.mkdir(exist_ok=True)
    extra = ["-Xptxas", "-v"] if os.environ.get("RPS_PTXAS_VERBOSE") else []
    jobs = []
    for lib, units in LIBS.items():
        for u in units:
            src = CSRC / u
            obj = BUILD / (Path(u).stem + ".o")
            if force or _stale(obj, [src, *HEADERS]):
                cmd = [NVCC, *FLAGS, *extra, "-c", str(src), "-o", str(obj)]
                jobs.append((cmd, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)))
    failed = []
    for cmd, proc in jobs:
        out, _ = proc.communicate()
        if proc.returncode != 0 or verbose or extra:
            sys.stdout.write(out)
        if proc.returncode != 0:
            failed.append(" ".join(cmd))
    if failed:
        raise RuntimeError("nvcc failed:\n" + "\n".join(failed))
    built = {}
    for lib, units in LIBS.items():
        target = PKG / lib
        objs = [BUILD / (Path(u).stem + ".o") for u in units]
        if force or _stale(target, objs):
            tmp = target.with_name(target.name + f".tmp{os.getpid()}")
            cmd = [NVCC, *ARCH, "-shared", "-o", str(tmp), *map(str, objs)]
            subprocess.run(cmd, check=True)
            os.replace(tmp, target)
        built[lib] = target
    return built


if __name__ == "__main__":
    for name, path in build(force="--force" in sys.argv, verbose=True).items():
        print(name, path)
