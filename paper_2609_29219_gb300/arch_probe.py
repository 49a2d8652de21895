"""Architecture microbenchmarks of the analytic model (paper Sec. 2.7).

Builds ``csrc/arch_probe.cu`` into ``_build/arch_probe`` for sm_103a and runs it on the
current GPU; the program prints one JSON object with the MUFU/FMA pipe rates, single
tcgen05.mma rates, and the prefill kernel's MMA stream under added load.

    python -m paper_2609_29219_gb300.arch_probe
"""
from __future__ import annotations

import json
import os
import subprocess
import sys

from . import build as _build

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "csrc", "arch_probe.cu")
EXE = os.path.join(_build.BUILD, "arch_probe")


def build(force: bool = False) -> str:
    os.makedirs(_build.BUILD, exist_ok=True)
    deps = [SRC] + _build._headers()
    if force or _build._stale(EXE, deps):
        cmd = [_build._nvcc(), *_build.ARCH, "-O3", "-std=c++17", "--expt-relaxed-constexpr", "-o", EXE, SRC]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed:\n{r.stdout}\n{r.stderr}")
    return EXE


def run(timeout: float = 300.0) -> dict:
    out = subprocess.run([build()], capture_output=True, text=True, timeout=timeout)
    if out.returncode != 0:
        raise RuntimeError(out.stdout + out.stderr)
    return json.loads(out.stdout.strip().splitlines()[-1])


if __name__ == "__main__":
    res = run()
    json.dump(res, sys.stdout, indent=1)
    print()
