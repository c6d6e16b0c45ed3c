"""Compile the oracle's C part (gcc, no FP contraction): oracle/liboracle.so in fp64
(the parity oracle) and oracle/liboracle_f32.so, the same source in fp32 (the plain fp32
forward the benchmark times as its CPU baseline).

Test infrastructure: only the tests, the smoke check and the benchmark's
CPU-baseline leg load the result.
"""
from __future__ import annotations

import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "oracle_conv.c")
LIB = os.path.join(HERE, "liboracle.so")
LIB_F32 = os.path.join(HERE, "liboracle_f32.so")


def _build_one(lib, defines, force):
    if not force and os.path.exists(lib) and os.path.getmtime(lib) >= os.path.getmtime(SRC):
        return lib
    tmp = lib + ".tmp.%d" % os.getpid()
    # -ffp-contract=off: no fused multiply-add, so that the full-map and the
    # region loops round identically on every host (x86-64 and aarch64).
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
           "-fopenmp"] + defines + [SRC, "-o", tmp]
    subprocess.check_call(cmd)
    os.replace(tmp, lib)
    return lib


def build_oracle(force: bool = False) -> str:
    """Build both libraries; returns the path of the fp64 one."""
    _build_one(LIB_F32, ["-DORACLE_REAL=float"], force)
    return _build_one(LIB, [], force)


if __name__ == "__main__":
    print(build_oracle(force="--force" in sys.argv))
