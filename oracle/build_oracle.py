"""Compile the C oracle into ``oracle/libdqt_oracle.so`` (test infrastructure).

Built with ``-O2 -ffp-contract=off`` so that the compiler forms no fused
multiply-add: every fp32 operation of the AdamW + stochastic-rounding step is
rounded on its own, as the oracle's source states.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "dqt_oracle.c")
LIB = os.path.join(HERE, "libdqt_oracle.so")


def build(force: bool = False) -> str:
    if (not force and os.path.exists(LIB)
            and os.path.getmtime(LIB) >= os.path.getmtime(SRC)):
        return LIB
    tmp = LIB + ".tmp.%d" % os.getpid()
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-o", tmp, SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
