"""Compile the C oracle (``laq_oracle.c``) into ``liblaq_oracle.so`` next to it with gcc.

Test infrastructure: building the checker is not using it.  Plain C, no architecture-specific
flags, so the same source builds on x86_64 and aarch64 hosts.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "laq_oracle.c")
LIB = os.path.join(HERE, "liblaq_oracle.so")


def build(force: bool = False) -> str:
    """Build the oracle library if it is missing or older than its source; return its path."""
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
           "-ffp-contract=off", "-o", tmp, SRC, "-lm"]
    # OpenMP only splits laqo_gemm_threads' output columns over the host cores; without it the
    # same source builds single-threaded
    if subprocess.run(cmd[:1] + ["-fopenmp"] + cmd[1:], stdout=subprocess.DEVNULL,
                      stderr=subprocess.DEVNULL).returncode != 0:
        subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
