"""Compile the C oracle into ``oracle/librsref.so`` with gcc.

TEST INFRASTRUCTURE ONLY: the oracle is the plain fp64 CPU statement of the
method that the CUDA library is checked against.  ``-ffp-contract=off`` keeps
gcc from fusing multiply-adds (aarch64 has FMA in its base ISA, x86-64 does
not), so the oracle rounds identically on both hosts.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SOURCES = ["entropy.c", "match.c", "attn.c", "accept.c", "sample.c"]
LIB = os.path.join(HERE, "librsref.so")


def build(force: bool = False) -> str:
    srcs = [os.path.join(HERE, s) for s in SOURCES]
    deps = srcs + [os.path.join(HERE, "rsref.h")]
    if not force and os.path.exists(LIB):
        lib_mtime = os.path.getmtime(LIB)
        if all(os.path.getmtime(p) <= lib_mtime for p in deps):
            return LIB
    tmp = LIB + ".tmp.%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
           "-fno-fast-math", "-Wall", "-Wextra", "-Wno-unused-parameter",
           "-o", tmp] + srcs + ["-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
