"""Build the oracle's shared libraries with gcc (no CUDA involved).

Test infrastructure: produces liboracle.so (double arithmetic) and
liboracle_f32.so (float arithmetic, a self-check build) next to this file.
"""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
FLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
         "-fno-fast-math", "-Wall", "-Wextra", "-Wno-unused-parameter"]


def _stale(out, srcs):
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(s) > t for s in srcs)


def build(force=False):
    srcs = [os.path.join(HERE, "oracle.c"), os.path.join(HERE, "oracle.h")]
    outs = {"liboracle.so": [], "liboracle_f32.so": ["-DORACLE_REAL=float"]}
    for name, extra in outs.items():
        out = os.path.join(HERE, name)
        if force or _stale(out, srcs):
            cmd = ["gcc", *FLAGS, *extra, srcs[0], "-o", out + ".tmp", "-lm"]
            subprocess.run(cmd, check=True)
            os.replace(out + ".tmp", out)
    return [os.path.join(HERE, n) for n in outs]


if __name__ == "__main__":
    print(build(force=True))
