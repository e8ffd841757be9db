"""Build the synthetic-input generator: a host library (gcc) and a device
filler library (nvcc, sm_103a).  Neither holds any of the method's arithmetic."""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CUDA_HOME = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _stale(out, srcs):
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(s) > t for s in srcs)


def build_host(force=False):
    src = os.path.join(HERE, "synth.c")
    out = os.path.join(HERE, "libsynth_host.so")
    if force or _stale(out, [src, os.path.join(HERE, "synth.h")]):
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                        "-ffp-contract=off", "-Wall", src, "-o", out + ".tmp", "-lm"],
                       check=True)
        os.replace(out + ".tmp", out)
    return out


def build_cuda(force=False):
    src = os.path.join(HERE, "synth_cuda.cu")
    out = os.path.join(HERE, "libsynth_cuda.so")
    if force or _stale(out, [src, os.path.join(HERE, "synth.h")]):
        nvcc = os.path.join(CUDA_HOME, "bin", "nvcc")
        subprocess.run([nvcc, "-O3", "-gencode", "arch=compute_103a,code=sm_103a",
                        "-shared", "-Xcompiler", "-fPIC", "-cudart", "shared",
                        "-fmad=false", "-Xlinker", f"-rpath,{CUDA_HOME}/lib64",
                        src, "-o", out + ".tmp"], check=True)
        os.replace(out + ".tmp", out)
    return out


def build(force=False, cuda=True):
    outs = [build_host(force)]
    if cuda:
        outs.append(build_cuda(force))
    return outs


if __name__ == "__main__":
    print(build(force=True))
