"""Builds mlkv_synth/libmlkv_synth.so (device side of the input generator) with nvcc."""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "synth_gpu.cu")
LIB = os.path.join(HERE, "libmlkv_synth.so")
NVCC = "/usr/local/cuda/bin/nvcc" if os.path.exists("/usr/local/cuda/bin/nvcc") else "nvcc"


def command():
    return [NVCC, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
            "-Xcompiler", "-fPIC", "-shared", "-cudart", "static", "-o", LIB, SRC]


def needs_build():
    return (not os.path.exists(LIB)) or os.path.getmtime(LIB) < max(
        os.path.getmtime(SRC), os.path.getmtime(os.path.abspath(__file__)))


def build(force=False):
    if force or needs_build():
        subprocess.run(command(), check=True)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
