"""Builds mlkv_synth/libmlkv_synth.so (device side of the input generator) with nvcc."""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "synth_gpu.cu")
LIB = os.path.join(HERE, "libmlkv_synth.so")
NVCC = "/usr/local/cuda/bin/nvcc" if os.path.exists("/usr/local/cuda/bin/nvcc") else "nvcc"


HOST_SRC = os.path.join(HERE, "synth_host.c")
HOST_LIB = os.path.join(HERE, "libmlkv_synth_host.so")


def host_command():
    cc = os.environ.get("CC", "gcc")
    return [cc, "-std=c99", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-o", HOST_LIB,
            HOST_SRC]


def command():
    return [NVCC, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
            "-Xcompiler", "-fPIC", "-shared", "-cudart", "static", "-o", LIB, SRC]


def needs_build():
    return (not os.path.exists(LIB)) or os.path.getmtime(LIB) < max(
        os.path.getmtime(SRC), os.path.getmtime(os.path.abspath(__file__)))


def build(force=False):
    if force or not os.path.exists(HOST_LIB) or os.path.getmtime(HOST_LIB) < os.path.getmtime(
            HOST_SRC):
        subprocess.run(host_command(), check=True)
    if force or needs_build():
        subprocess.run(command(), check=True)
    return LIB


def build_host():
    """Only the host generator (no nvcc needed)."""
    if not os.path.exists(HOST_LIB) or os.path.getmtime(HOST_LIB) < os.path.getmtime(HOST_SRC):
        subprocess.run(host_command(), check=True)
    return HOST_LIB


if __name__ == "__main__":
    print(build(force=True))
