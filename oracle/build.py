"""Builds the oracle's C library with the host C compiler (test infrastructure).

Outputs oracle/_build/liborc.so (fp32 accumulation: the reference) and liborc_f64acc.so
(the same code with fp64 accumulators, used by tests only to measure the logit drift between
two valid summation orders).  Flags: -O3, -fopenmp to spread output features over cores (each
dot product still runs on one thread in one fixed order), -ffp-contract=off so no product is
fused into an add: every operation rounds once, identically on x86-64 and aarch64.
"""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "pbd_oracle.c")
OUT_DIR = os.path.join(HERE, "_build")
LIBS = {"f32": os.path.join(OUT_DIR, "liborc.so"), "f64acc": os.path.join(OUT_DIR, "liborc_f64acc.so")}
LIB = LIBS["f32"]


def build(force: bool = False, variant: str = "f32") -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    lib = LIBS[variant]
    if not force and os.path.exists(lib) and os.path.getmtime(lib) >= os.path.getmtime(SRC):
        return lib
    tmp = lib + ".tmp.%d" % os.getpid()
    cmd = ["gcc", "-O3", "-fopenmp", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           "-std=c11", "-Wall", "-o", tmp, SRC, "-lm"]
    if variant == "f64acc":
        cmd.insert(1, "-DORC_ACC_DOUBLE")
    subprocess.run(cmd, check=True)
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(force=True), build(force=True, variant="f64acc"))
