"""Compile the fp64 CPU oracle (test infrastructure) into oracle/_build.

Plain gcc, no CUDA: the oracle shares nothing with the GPU library.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "parason_oracle.c")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "libparason_oracle.so")


def _compile(src: str, out: str) -> None:
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-fno-fast-math", "-ffp-contract=off", "-Wall", "-Wextra",
           "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)


def build_variant(source_text: str, out_dir: str, name: str) -> str:
    """Compile an edited copy of the oracle source (used by the tests that
    plant a mistake in the oracle and check that a pin catches it)."""
    os.makedirs(out_dir, exist_ok=True)
    src = os.path.join(out_dir, name + ".c")
    with open(src, "w") as f:
        f.write(source_text)
    out = os.path.join(out_dir, "lib" + name + ".so")
    _compile(src, out)
    return out


def build(force: bool = False) -> str:
    """Build the oracle shared library if it is missing or older than its source."""
    if (not force and os.path.exists(LIB)
            and os.path.getmtime(LIB) >= os.path.getmtime(SRC)):
        return LIB
    os.makedirs(OUT_DIR, exist_ok=True)
    _compile(SRC, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
