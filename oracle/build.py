"""Compile the float64 CPU oracle (test infrastructure only) with gcc.

The oracle is plain C with OpenMP. It is built without -ffast-math so the compiler keeps
the written summation order. ``plant`` builds a variant with one deliberate mistake,
which the pin tests use to show that they reject it.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "flarepp_oracle.c")
BUILD_DIR = os.path.join(HERE, "_build")


def lib_path(plant: int = 0, build_dir: str = BUILD_DIR) -> str:
    name = "libflarepp_oracle.so" if plant == 0 else f"libflarepp_oracle_plant{plant}.so"
    return os.path.join(build_dir, name)


def build(plant: int = 0, build_dir: str = BUILD_DIR, force: bool = False) -> str:
    """Build the oracle shared library and return its path (rebuilds when the source is newer)."""
    out = lib_path(plant, build_dir)
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(SRC)):
        return out
    os.makedirs(build_dir, exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
           "-ffp-contract=off", f"-DORACLE_PLANT={int(plant)}", SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(int(sys.argv[1]) if len(sys.argv) > 1 else 0, force=True))
