"""Builds the oracle shared library with g++ (TEST INFRASTRUCTURE ONLY).

The oracle is plain C++17 compiled with -ffp-contract=off, so that every fp32
operation it states is rounded on its own (no fused multiply-add).  A planted
mistake variant (ORACLE_MUTANT=n) is built only for the test that checks the
pins catch mistakes.
"""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "mlkv_oracle.cpp")


def lib_path(mutant: int = 0, out_dir: str | None = None) -> str:
    name = "libmlkv_oracle.so" if mutant == 0 else f"libmlkv_oracle_m{mutant}.so"
    return os.path.join(out_dir or HERE, name)


def build(mutant: int = 0, out_dir: str | None = None, force: bool = False) -> str:
    out = lib_path(mutant, out_dir)
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(SRC)
            and os.path.getmtime(out) >= os.path.getmtime(__file__)):
        return out
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", f"-DORACLE_MUTANT={mutant}", SRC, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(force=True))
