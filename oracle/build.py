"""Build the fp64 CPU oracle (test infrastructure only).

Compiles ``oracle/delta_oracle.c`` with gcc into ``oracle/_build/liboracle.so``.
Plain portable C: no -march flags, so the same source builds on x86_64 and on
aarch64 hosts.
"""
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "delta_oracle.c")
OUT_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(OUT_DIR, "liboracle.so")


def build(force: bool = False, extra_flags=(), out: str = LIB) -> str:
    """Compile the oracle shared library; returns its path."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(SRC) and not extra_flags):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-D_GNU_SOURCE", "-Wall", "-fPIC", "-shared", "-pthread",
           *extra_flags, "-o", tmp, SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(force=True))
