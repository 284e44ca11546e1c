"""Build the fp64 CPU oracle (test infrastructure) into oracle/libsn_oracle.so.

Plain gcc; no fused multiply-add so x86-64 and aarch64 produce the same bits.
"""
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "sn_oracle.c")
LIB = os.path.join(HERE, "libsn_oracle.so")

CFLAGS = ["-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
          "-Wall", "-Wextra"]


def build(src=SRC, out=LIB, extra_flags=()):
    """Compile `src` into the shared library `out` (rebuilds only when stale)."""
    if (os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src)
            and os.path.getmtime(out) >= os.path.getmtime(os.path.join(HERE, "sn_oracle.h"))
            and not extra_flags):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", *CFLAGS, "-I", HERE, *extra_flags, src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build())
    sys.exit(0)
