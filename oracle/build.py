"""Compile the CPU oracle (test infrastructure) into ``oracle/liboracle.so``.

Plain gcc, no vendor code.  ``-ffp-contract=off`` keeps every multiply and add
separately rounded, so the oracle gives the same bits on x86-64 and aarch64.
"""
import os
import subprocess
import sys
import tempfile

HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(HERE, "spec_oracle.c")
LIBRARY = os.path.join(HERE, "liboracle.so")


def build(force: bool = False, extra_flags=(), output: str = LIBRARY) -> str:
    """Build the oracle library if it is missing or older than its source."""
    if (not force and os.path.exists(output)
            and os.path.getmtime(output) >= os.path.getmtime(SOURCE)):
        return output
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=os.path.dirname(output))
    os.close(fd)
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared",
           *extra_flags, SOURCE, "-o", tmp, "-lm"]
    try:
        subprocess.run(cmd, check=True)
        os.replace(tmp, output)  # atomic: concurrent builders never see a partial file
    finally:
        if os.path.exists(tmp):
            os.remove(tmp)
    return output


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
