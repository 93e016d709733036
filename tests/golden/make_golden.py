"""Write tests/golden/oracle_tiny_*.txt: oracle outputs on a tiny seeded workload.

These files are regression fixtures for the oracle itself: they are written by
this script, which calls only ``oracle`` and the seeded input generator in
``workloads``.  A change of the oracle's arithmetic that moves them must cite
the passage of the paper (or the reading of it) that justifies it.

    python tests/golden/make_golden.py
"""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import workloads  # noqa: E402

HERE = os.path.dirname(os.path.abspath(__file__))
TINY = workloads.small_case(B=1, D=3, N=2, H=2, W=3, seed=99)


def tiny_outputs():
    inp = workloads.make_inputs(TINY)
    u, yf, outf = oracle.ss2d_full(inp)
    _, ym, ybar, outm = oracle.ss2d_mean(inp)
    return {"u": u, "y_full": yf, "out_full": outf, "y_mean": ym, "ybar": ybar, "out_mean": outm}


def main():
    for name, arr in tiny_outputs().items():
        path = os.path.join(HERE, f"oracle_tiny_{name}.txt")
        with open(path, "w") as f:
            f.write(f"# oracle output '{name}' on workloads.small_case(B=1, D=3, N=2, H=2, W=3, seed=99)\n")
            f.write(f"# shape {' '.join(str(s) for s in arr.shape)}; written by tests/golden/make_golden.py\n")
            for v in arr.reshape(-1):
                f.write(f"{v:.17e}\n")


if __name__ == "__main__":
    main()
