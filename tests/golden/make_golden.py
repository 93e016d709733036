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
    dA, dBu = oracle.discretise(u, inp.draw, inp.A, inp.Bs, inp.bias)
    dAm, dBum = oracle.discretise_mean(u, inp.draw, inp.A, inp.Bs, inp.bias)
    _, ybar_g = oracle.mean_scan_grouped(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, 3)
    rng = np.random.default_rng(5)  # selection weights: K = 4, D = 3, N = 2, R = 2
    ws = [rng.standard_normal(s) for s in ((4, 2, 3), (4, 2, 3), (4, 2, 3), (4, 3, 2))]
    sel_dr, sel_B, _ = oracle.selection(u, *ws)
    return {"u": u, "y_full": yf, "out_full": outf, "y_mean": ym, "ybar": ybar, "out_mean": outm,
            "dA": dA, "dBu": dBu, "scan_only": oracle.scan_only(dA, dBu, inp.Cs),
            "scan_only_mean": oracle.scan_only(dAm, dBum, inp.Cs), "ybar_grouped3": ybar_g,
            "selection_delta": sel_dr, "selection_B": sel_B}


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
