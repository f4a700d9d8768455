"""Writes contract_vs_fp64.txt: per workload state of the GPU parity tests, the number of
scored (t, j), the largest |contract - fp64| score difference and the number of kept-set
differences between BottomK on contract scores and BottomK on fp64 scores (Sec. 4.3, Eq. 3).
Calls only the oracle and the workload generator:  python tests/golden/make_contract_vs_fp64.py"""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path[:0] = [os.path.dirname(HERE), os.path.dirname(os.path.dirname(HERE))]

import contract_fp64 as C  # noqa: E402


def main():
    lines = ["# Contract (fp32 score contract) vs fp64 cosine on the workload states of the GPU",
             "# parity tests (Sec. 4.3, Eq. 3); written by make_contract_vs_fp64.py from the oracle.",
             "# name scored max_abs_diff kept_set_differences"]
    for name, fn in C.CASES.items():
        r = fn()
        lines.append("%s %d %.3e %d" % (name, r["scored"], r["max_abs"], r["disagree"]))
        print(lines[-1], "unexplained", r["unexplained"], flush=True)
    open(os.path.join(HERE, "contract_vs_fp64.txt"), "w").write("\n".join(lines) + "\n")


if __name__ == "__main__":
    main()
