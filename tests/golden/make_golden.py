"""Write tests/golden/oracle_small_case.txt from the float64 oracle alone.

The stored values guard the oracle against unintended changes: a later edit of
its arithmetic must either reproduce them or regenerate them in a commit that
names the paper passage justifying the change.  Only oracle/ is called here.
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402

CASE = dict(M=3, S=4, T=9.0, L=10, d=3, seed=2024)


def case_inputs():
    g = np.random.default_rng(CASE["seed"])
    L, d = CASE["L"], CASE["d"]
    q, k, v, do = (np.round(g.standard_normal((1, 1, L, d)), 3) for _ in range(4))
    return q, k, v, do


def compute():
    q, k, v, do = case_inputs()
    r = oracle.forward(q, k, v, CASE["M"], CASE["S"], CASE["T"], form="naive", return_state=True)
    dq, dk, dv = oracle.backward(q, k, v, do, CASE["M"], CASE["S"], CASE["T"])
    return {"o": r["o"], "lse": r["lse"], "state": r["state"], "dq": dq, "dk": dk, "dv": dv}


def main():
    out = compute()
    path = os.path.join(HERE, "oracle_small_case.txt")
    with open(path, "w") as f:
        f.write("# float64 oracle (Alg. 2 forward, chain-rule VJP) on a tiny case; written by make_golden.py\n")
        f.write("# case: %s; q,k,v,dO = round(N(0,1), 3) from default_rng(seed) in that order\n" % CASE)
        for name, arr in out.items():
            f.write("%s %s\n" % (name, " ".join(repr(float(x)) for x in np.ravel(arr))))
    print(path)


if __name__ == "__main__":
    main()
