"""Loader of tests/golden/compare_cases.txt (hand-computed Eq. 1 verdicts)."""
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
BYTES = {"f32": 4, "f16": 2, "bf16": 2, "i32": 4, "i64": 8, "u32": 4}
NP_UINT = {2: np.uint16, 4: np.uint32, 8: np.uint64}


def load_compare_cases():
    cases = []
    with open(os.path.join(HERE, "golden", "compare_cases.txt")) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            lhs, rhs = line.split("->")
            dt, xb, yb, atol, rtol, eqn = lhs.split()
            match, nd, idis, mabs = rhs.split()
            cases.append(dict(dtype=dt, x=int(xb, 16), y=int(yb, 16), atol=float(atol), rtol=float(rtol),
                              equal_nan=bool(int(eqn)), match=int(match), nan_disagree=int(nd),
                              inf_disagree=int(idis), max_abs_u64=int(mabs, 0)))
    return cases


def case_arrays(c):
    """(cand_bytes, ref_bytes) of a one-element pair."""
    t = NP_UINT[BYTES[c["dtype"]]]
    return np.array([c["x"]], dtype=t).view(np.uint8), np.array([c["y"]], dtype=t).view(np.uint8)
