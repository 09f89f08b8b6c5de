"""Write tests/golden/*.json: fp64 oracle outputs on small, hand-written inputs.

The paper prints no numeric worked example for the layer core, so these
fixtures are regression anchors, not paper values: they are produced by this
script from the oracle alone (``oracle.scan``, ``oracle.rollback``) and guard
against any later, unjustified change of the oracle's arithmetic. The inputs
are spelled out below so that the fixtures can be recomputed by hand.

Run:  python tests/golden/make_golden.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import numpy as np  # noqa: E402

import oracle  # noqa: E402

# Layer core with batch 1, L = 4, d_inner = 2, d_state = 2 (Eq. 2-3; Table 6
# output and gating rows; Euler B as Mamba uses it).
CASE = dict(
    x=[[[0.5, -1.0], [1.0, 0.25], [-0.75, 2.0], [0.125, -0.5]]],
    z=[[[1.0, -0.5], [0.0, 2.0], [0.5, 0.5], [-1.0, 1.5]]],
    dt=[[[0.0, -1.0], [0.5, -2.0], [-0.25, 1.0], [1.5, 0.0]]],
    B=[[[1.0, -0.5], [0.25, 2.0], [-1.0, 0.5], [0.75, 0.0]]],
    C=[[[0.5, 1.0], [-1.0, 0.25], [2.0, -0.5], [1.0, 1.0]]],
    A=[[-1.0, -2.0], [-0.5, -3.0]],
    D=[1.0, -0.25],
    dt_bias=[-1.0, 0.5],
    h0=[[[0.1, -0.2], [0.3, 0.0]]],
    accept=[2],
)


def main():
    a = {k: np.array(v, dtype=np.float64) for k, v in CASE.items() if k != "accept"}
    y, h_last, h_all = oracle.scan(a["x"], a["dt"], a["B"], a["C"], a["A"], z=a["z"], D=a["D"],
                                   dt_bias=a["dt_bias"], h0=a["h0"], want_h_all=True)
    kept = oracle.rollback(a["h0"], h_all, np.array(CASE["accept"], dtype=np.int32))
    out = dict(source="oracle.scan / oracle.rollback (fp64), Euler B; see make_golden.py",
               inputs=CASE, y=y.tolist(), h_last=h_last.tolist(), h_all=h_all.tolist(),
               rollback=kept.tolist())
    with open(os.path.join(HERE, "tiny_scan.json"), "w") as f:
        json.dump(out, f, separators=(",", ":"))
        f.write("\n")


if __name__ == "__main__":
    main()
