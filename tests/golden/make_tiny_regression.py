"""Write tiny_oracle.json: the oracle's selection on the seeded tiny workload.

The file is a regression record of the oracle itself (2 layers, 4 kv-heads,
640 tokens, window 32, pool 7, budget 64, seed 0): per (layer, kv-head) the
kept positions, lambda of Eq. 15, the score gap at the top-K boundary and
the scores S of Eq. 16 at 16 fixed positions.  It is written by this script
from the oracle alone, so a later change to the oracle's arithmetic shows
up in tests/test_golden.py and has to be justified by the paper before the
record is rewritten.

    python tests/golden/make_tiny_regression.py
"""

import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2606_14782_gb300 import workloads  # noqa: E402  (seeded inputs only)

SAMPLE = [0, 1, 15, 16, 17, 100, 200, 255, 300, 420, 512, 590, 591, 592, 606, 607]


def compute():
    wl = workloads.CONFIGS["tiny"]
    x = workloads.generate(wl, seed=0, device="cpu")
    qb, kb, vb = (workloads.bf16_bits(t) for t in (x.qwin, x.k, x.v))
    budget = wl.budgets[0]
    ref = oracle.compress(qb, kb, vb, budget, oracle.Params(pool_kernel=wl.pool),
                          threads=1, keep_scores=True)
    units = []
    for (r, l, h) in sorted(ref):
        o = ref[(r, l, h)]
        units.append({"request": r, "layer": l, "kv_head": h,
                      "idx": [int(i) for i in o["idx"]],
                      "lambda": float(o["lambda"]), "gap": float(o["gap"]),
                      "S_sample": [float(o["S"][i]) for i in SAMPLE]})
    return {"workload": "tiny: 2 layers, 4/4 heads, d 64, N 640, W 32, pool 7, budget 64, seed 0",
            "S_positions": SAMPLE, "units": units}


if __name__ == "__main__":
    rec = compute()
    units = rec.pop("units")
    with open(os.path.join(HERE, "tiny_oracle.json"), "w") as f:
        head = json.dumps(rec)[:-1]
        f.write(head + ', "units": [\n')
        f.write(",\n".join(json.dumps(u) for u in units))
        f.write("\n]}\n")
