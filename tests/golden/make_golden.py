"""Writes tests/golden/tiny_oracle_pass.json: the oracle's update pass on the Tiny workload.

The paper prints no worked example with numbers, so the stored values are the oracle's own,
written by this script (it calls only oracle/ and the seeded input generator). They serve as a
regression record of the oracle and as expected values the CUDA path is checked against without
re-running the oracle.

    python tests/golden/make_golden.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import numpy as np  # noqa: E402

from oracle.pipeline import run, widen  # noqa: E402
from synthetic import get_config, make_batch  # noqa: E402


def main():
    cfg = get_config("tiny")
    b = make_batch(cfg)                 # host inputs (old log-probs by numpy): the tests use these too
    o = run(b.q, b.L, cfg.K, b.R, b.tok_full, b.oldlogp_full, widen(cfg, b.hid_full), widen(cfg, b.W),
            cfg.eps, cfg.loss_scale, cfg.seed, cfg.step)
    f = o["fwd"]
    N = int(o["pack"]["N"])
    rows = [0, 1, 2, 17, 100, N - 1]
    vocab = [0, 3, 500, cfg.V - 1]
    out = {
        "source": "oracle (tests/golden/make_golden.py); the paper prints no worked numeric example",
        "workload": "tiny: 2 prompts x 4 completions, lengths U[32,256], d=128, V=1024, f32, seed 0, step 0",
        "H": [int(x) for x in o["H"]],
        "N": N,
        "loss": float(f["loss"]),
        "rows": rows,
        "lse": [float(f["lse"][i]) for i in rows],
        "coef": [float(f["coef"][i]) for i in rows],
        "dH_row_sums": [float(o["dH"][i].sum()) for i in rows],
        "vocab": vocab,
        "dW_row_sums": [float(o["dW"][v].sum()) for v in vocab],
        "dW_abs_sum": float(np.abs(o["dW"]).sum()),
    }
    with open(os.path.join(HERE, "tiny_oracle_pass.json"), "w") as fh:
        json.dump(out, fh, indent=1)
        fh.write("\n")


if __name__ == "__main__":
    main()
