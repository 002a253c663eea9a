"""Writes oracle_golden.json: float64 oracle meta-gradients on small seeded workloads.

The paper prints no worked example with numeric values (its tables report memory and
seconds), so no fixture here comes from the paper. These values are written by the oracle
alone (`oracle/` and the seeded input generators, nothing else) and pin the oracle's own
arithmetic against silent changes: `tests/test_oracle_pins.py` recomputes them to 1e-12. A
deliberate change to the oracle's arithmetic regenerates the file, and the commit names the
passage of the paper that justifies it.

Usage: python tests/golden/make_oracle_golden.py
"""
import json
import math
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from paper_2505_00793_gb300 import synth  # noqa: E402
from oracle import metagrad as om  # noqa: E402

CASES = {
    # the loss-weighting task (Section 5) on the 16-32-1 tanh MLP, T = 4 plain SGD steps
    "tiny": synth.WORKLOADS["tiny"],
    # heavy ball with a scalar log learning rate and weight logits
    "mom_ex_slr": synth.Workload("g_mom", [5, 7, 2], "tanh", "squared", "fp32", B=4, T=3,
                                 B_outer=6, momentum=0.5, meta_kind=synth.EXAMPLE_WEIGHTS
                                 | synth.SCALAR_LOGLR, noise_std=0.1,
                                 extra={"scalar_loglr": math.log(0.3)}),
    # Adam (Section 5's inner optimiser) with per-parameter log learning rates
    "adam_plr": synth.Workload("g_adam", [4, 5, 2], "tanh", "squared", "fp32", B=5, T=3,
                               B_outer=4, meta_kind=synth.PARAM_LOGLR, optimizer="adam",
                               beta1=0.8, beta2=0.95, adam_eps=1e-2,
                               loglr_mean=math.log(0.02), loglr_std=0.1, noise_std=0.1),
    # the motivating example of Section 3 (Eq. 8), M = 3, theta_0 the meta-parameter
    "toy_m3": synth.toy("g_toy", 4, 3, 3, precision="fp32"),
}


def main():
    out = {}
    for name, w in CASES.items():
        r = om.meta_grad(w, synth.make_inputs(w))
        out[name] = {"V": r["V"], "d_eta": [float(v) for v in r["d_eta"]],
                     "d_theta0": [float(v) for v in r["d_theta0"]]}
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_golden.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
