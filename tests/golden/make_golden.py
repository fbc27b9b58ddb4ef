"""Writes closed_form_layer.json from the CPU oracle (and nothing else).

The fixture is the oracle's output on the hand-checkable layer of
closed_form.py; tests check the oracle still reproduces it on any machine and
that the CUDA path matches it.
"""
import json
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))

import oracle  # noqa: E402
from tests.golden.closed_form import build_case  # noqa: E402


def main():
    case = build_case()
    r = oracle.moe_decode(case["x"], case["router_w"], case["retained"],
                          case["w_gate_up"], case["w_down"], case["k"])
    doc = {
        "source": "CPU oracle on the closed-form layer of tests/golden/closed_form.py; "
                  "routing per Sec. 3.1 Eq. 2 (mask) and the renormalised top-k gates, "
                  "SwiGLU experts, gate-weighted combine",
        "idx": r["idx"].tolist(),
        "gates": [[float(v) for v in row] for row in r["gates"]],
        "out": [[float(v) for v in row] for row in r["out"]],
    }
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "closed_form_layer.json")
    with open(path, "w") as f:
        json.dump(doc, f, indent=0)
        f.write("\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
