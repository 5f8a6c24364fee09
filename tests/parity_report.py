"""Worst per-matrix error of libslorr against the fp64 oracle, per weight set,
operand mode and variant (a report for the GPU machine, not a test).

Each (set, operand mode, variant) is one forward + backward of the whole set
through the C ABI (`Regularizer`), as bench.py times it; the listed matrices'
values and gradients are compared with `oracle.reg_single` by the parity
tests' own error measure (relative Frobenius error of the gradient, against
the first Hoyer term where the two terms cancel).

    python tests/parity_report.py [--json out.json]
"""

import argparse
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)

import numpy as np  # noqa: E402

import oracle  # noqa: E402
import workloads  # noqa: E402

SETS = [("resnet18", None), ("vit_b16", (0, 1, 2, 3, 47)), ("vit_l16", (0, 1, 2, 3, 95)),
        ("decoder_560m", (0, 1, 2, 4, 6, 164))]
COMPUTES = ("fp16", "bf16", "bf16_split")
VARIANTS = ("hoyer", "nuclear")
EPS = 1e-7


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--json", default=None, help="also write the table as JSON here")
    args = ap.parse_args()
    import torch
    from paper_2607_08754_gb300.slorr import Regularizer
    from test_gpu_parity import grad_err
    co = oracle.pe_coefficients(6)
    out = {}
    for name, samples in SETS:
        shapes = workloads.shapes(name)
        idx = range(len(shapes)) if samples is None else samples
        refs = {}
        for variant in VARIANTS:
            for i in idx:
                W = workloads.generate_one(name, i).astype(np.float64)
                refs[(variant, i)] = (W,) + oracle.reg_single(W, variant, co, EPS)[:2]
        for compute in COMPUTES:
            for variant in VARIANTS:
                reg = Regularizer(shapes, variant=variant, compute=compute, lam=1.0)
                w = [torch.from_numpy(workloads.generate_one(name, i)).cuda() for i in range(len(shapes))]
                g = [torch.zeros_like(x) for x in w]
                per = torch.empty(len(shapes), device="cuda")
                reg(w, g, per_matrix=per)
                torch.cuda.synchronize()
                assert reg.status() == 0, (name, compute, variant)
                per = per.double().cpu().numpy()
                ge = le = 0.0
                for i in idx:
                    W, L, G = refs[(variant, i)]
                    ge = max(ge, grad_err(g[i].double().cpu().numpy(), G, W, variant, 1.0, 1.0))
                    le = max(le, abs(per[i] - L) / abs(L))
                out[f"{name} {compute} {variant}"] = {"grad": ge, "value": le}
                print(f"{name:14s} {compute:10s} {variant:8s} grad {ge:.2e} value {le:.2e}", flush=True)
                del w, g, reg
                torch.cuda.empty_cache()
    if args.json:
        with open(args.json, "w") as f:
            json.dump(out, f, indent=1)


if __name__ == "__main__":
    main()
