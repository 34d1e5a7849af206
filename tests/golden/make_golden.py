"""Writes the oracle-computed fixtures of this folder. It calls only the
oracle (and the seeded input generators, which hold no method arithmetic), so
the stored values come from neither the CUDA path nor a tolerance choice.

  leduc_exact_small.txt: the exact expected first-seat payoff (enumeration of all
  deals and action sequences, Sec. 4.2's payoff-table entry without sampling
  noise) of every pair of a 2 x 2 population of fp32 MLP policies
  17-128-128-3 drawn by workloads.leduc(pop=2, hidden=128, with_bias=True,
  seed=2106075590).

Run from the repository root: python tests/golden/make_golden.py
"""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle      # noqa: E402
import workloads   # noqa: E402

LEDUC_SEED = 2106075590


def leduc_population():
    return workloads.leduc(pop=2, hidden=128, with_bias=True, seed=LEDUC_SEED)


def main():
    w = leduc_population()
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    lines = ["# Exact first-seat expected payoff of each pair (row: seat-0 policy, column:",
             "# seat-1 policy) of workloads.leduc(pop=2, hidden=128, with_bias=True,",
             f"# seed={LEDUC_SEED}); written by tests/golden/make_golden.py from oracle.leduc_exact.",
             "# Layout: pair_index seat0_id seat1_id value"]
    for k, (i, j) in enumerate(w.pair_ids):
        v = oracle.leduc_exact(params[i], params[j], dims)
        lines.append(f"{k} {int(i)} {int(j)} {v:.17g}")
    with open(os.path.join(HERE, "leduc_exact_small.txt"), "w") as f:
        f.write("\n".join(lines) + "\n")


if __name__ == "__main__":
    main()
