"""Writes eq1_pd.txt: Eq. 1's P_d (Sec. 4) for the group sizes and sparsity
ratios of Fig. 3a with an integer number of slots, computed by the oracle in
exact rational arithmetic.  Run from the repository root:
    python tests/golden/make_eq1_pd.py
"""
import os
import sys
from fractions import Fraction

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))
import oracle  # noqa: E402


def rows():
    for Ps in ("1/2", "3/4", "7/8", "15/16"):
        for G in (2, 4, 8, 16, 32, 64, 128, 256, 512, 1024):
            s = G * (1 - Fraction(Ps))
            if s.denominator == 1 and s >= 1:
                yield Ps, G, int(s), oracle.allocation_error_exact(G, Ps)


def main():
    path = os.path.join(HERE, "eq1_pd.txt")
    with open(path, "w") as f:
        f.write("# Eq. 1 (Sec. 4): P_d for group size G, sparsity Ps, s = G(1 - Ps) slots;\n")
        f.write("# written by tests/golden/make_eq1_pd.py from oracle.allocation_error_exact\n")
        f.write("# Ps G s P_d\n")
        for Ps, G, s, pd in rows():
            f.write(f"{Ps} {G} {s} {float(pd):.17g}\n")
    print(path)


if __name__ == "__main__":
    main()
