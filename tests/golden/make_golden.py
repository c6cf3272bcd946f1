"""Writes rmmc_closed_form_mu095.txt: closed-form RMMC sequences at the paper's momentum.

Run from the repository root:  python tests/golden/make_golden.py

The values are mathematics, not program output; nothing here calls the oracle or the GPU
library.  Setting: momentum mu = 0.95 (Section 4: "momentum mu = 0.95"), a constant
gradient G, M_0 = 0 and prev_norm_0 = 0 (Algorithm 2's initialization), eps -> 0.

* Dion with full rank r = min(m, n): P P^T B = B, so the error-feedback line of
  Algorithm 1 leaves M_t = mu B_t and the buffer obeys the momentum recurrence of
  Section 2.1, B_t = mu B_{t-1} + G.  Hence ||B_t|| = ||G|| (1 - mu^t) / (1 - mu) and
  RMMC_t = mu^(t-1) (1 - mu) / (1 - mu^(t-1)) for t >= 2.
* Local branch every step (Algorithm 2's else-branch, M <- B): B_t = t G, so
  RMMC_t = 1 / (t - 1) for t >= 2.
"""
import os

MU = 0.95


def dion_full_rank(t: int) -> float:
    return MU ** (t - 1) * (1.0 - MU) / (1.0 - MU ** (t - 1))


def local(t: int) -> float:
    return 1.0 / (t - 1)


def main():
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "rmmc_closed_form_mu095.txt")
    with open(path, "w") as f:
        f.write("# Closed-form RMMC_t (Algorithm 2, eps -> 0) for a constant gradient, mu = 0.95 (Section 4).\n")
        f.write("# Derivation: Section 2.1 momentum recurrence + Algorithm 1/2; see make_golden.py.\n")
        f.write("# t  dion_full_rank  local_only\n")
        for t in range(2, 13):
            f.write(f"{t} {dion_full_rank(t):.15e} {local(t):.15e}\n")


if __name__ == "__main__":
    main()
