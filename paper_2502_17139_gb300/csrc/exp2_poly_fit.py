"""Coefficients of the polynomial exp2 used by the tree-attention softmax.

2^x = 2^n * 2^f with n = round(x) and f = x - n in [-1/2, 1/2].  2^f is
approximated by p(f) = 1 + c1 f + c2 f^2 + c3 f^3: the constant term is fixed
at 1 (so p(0) = 1 exactly) and c1..c3 minimise the relative error
(p(f) - 2^f) / 2^f in the least-squares sense on a dense grid of [-1/2, 1/2].
The kernel rounds P to bf16 afterwards (relative step 2^-8), so a cubic's
~1e-4 error is far below what survives.

Run:  python paper_2502_17139_gb300/csrc/exp2_poly_fit.py
"""
import numpy as np


def fit(deg=3, n=20001):
    f = np.linspace(-0.5, 0.5, n)
    y = np.exp2(f)
    A = np.stack([f ** k for k in range(1, deg + 1)], axis=1) / y[:, None]
    rhs = (y - 1.0) / y
    c, *_ = np.linalg.lstsq(A, rhs, rcond=None)
    p = 1.0 + sum(c[k - 1] * f ** k for k in range(1, deg + 1))
    return c, float(np.max(np.abs(p / y - 1.0)))


if __name__ == "__main__":
    for deg in (3, 4):
        c, err = fit(deg)
        cs = ", ".join(f"{float(np.float32(x))!r}f" for x in c)
        print(f"degree {deg}: c1..c{deg} = {cs}   max rel err {err:.3e}")
