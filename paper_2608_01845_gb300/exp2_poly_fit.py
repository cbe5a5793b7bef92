"""Fits the polynomial the tcgen05 attention uses for part of its softmax
exponentials on the FMA pipe.

2^x is evaluated by Cody-Waite range reduction (W. J. Cody and W. Waite,
"Software Manual for the Elementary Functions", 1980): x = n + f with n the
nearest integer and f in [-1/2, 1/2], 2^x = 2^n * 2^f, where 2^n is put into
the exponent field and 2^f is a polynomial.  The polynomial here is the
degree-3 minimax approximation of 2^f on [-1/2, 1/2] in relative error,
found with the Remez exchange algorithm (E. Ya. Remez, 1934): solve for the
coefficients and the levelled error on d+2 reference points, move the
references to the extrema of the error, repeat.  The attention rounds each
result to fp16 (11 significant bits), so a relative error near 1e-4 (2^-13)
is below that rounding.

  python -m paper_2608_01845_gb300.exp2_poly_fit     # prints the coefficients
"""
import numpy as np

DEGREE = 3
LO, HI = -0.5, 0.5


def _rel_err(c, x):
    return np.polynomial.polynomial.polyval(x, c) / np.exp2(x) - 1.0


def remez(degree=DEGREE, iters=30):
    """Coefficients c[0..degree] (lowest first) minimising max |p(f)/2^f - 1|
    on [LO, HI], and that maximum."""
    m = degree + 2
    # Chebyshev extrema as the first reference set
    ref = 0.5 * (LO + HI) + 0.5 * (HI - LO) * np.cos(np.pi * np.arange(m)[::-1] / (m - 1))
    grid = np.linspace(LO, HI, 200001)
    c = None
    for _ in range(iters):
        # p(x_i) - (-1)^i E 2^{x_i} = 2^{x_i}
        A = np.zeros((m, m))
        for i, x in enumerate(ref):
            A[i, :degree + 1] = x ** np.arange(degree + 1)
            A[i, degree + 1] = -((-1) ** i) * np.exp2(x)
        sol = np.linalg.solve(A, np.exp2(ref))
        c = sol[:degree + 1]
        e = _rel_err(c, grid)
        # new references: the extremum of each sign-alternating segment
        sign = np.sign(e)
        cuts = np.flatnonzero(np.diff(sign) != 0) + 1
        segs = np.split(np.arange(len(grid)), cuts)
        ext = [s[np.argmax(np.abs(e[s]))] for s in segs if len(s)]
        if len(ext) < m:
            break
        # keep the m largest alternating extrema
        while len(ext) > m:
            a = np.abs(e[ext])
            drop = 0 if a[0] < a[-1] else len(ext) - 1
            ext.pop(drop)
        ref = grid[ext]
    return c, float(np.max(np.abs(_rel_err(c, grid))))


if __name__ == "__main__":
    c, err = remez()
    print("coefficients (lowest order first):", ", ".join(f"{v:.9e}" for v in c))
    print(f"max relative error on [{LO}, {HI}]: {err:.3e} (2^{np.log2(err):.2f})")
