"""Error bounds of the binding methods, shared by the GPU parity tests and their CPU check.

Per output of block b, with ||x_b||, ||y_b|| the norms of the row's blocks:
  direct sum (fp32, L products in j order): L 2^-22 ||x_b|| ||y_b||;
  spectral method (fp32 radix-2^k transforms of the blocks, the product, the inverse):
  sqrt(2L) (3e + 4u) ||x_b|| ||y_b||, u = 2^-24, e = K eta / (1 - K eta) + 10u, eta = 10u,
  K = log2(L) + 1 for two Stockham passes (L <= 512), log2(L) + 2 for three: the radix-2 FFT
  bound ||fl(F w) - F w|| <= K eta ||F w|| (Higham, Accuracy and Stability of Numerical
  Algorithms, Thm 24.2; one extra twiddle multiply per pass) carried through the split, the
  product (max |Y_k| <= sqrt(L) ||y_b||) and the inverse transform.
"""
import numpy as np

U32 = 2.0 ** -24


def bind_error_factor(L, method):
    if method == "direct":
        return L * 2.0 ** -22
    K = int(np.log2(L)) + (1 if L <= 512 else 2)
    eta = 10 * U32
    e = K * eta / (1 - K * eta) + 10 * U32
    return np.sqrt(2 * L) * (3 * e + 4 * U32)
