"""The replay kernel's division-free quotient n / c (replay.cu, DivTable and divq).

The element walks of matrix instructions take row and column of element n of a matrix
with c columns as q = (n * ceil(2^20 / c)) >> 20 in 32-bit unsigned arithmetic.  This
checks, over the whole domain the kernel uses (element indices below 4096 of matrices
at most 64 x 64, strides of up to 256 threads, divisors 1..255), that q equals the
integer quotient and that the product never wraps.
"""
import re
import os

import numpy as np

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                   "paper_2607_03574_gb300", "csrc", "replay.cu")


def test_quotient_is_exact_on_the_kernel_domain():
    n = np.arange(4096, dtype=np.uint64)[:, None]
    c = np.arange(1, 256, dtype=np.uint64)[None, :]
    m = ((1 << 20) + c - 1) // c
    prod = n * m
    assert (prod < (1 << 32)).all()
    assert ((prod >> 20) == n // c).all()


def test_kernel_uses_the_checked_constants():
    src = open(SRC).read()
    assert "m[c] = ((1u << 20) + c - 1) / c;" in src
    assert re.search(r"\(\(uint32_t\)n \* m\) >> 20", src)
    assert "constexpr int kMaxDim = 64;" in open(SRC.replace("replay.cu", "tape.h")).read()
