"""The occupancy division used by the kernel: ceil(n/d) from the constant
M = ceil(2^64/d) as floor(M*n / 2^64) plus a remainder test (Lemire, Kaser,
Kurz 2019, exact for 32-bit n and d).  Checked here in exact integer
arithmetic against Python's own division, at the edges and at random."""
import numpy as np


def cdiv_method(n, d):
    if d == 1:
        return n
    M = (2**64 - 1) // d + 1
    q = (M * n) >> 64
    return q + (1 if q * d != n else 0)


def test_edges():
    ds = [1, 2, 3, 5, 7, 100, 128, 505, 1565, 2048, 4040, 4096, 65535, 65536, 2**31 - 1, 2**31, 2**32 - 1]
    ns = [0, 1, 2, 99, 100, 101, 49152, 1048576, 2**31 - 1, 2**31, 2**32 - 2, 2**32 - 1]
    for d in ds:
        for n in ns + [d - 1, d, d + 1, 2 * d - 1, 2 * d, (2**32 - 1) // d * d]:
            if 0 <= n < 2**32:
                assert cdiv_method(n, d) == -(-n // d), (n, d)


def test_random():
    rng = np.random.default_rng(5)
    for _ in range(20000):
        d = int(rng.integers(1, 2**32))
        n = int(rng.integers(0, 2**32))
        assert cdiv_method(n, d) == -(-n // d)
        d = int(rng.integers(1, 5000))
        assert cdiv_method(n, d) == -(-n // d)
