"""The divisions used by the kernel, checked in exact integer arithmetic
against Python's own division:

* occupancy: ceil(n/d) from the constant M = ceil(2^64/d) as floor(M*n / 2^64)
  plus a remainder test (Lemire, Kaser, Kurz 2019, exact for 32-bit n and d),
  at the edges and at random;
* slot -> CTA slot -> SM: floor(n/d) for n < 2^16 as floor(n*m / 2^32) with
  m = ceil(2^32/d) (0 for d = 1), exhaustively over n for every divisor the
  kernel can meet (warps per CTA <= 128) and many CTA-slot counts."""
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


def div16_method(n, d):
    m = 0 if d <= 1 else (2**32 - 1) // d + 1
    return n if m == 0 else (n * m) >> 32


def test_floor_division_below_2_16_exhaustive():
    n = np.arange(2**16, dtype=np.uint64)
    rng = np.random.default_rng(6)
    ds = list(range(1, 1025)) + [int(x) for x in rng.integers(1025, 2**20, 300)] + [2**16 - 1, 2**16, 2**31, 2**32 - 1]
    for d in ds:
        m = np.uint64(0 if d <= 1 else (2**32 - 1) // d + 1)
        q = n if d <= 1 else (n * m) >> np.uint64(32)
        assert np.array_equal(q, n // np.uint64(d)), d
    assert div16_method(65535, 3) == 21845 and div16_method(7, 1) == 7
