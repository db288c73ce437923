"""The float32 arithmetic the 8-bit GEMM relies on, checked with numpy's
IEEE float32 (no GPU).

- A run of products of 8-bit codes (|c| <= 127) summed in float32 is exact
  while every partial sum is an integer below 2^24: a run of 512 K stays
  below 512 * 127^2 < 2^23, and one past 2^24 / 127^2 = 1040.2 K is not.
- The conversion by one add: for an integer v with |v| <= 2^22,
  fl(v + 1.5 * 2^23) is exact and its bits are 0x4B400000 + v; one past
  the bound on either side it is not.
- Run values with that offset, summed in wrapping 32-bit arithmetic, give
  the exact int32 total once runs * 0x4B400000 is subtracted.
"""

import numpy as np

MAGIC = np.float32(12582912.0)          # 1.5 * 2^23
OFFSET = 0x4B400000


def f32_sequential_sum(x):
    acc = np.float32(0)
    for v in x:
        acc = np.float32(acc + np.float32(v))
    return acc


def magic_bits(v):
    return (np.asarray(v, np.float32) + MAGIC).astype(np.float32).view(np.uint32).astype(np.int64)


def test_run_sum_exact_below_2_24():
    for n in (256, 512, 1040):
        prods = np.full(n, 127 * 127, np.int64)
        assert int(f32_sequential_sum(prods)) == 127 * 127 * n < 2 ** 24
    # past the bound the running sum leaves the exactly representable integers
    prods = np.full(1100, 127 * 127, np.int64)
    assert int(f32_sequential_sum(prods)) != 127 * 127 * 1100
    rng = np.random.default_rng(0)
    for _ in range(20):                              # mixed signs, any order
        prods = rng.integers(-127, 128, 512) * rng.integers(-127, 128, 512)
        assert int(f32_sequential_sum(prods)) == int(prods.sum())


def test_add_conversion_identity():
    B = 2 ** 22
    v = np.concatenate([np.arange(-B, -B + 1000), np.arange(-1000, 1001), np.arange(B - 1000, B + 1),
                        np.random.default_rng(1).integers(-B, B + 1, 100000)])
    assert np.array_equal(magic_bits(v), OFFSET + v)
    # a run of 256 K is inside the bound, one of 512 K is not
    assert 256 * 127 * 127 <= B < 512 * 127 * 127
    for out in (B + 1, -B - 1):
        assert magic_bits([out])[0] != OFFSET + out


def test_wrapping_offset_sum():
    rng = np.random.default_rng(2)
    B = 2 ** 22
    for runs in (1, 2, 8, 16, 64):
        v = rng.integers(-B, B + 1, (runs, 1000))
        acc = np.zeros(1000, np.uint32)
        for r in range(runs):
            acc = (acc + magic_bits(v[r]).astype(np.uint32)).astype(np.uint32)   # wraps mod 2^32
        total = (acc - np.uint32((runs * OFFSET) % 2 ** 32)).astype(np.uint32).view(np.int32)
        exact = v.sum(axis=0)
        ok = np.abs(exact) < 2 ** 31
        assert np.array_equal(total[ok].astype(np.int64), exact[ok])
