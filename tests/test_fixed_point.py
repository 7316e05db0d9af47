"""CPU pins of the integer identities the GPU decoders rely on (no GPU, no oracle): the byte-plane
split of a fixed-point activation X with |X| < 2^22 (two unsigned planes and a signed top plane),
the exactness of sum c X through four-lane byte dot products (dp4a), the grouping of four base-3
bytes' fifth codes into one word, and the int32 headroom of a block's sums."""
import numpy as np


def planes(X):
    """X = p0 + 256 p1 + 65536 p2 with p0, p1 in [0, 255] and p2 signed (the kernels' split)."""
    X = np.asarray(X, np.int64)
    p0 = X & 0xFF
    p1 = (X >> 8) & 0xFF
    p2 = ((X >> 16) & 0xFF).astype(np.int64)
    p2 = np.where(p2 >= 128, p2 - 256, p2)  # read as a signed byte
    return p0, p1, p2


def dp4a(a4, b4):
    """sum of four byte products (the operands given as length-4 integer vectors)."""
    return int(np.dot(np.asarray(a4, np.int64), np.asarray(b4, np.int64)))


def test_planes_reassemble_every_22_bit_value():
    rng = np.random.default_rng(0)
    X = np.concatenate([rng.integers(-(1 << 22) + 1, 1 << 22, size=200000),
                        np.array([0, 1, -1, (1 << 22) - 1, -(1 << 22) + 1, 255, 256, -256, 65535, -65536])])
    p0, p1, p2 = planes(X)
    assert np.all((p0 >= 0) & (p0 <= 255) & (p1 >= 0) & (p1 <= 255))
    assert np.all((p2 >= -64) & (p2 <= 63))  # |X| < 2^22: the top plane fits a signed byte with room
    assert np.array_equal(p0 + 256 * p1 + 65536 * p2, X)


def test_plane_dot_products_give_the_exact_sum():
    """sum_j c_j X_j over a code byte's five columns and over a group of four bytes, as the base-3
    kernel forms it: per plane, one dp4a per byte for the first four columns and one dp4a over the
    four bytes' fifth columns, then 65536 s2 + 256 s1 + s0, minus S = sum X for T = c - 1."""
    rng = np.random.default_rng(1)
    for _ in range(2000):
        X = rng.integers(-(1 << 22) + 1, 1 << 22, size=20)  # four bytes x five columns
        c = rng.integers(0, 3, size=20)
        P = planes(X)
        s = [0, 0, 0]
        for pl in range(3):
            for b in range(4):
                s[pl] += dp4a(c[5 * b:5 * b + 4], P[pl][5 * b:5 * b + 4])
            s[pl] += dp4a(c[4::5], P[pl][4::5])  # the fifth columns of the four bytes
        total = 65536 * s[2] + 256 * s[1] + s[0]
        assert total == int(np.dot(c, X))
        assert total - int(X.sum()) == int(np.dot(c - 1, X))
        assert abs(total) < 2 ** 31  # one group's intermediate fits int32


def test_block_sum_headroom():
    """A 128-column block's sum_j T_j X_j is at most 128 * 2^22 = 2^29 in magnitude (int32 in the
    base-3 kernel); the batch-1 kernel's sum c X over 512 columns of 24-bit X stays below 2^33 and is
    formed in int64."""
    assert 128 * ((1 << 22) - 1) < 2 ** 29
    assert 2 * 512 * ((1 << 23) - 1) < 2 ** 33  # sum c X before the sum X correction, in int64 there

