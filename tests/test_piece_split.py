"""Host-side checks of the operand split the fp32-compute path's tensor-core
contraction uses: x = h + m + l with h = bf16(x), m = bf16(x - h),
l = bf16(x - h - m), each rounded to nearest even and each difference taken in
fp32.  Three pieces hold every fp32 value exactly (24 bits), so the six piece
products with i + j < 3 carry an fp32 product to about 2^-24; two pieces hold
16 bits.  No GPU: torch's bf16 rounding is the same round-to-nearest-even the
kernel's conversion performs."""
import numpy as np
import torch


def split(x32, n):
    """Pieces of fp32 array x32 as fp32 arrays, in the kernel's order."""
    pieces = []
    r = torch.from_numpy(x32.copy())
    for _ in range(n):
        h = r.to(torch.bfloat16).to(torch.float32)
        pieces.append(h)
        r = r - h  # exact: h is r rounded to 8 significant bits
    return [p.numpy() for p in pieces], r.numpy()


def sample(seed=0, n=200_000):
    """fp32 values over 120 binades, with zero, +-1 and the range's ends.
    The split is exact for 2^-110 <= |x| <= 2^127: the third piece (16 bits
    below the first) is still a normal number, and the first piece does not
    round up past bf16's largest finite value; the path's operands
    (features, states, gradients) are far inside that range."""
    g = np.random.default_rng(seed)
    mant = g.uniform(-1.0, 1.0, n)
    expo = g.integers(-60, 60, n)
    x = (mant * np.exp2(expo)).astype(np.float32)
    return np.concatenate([x, np.float32([0.0, 1.0, -1.0, 2.0 ** 127, -2.0 ** -110])])


def test_three_pieces_are_exact():
    x = sample()
    (h, m, l), rest = split(x, 3)
    assert np.all(rest == 0)
    # the sum of the pieces, in fp64, is x exactly
    assert np.array_equal(h.astype(np.float64) + m + l, x.astype(np.float64))
    # each piece is a bf16 value (low 16 bits of its fp32 pattern are zero)
    for p in (h, m, l):
        assert np.all(p.view(np.uint32) & 0xFFFF == 0)


def test_two_pieces_hold_16_bits():
    x = sample(1)
    (h, m), rest = split(x, 2)
    nz = x != 0
    rel = np.abs(rest[nz].astype(np.float64)) / np.abs(x[nz].astype(np.float64))
    assert rel.max() <= 2.0 ** -16


def test_piece_products_are_exact_in_fp32():
    """bf16 x bf16 has at most 16 significant bits, so the tensor core's
    products of pieces are exact in its fp32 accumulator's format."""
    g = np.random.default_rng(2)
    a = g.standard_normal(10_000).astype(np.float32)
    b = g.standard_normal(10_000).astype(np.float32)
    (ah, am, al), _ = split(a, 3)
    (bh, bm, bl), _ = split(b, 3)
    for p, q in ((ah, bh), (ah, bm), (am, bh), (ah, bl), (am, bm), (al, bh)):
        prod64 = p.astype(np.float64) * q.astype(np.float64)
        assert np.array_equal(prod64.astype(np.float32).astype(np.float64), prod64)


def test_six_products_reach_fp32_accuracy():
    """Summing the six piece products with i + j < 3 (smallest first, fp32
    accumulation) gives a dot product within a few fp32 ulps of the fp64
    one; with two pieces (three products) about 2^-16."""
    g = np.random.default_rng(3)
    k = 128
    A = g.standard_normal((64, k)).astype(np.float32)
    B = g.standard_normal((k, 64)).astype(np.float32)
    ref = A.astype(np.float64) @ B.astype(np.float64)
    scale = np.abs(A).astype(np.float64) @ np.abs(B).astype(np.float64)
    for n, bound in ((3, 2.0 ** -20), (2, 2.0 ** -14)):
        Ap, _ = split(A, n)
        Bp, _ = split(B, n)
        acc = np.zeros((64, 64), dtype=np.float32)
        for o in range(n - 1, -1, -1):
            for i in range(o + 1):
                acc = (acc.astype(np.float64) + Ap[i].astype(np.float64) @ Bp[o - i]).astype(np.float32)
        err = np.abs(acc.astype(np.float64) - ref) / scale
        assert err.max() <= bound, (n, err.max())
