"""Pins for the CPU oracle: checks against things other than the oracle itself.

Every check here compares the oracle with something it does not share code
with: hand-worked exact examples (tests/golden), Python's exact rational
arithmetic on tiny brute-force enumerations, the generic least-squares
optimum, the Eq. 4 closed form, torch's fp64 conv2d / max_pool2d and numpy's
matmul, and closed forms (box filter).  ``test_planted_mistakes_are_caught``
compiles copies of the oracle with one plausible mistake each and requires
that at least one pin fails for every copy.
"""
import itertools
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from conftest import read_golden

F32 = np.float32


def _fr(x):
    return Fraction(float(x))


# --------------------------------------------------------------------------
# pin functions: each takes an Oracle instance and raises AssertionError on a
# mismatch, so they can also be run against planted-mistake builds.
# --------------------------------------------------------------------------

def pin_quantize_worked_example(orc):
    g = read_golden("quantize_worked_example.txt")
    W = np.array([float(v) for v in g["W"]], dtype=F32)[None, :]
    wt, al = orc.quantize(W)
    assert wt[0].tolist() == [int(v) for v in g["codes"]]
    want = Fraction(int(g["alpha_num"][0]), int(g["alpha_den"][0]))
    assert abs(_fr(al[0]) - want) <= Fraction(1, 10**15) * want
    words = orc.pack(wt)
    assert words.shape == (1, 1) and int(words[0, 0]) == int(g["packed"][0], 16)
    J = orc.quant_error(W[0], wt[0], al[0])
    wantJ = Fraction(int(g["J_num"][0]), int(g["J_den"][0]))
    assert abs(_fr(J) - wantJ) <= Fraction(1, 10**12)


def pin_discretize_boundaries(orc):
    one_up = float(np.nextafter(F32(1), F32(2)))
    one_dn = float(np.nextafter(F32(1), F32(0)))
    m_one_dn = float(np.nextafter(F32(-1), F32(-2)))
    m_one_up = float(np.nextafter(F32(-1), F32(0)))
    tiny = float(np.nextafter(F32(0), F32(1)))
    # (value, code) per the four intervals of Eq. 3:
    # (-inf,-1) -> -2, [-1,0] -> -1, (0,1] -> 1, (1,inf) -> 2
    table = [(-1.0, -1), (-0.0, -1), (0.0, -1), (1.0, 1), (one_up, 2), (one_dn, 1),
             (m_one_dn, -2), (m_one_up, -1), (tiny, 1), (-tiny, -1), (0.5, 1),
             (-0.5, -1), (1.5, 2), (-1.5, -2), (3.0e38, 2), (-3.0e38, -2)]
    W = np.array([v for v, _ in table], dtype=F32)
    got = orc.discretize(W).tolist()
    assert got == [c for _, c in table], list(zip(W.tolist(), got))
    for v, c in table:
        assert orc.discretize_one(v) == c


def pin_alpha_is_least_squares_optimum(orc):
    # Eq. 5 is the stationary point of Eq. 4; equivalently, for fixed codes
    # the least-squares scale <W, W~> / <W~, W~>.  Computed here in exact
    # rationals from the oracle's own codes.
    rng = np.random.default_rng(11)
    for dist in range(4):
        for n in (1, 2, 5, 16, 37, 300):
            if dist == 0:
                W = rng.normal(0, 0.1, size=n)
            elif dist == 1:
                W = rng.uniform(-3, 3, size=n)
            elif dist == 2:
                W = rng.normal(0, 1.5, size=n)
            else:
                W = rng.choice([-2.5, -1.0, -0.0, 0.0, 0.25, 1.0, 1.75], size=n)
            W = W.astype(F32)
            wt = orc.discretize(W)
            a = orc.alpha(W)
            num = sum(_fr(w) * int(c) for w, c in zip(W, wt))
            den = sum(int(c) * int(c) for c in wt)
            want = num / den
            assert abs(_fr(a) - want) <= Fraction(1, 10**13) * abs(want) + Fraction(1, 10**300)


def pin_alpha_minimizes_J(orc):
    rng = np.random.default_rng(12)
    for n in (3, 9, 64, 500):
        W = rng.uniform(-2.5, 2.5, size=n).astype(F32)
        wt = orc.discretize(W)
        a = orc.alpha(W)
        J0 = orc.quant_error(W, wt, a)
        for f in (1 - 1e-3, 1 + 1e-3, 0.9, 1.1, 0.5, 2.0):
            assert J0 <= orc.quant_error(W, wt, a * f) + 1e-12


def pin_eq4_closed_form(orc):
    # Eq. 4: J(alpha) = (|B1| + 4|B2|) alpha^2 - 2 (S1 + 2 S2) alpha + sum W^2,
    # evaluated in exact rationals and compared with the oracle's direct Eq. 2.
    rng = np.random.default_rng(13)
    for n in (1, 7, 40):
        W = rng.uniform(-3, 3, size=n).astype(F32)
        wt = orc.discretize(W)
        b1 = [w for w in W if abs(w) <= 1]
        b2 = [w for w in W if abs(w) > 1]
        C = sum(_fr(w) ** 2 for w in W)
        for a in (0.3, 0.77, 1.4):
            A = _fr(a)
            J = (len(b1) + 4 * len(b2)) * A * A \
                - 2 * (sum(abs(_fr(w)) for w in b1) + 2 * sum(abs(_fr(w)) for w in b2)) * A + C
            got = orc.quant_error(W, wt, a)
            assert abs(_fr(got) - J) <= Fraction(1, 10**9) * (1 + abs(J))


def _bruteforce_min(W):
    """Joint minimum of Eq. 2 over all 4^n code vectors and alpha > 0,
    in exact rationals (alpha = max(<W,c>,0)/<c,c> for each c)."""
    Wf = [_fr(w) for w in W]
    C = sum(w * w for w in Wf)
    best = None
    for codes in itertools.product((-2, -1, 1, 2), repeat=len(W)):
        num = sum(w * c for w, c in zip(Wf, codes))
        den = sum(c * c for c in codes)
        J = C - num * num / den if num > 0 else C
        if best is None or J < best[0]:
            best = (J, codes)
    return best


def pin_bruteforce_tiny(orc):
    rng = np.random.default_rng(14)
    strictly_worse = 0
    for trial in range(12):
        n = 1 + trial % 5
        W = rng.uniform(-3, 3, size=n).astype(F32)
        wt = orc.discretize(W)
        a = orc.alpha(W)
        Jor = _fr(orc.quant_error(W, wt, a))
        Jmin, _ = _bruteforce_min(W)
        # the two-step rule can never beat the joint optimum of Eq. 2 ...
        assert Jor >= Jmin - Fraction(1, 10**9)
        # ... and, given its codes, alpha is the exact optimum over alpha
        num = sum(_fr(w) * int(c) for w, c in zip(W, wt))
        den = sum(int(c) ** 2 for c in wt)
        Jbest_given_codes = sum(_fr(w) ** 2 for w in W) - (num * num / den if num > 0 else 0)
        assert abs(Jor - Jbest_given_codes) <= Fraction(1, 10**9)
        if Jor > Jmin + Fraction(1, 10**6):
            strictly_worse += 1
    # Eq. 3 is a fixed rule ("for simplicity"), not the joint argmin of Eq. 2:
    # on the worked example the joint optimum is strictly lower.
    g = read_golden("quantize_worked_example.txt")
    W = np.array([float(v) for v in g["W"]], dtype=F32)
    Jmin, codes = _bruteforce_min(W)
    wantJ = Fraction(int(g["J_num"][0]), int(g["J_den"][0]))
    assert Jmin < wantJ
    assert list(codes) != [int(v) for v in g["codes"]]
    assert strictly_worse >= 1


def pin_exact_special_case(orc):
    g = read_golden("exact_special_case.txt")
    a0 = F32(2.0 / 3.0)
    W = np.array([a0, -a0, 2 * a0, -2 * a0], dtype=F32)
    wt = orc.discretize(W)
    assert wt.tolist() == [int(v) for v in g["codes"]]
    a = orc.alpha(W)
    assert a == float(a0)
    assert orc.quant_error(W, wt, a) == 0.0
    # and this is the joint optimum of Eq. 2 (J = 0)
    assert _bruteforce_min(W)[0] == 0


def _planar_bits(i, field):
    """Bit mask of code i's field in its word, written out per bit position:
    magnitude at 16 (l % 2) + l // 2, sign 8 above it, l = i % 16."""
    l = i % 16
    mb = 16 * (l % 2) + l // 2
    return ((field & 1) << mb) | ((field >> 1) << (mb + 8))


def pin_pack_bit_layout(orc):
    # codes 1, 2, -1, -2 (fields 0, 1, 2, 3): code 1 = pair 0 odd half ->
    # magnitude at bit 16; code 2 = pair 1 even half -> sign at bit 9;
    # code 3 = pair 1 odd half -> magnitude at bit 17 and sign at bit 25
    words = orc.pack(np.array([[1, 2, -1, -2]], dtype=np.int8))
    assert int(words[0, 0]) == (1 << 16) | (1 << 9) | (1 << 17) | (1 << 25)
    # code 15 is the odd half of pair 7 (bits 23 and 31); code 16 starts the next word
    c = np.ones((1, 17), dtype=np.int8)
    c[0, 15] = -2
    c[0, 16] = 2
    words = orc.pack(c)
    assert words.shape == (1, 2)
    assert int(words[0, 0]) == (1 << 23) | (1 << 31) and int(words[0, 1]) == 1
    # every filter starts on a fresh word; all -2 fills bytes 0,1 (pairs 0..2)
    # and bytes 2,3 (pairs 0..2) for six codes
    c2 = np.array([[1] * 5 + [-1], [-2] * 6], dtype=np.int8)
    w2 = orc.pack(c2)
    assert w2.shape == (2, 1)
    assert int(w2[0, 0]) == 1 << 26 and int(w2[1, 0]) == 0x07070707
    # each single code in each position, against the per-bit formula
    for i in range(16):
        for v, f in ((1, 0), (2, 1), (-1, 2), (-2, 3)):
            c = np.ones((1, 16), dtype=np.int8)
            c[0, i] = v
            assert int(orc.pack(c)[0, 0]) == _planar_bits(i, f), (i, v)


def pin_pack_roundtrip(orc):
    rng = np.random.default_rng(15)
    for n in (1, 15, 16, 17, 25, 33, 100, 4608):
        K = 3
        codes = rng.choice(np.array([-2, -1, 1, 2], dtype=np.int8), size=(K, n))
        words = orc.pack(codes)
        assert words.shape == (K, (n + 15) // 16)
        assert np.array_equal(orc.unpack(words, n), codes)
        rnd = rng.integers(0, 2**32, size=words.shape, dtype=np.uint64).astype(np.uint32)
        if n % 16:
            keep = 0
            for i in range(n % 16):
                keep |= _planar_bits(i, 3)
            rnd[:, -1] &= np.uint32(keep)
        assert np.array_equal(orc.pack(orc.unpack(rnd, n)), rnd)
        if n % 16:
            bad = rnd.copy()
            bad[0, -1] |= np.uint32(_planar_bits(15, 2))
            with pytest.raises(ValueError):
                orc.unpack(bad, n)


def pin_dequantized_values(orc):
    rng = np.random.default_rng(16)
    W = rng.normal(0, 1.2, size=(8, 50)).astype(F32)
    wt, al = orc.quantize(W)
    for k in range(8):
        deq = al[k] * wt[k].astype(np.float64)
        allowed = al[k] * np.array([-2.0, -1.0, 1.0, 2.0])
        assert np.all(np.isin(deq, allowed))
        assert al[k] > 0


def pin_conv_worked_example(orc):
    g = read_golden("conv_worked_example.txt")
    x = np.array([float(v) for v in g["x"]], dtype=F32).reshape(1, 1, 3, 3)
    W = np.array([float(v) for v in g["W"]], dtype=F32).reshape(1, 4)
    wt, al = orc.quantize(W)
    assert wt[0].tolist() == [int(v) for v in g["codes"]]
    want_a = Fraction(int(g["alpha_num"][0]), int(g["alpha_den"][0]))
    assert abs(_fr(al[0]) - want_a) <= Fraction(1, 10**15)
    assert int(orc.pack(wt)[0, 0]) == int(g["packed"][0], 16)
    y, bound = orc.conv2d_nchw(x, wt.reshape(1, 1, 2, 2), al)
    acc = [int(v) for v in g["acc"]]
    abs_sum = [int(v) for v in g["abs_sum"]]
    for i in range(4):
        assert abs(_fr(y.ravel()[i]) - want_a * acc[i]) <= Fraction(1, 10**14)
        assert abs(_fr(bound.ravel()[i]) - want_a * abs_sum[i]) <= Fraction(1, 10**14)


CONV_CASES = [
    # N, C, H, W, K, R, S, stride, pad
    (2, 3, 7, 9, 4, 3, 3, (1, 1), (1, 1)),
    (1, 2, 8, 8, 3, 3, 3, (2, 2), (0, 0)),
    (2, 4, 11, 10, 5, 5, 5, (2, 2), (2, 2)),
    (3, 5, 6, 6, 2, 1, 1, (1, 1), (0, 0)),
    (1, 3, 9, 7, 3, 3, 1, (1, 2), (0, 1)),
    (1, 1, 12, 12, 2, 11, 11, (4, 4), (0, 0)),
]


def _conv_inputs(case, seed):
    N, C, H, W, K, R, S, stride, pad = case
    rng = np.random.default_rng(seed)
    x = rng.normal(0, 1, size=(N, C, H, W)).astype(F32)
    Wt = rng.uniform(-2.5, 2.5, size=(K, C * R * S)).astype(F32)
    return x, Wt


def pin_conv_vs_torch(orc):
    for i, case in enumerate(CONV_CASES):
        N, C, H, W, K, R, S, stride, pad = case
        x, Wt = _conv_inputs(case, 100 + i)
        wt, al = orc.quantize(Wt)
        wt4 = wt.reshape(K, C, R, S)
        y, bound = orc.conv2d_nchw(x, wt4, al, stride, pad)
        deq = torch.from_numpy(al[:, None, None, None] * wt4.astype(np.float64))
        ref = torch.nn.functional.conv2d(torch.from_numpy(x.astype(np.float64)), deq,
                                         stride=stride, padding=pad).numpy()
        assert y.shape == ref.shape
        assert np.all(np.abs(y - ref) <= 1e-12 * (1 + bound)), case
        # bound is alpha times the conv of |x| with an all-ones filter
        ones = torch.ones((K, C, R, S), dtype=torch.float64) * torch.from_numpy(
            np.abs(al))[:, None, None, None]
        bref = torch.nn.functional.conv2d(torch.from_numpy(np.abs(x).astype(np.float64)),
                                          ones, stride=stride, padding=pad).numpy()
        assert np.allclose(bound, bref, rtol=1e-12, atol=1e-12), case


def pin_conv_vs_im2col(orc):
    case = CONV_CASES[2]
    N, C, H, W, K, R, S, stride, pad = case
    x, Wt = _conv_inputs(case, 200)
    wt, al = orc.quantize(Wt)
    y, _ = orc.conv2d_nchw(x, wt.reshape(K, C, R, S), al, stride, pad)
    P, Q = oracle.out_hw(H, W, R, S, stride, pad)
    xp = np.zeros((N, C, H + 2 * pad[0], W + 2 * pad[1]))
    xp[:, :, pad[0]:pad[0] + H, pad[1]:pad[1] + W] = x
    cols = np.empty((N, P, Q, C * R * S))
    for b in range(N):
        for p in range(P):
            for q in range(Q):
                patch = xp[b, :, p * stride[0]:p * stride[0] + R, q * stride[1]:q * stride[1] + S]
                cols[b, p, q] = patch.reshape(-1)
    ref = np.einsum("bpqj,kj->bkpq", cols, wt.astype(np.float64)) * al[None, :, None, None]
    assert np.allclose(y, ref, rtol=1e-12, atol=1e-12)


def pin_conv_sites(orc):
    case = CONV_CASES[0]
    N, C, H, W, K, R, S, stride, pad = case
    x, Wt = _conv_inputs(case, 300)
    wt, al = orc.quantize(Wt)
    wt4 = wt.reshape(K, C, R, S)
    y, bound = orc.conv2d_nchw(x, wt4, al, stride, pad)
    rng = np.random.default_rng(301)
    sites = np.stack([rng.integers(0, d, size=40) for d in y.shape], axis=1)
    ys, bs = orc.conv2d_sites(x, wt4, al, sites, stride, pad)
    assert np.array_equal(ys, y[tuple(sites.T)])
    assert np.array_equal(bs, bound[tuple(sites.T)])


def pin_box_filter(orc):
    # all weights in (0, 1] -> every code is +1 and alpha = mean(W), so the
    # layer is alpha times a box filter: sums of input windows.
    rng = np.random.default_rng(17)
    x = rng.normal(0, 1, size=(2, 2, 6, 6)).astype(F32)
    Wt = rng.uniform(0.05, 1.0, size=(3, 2 * 3 * 3)).astype(F32)
    wt, al = orc.quantize(Wt)
    assert np.all(wt == 1)
    assert np.allclose(al, Wt.astype(np.float64).mean(axis=1), rtol=1e-14)
    y, _ = orc.conv2d_nchw(x, wt.reshape(3, 2, 3, 3), al)
    for b in range(2):
        for k in range(3):
            for p in range(4):
                for q in range(4):
                    s = x[b, :, p:p + 3, q:q + 3].astype(np.float64).sum()
                    assert abs(y[b, k, p, q] - al[k] * s) <= 1e-12 * (1 + abs(al[k] * s))


def pin_linear(orc):
    rng = np.random.default_rng(18)
    B, Kin, Kout = 3, 37, 5
    x = rng.normal(0, 1, size=(B, Kin)).astype(F32)
    Wt = rng.normal(0, 1.1, size=(Kout, Kin)).astype(F32)
    wt, al = orc.quantize(Wt)
    y, bound = orc.linear(x, wt, al)
    ref = (x.astype(np.float64) @ wt.astype(np.float64).T) * al[None, :]
    assert np.allclose(y, ref, rtol=1e-12, atol=1e-12)
    assert np.allclose(bound, np.abs(x).astype(np.float64).sum(1)[:, None] * al[None, :],
                       rtol=1e-12)
    # Section 3: a fully-connected layer is a 1x1 convolution on a 1x1 image
    yc, bc = orc.conv2d_nchw(x.reshape(B, Kin, 1, 1), wt.reshape(Kout, Kin, 1, 1), al)
    assert np.array_equal(yc.reshape(B, Kout), y)
    assert np.array_equal(bc.reshape(B, Kout), bound)


def pin_glue(orc):
    rng = np.random.default_rng(19)
    x = rng.normal(0, 1, size=(2, 3, 9, 8))
    for k, s in (((2, 2), (2, 2)), ((3, 3), (2, 2))):
        ref = torch.nn.functional.max_pool2d(torch.from_numpy(x), k, s).numpy()
        assert np.array_equal(orc.maxpool2d_nchw(x, k, s), ref)
    y = rng.normal(0, 1, size=(50,))
    r = rng.normal(0, 1, size=(50,))
    assert np.array_equal(orc.epilogue(y, r, relu=True), np.maximum(y + r, 0))
    assert np.array_equal(orc.epilogue(y, None, relu=False), y)



def pin_canonical_layout(orc):
    """The canonical interchange layout: the hand-derived words of both worked
    examples (0x50AB, 0x6C: field f = m + 2 s of code i at bits 2i, 2i+1),
    round trips, the padding check, and the same field values as the
    byte-planar layout code by code."""
    gq = read_golden("quantize_worked_example.txt")
    wq = np.array([[int(v) for v in gq["codes"]]], dtype=np.int8)
    assert int(orc.pack_canonical(wq)[0, 0]) == int(gq["packed_canonical"][0], 16)
    gc = read_golden("conv_worked_example.txt")
    wc = np.array([[int(v) for v in gc["codes"]]], dtype=np.int8)
    assert int(orc.pack_canonical(wc)[0, 0]) == int(gc["packed_canonical"][0], 16)
    rng = np.random.default_rng(31)
    field = {1: 0, 2: 1, -1: 2, -2: 3}
    for n in (1, 7, 16, 17, 40, 363):
        codes = rng.choice(np.array([-2, -1, 1, 2], dtype=np.int8), size=(3, n))
        words = orc.pack_canonical(codes)
        assert words.shape == (3, (n + 15) // 16)
        assert np.array_equal(orc.unpack_canonical(words, n), codes)
        # bit positions written out from the definition
        for k in range(3):
            for i in range(n):
                f = (int(words[k, i // 16]) >> (2 * (i % 16))) & 3
                assert f == field[int(codes[k, i])]
        if n % 16:
            bad = words.copy()
            bad[0, -1] |= np.uint32(1 << 30)
            with pytest.raises(ValueError):
                orc.unpack_canonical(bad, n)
    # both layouts hold the same codes
    codes = rng.choice(np.array([-2, -1, 1, 2], dtype=np.int8), size=(4, 50))
    assert np.array_equal(orc.unpack(orc.pack(codes), 50),
                          orc.unpack_canonical(orc.pack_canonical(codes), 50))


def pin_maxpool_padding(orc):
    """Max pooling with padding (ResNet-18's 3x3/2, pad 1) against torch,
    including all-negative inputs, where a zero pad would wrongly win."""
    rng = np.random.default_rng(32)
    for shape, k, st, pd in (((2, 3, 9, 8), (3, 3), (2, 2), (1, 1)),
                             ((1, 2, 7, 7), (3, 3), (2, 2), (1, 1)),
                             ((1, 1, 6, 5), (2, 3), (1, 2), (1, 0))):
        x = rng.normal(0, 1, size=shape) - 3.0
        ref = torch.nn.functional.max_pool2d(torch.from_numpy(x), k, st, pd).numpy()
        assert np.array_equal(orc.maxpool2d_nchw(x, k, st, pd), ref)


def pin_dense_layers(orc):
    """The full-precision first convolution, global average pool and last
    fully-connected layer: the hand-worked example, torch's fp64 conv2d, numpy
    means and matmuls."""
    g = read_golden("conv_worked_example.txt")
    x = np.array([float(v) for v in g["x"]], dtype=F32).reshape(1, 1, 3, 3)
    W = np.array([float(v) for v in g["W"]], dtype=F32).reshape(1, 1, 2, 2)
    y, bound = orc.dense_conv2d_nchw(x, W)
    assert y.ravel().tolist() == [float(v) for v in g["dense_y"]]
    assert bound.ravel().tolist() == [float(v) for v in g["dense_abs"]]
    rng = np.random.default_rng(33)
    for N, C, H, Wd, K, R, S, st, pd in ((2, 3, 15, 13, 4, 7, 7, (2, 2), (3, 3)),
                                        (1, 2, 8, 9, 3, 3, 1, (1, 2), (1, 0))):
        x = rng.normal(0, 1, size=(N, C, H, Wd)).astype(F32)
        w = rng.normal(0, 0.3, size=(K, C, R, S)).astype(F32)
        y, bound = orc.dense_conv2d_nchw(x, w, st, pd)
        xt, wt_ = torch.from_numpy(x.astype(np.float64)), torch.from_numpy(w.astype(np.float64))
        ref = torch.nn.functional.conv2d(xt, wt_, stride=st, padding=pd).numpy()
        mag = torch.nn.functional.conv2d(xt.abs(), wt_.abs(), stride=st, padding=pd).numpy()
        assert np.allclose(y, ref, rtol=1e-12, atol=1e-12)
        assert np.allclose(bound, mag, rtol=1e-12, atol=1e-12)
    x = rng.normal(0, 1, size=(3, 5, 7, 6))
    assert np.allclose(orc.avgpool_global_nchw(x), x.mean(axis=(2, 3)), rtol=1e-14, atol=1e-15)
    assert np.array_equal(orc.avgpool_global_nchw(np.full((1, 2, 4, 4), 2.5)),
                          np.full((1, 2), 2.5))
    xb = rng.normal(0, 1, size=(4, 37)).astype(F32)
    wb = rng.normal(0, 0.2, size=(9, 37)).astype(F32)
    y, bound = orc.dense_linear(xb, wb)
    xd, wd = xb.astype(np.float64), wb.astype(np.float64)
    assert np.allclose(y, xd @ wd.T, rtol=1e-12, atol=1e-12)
    assert np.allclose(bound, np.abs(xd) @ np.abs(wd).T, rtol=1e-12, atol=1e-12)
    # a fully-connected layer is a 1x1 convolution on a 1x1 image
    yc, bc = orc.dense_conv2d_nchw(xb.reshape(4, 37, 1, 1), wb.reshape(9, 37, 1, 1))
    assert np.array_equal(yc.reshape(4, 9), y) and np.array_equal(bc.reshape(4, 9), bound)


BWD_CASES = [
    # N, C, H, W, K, R, S, stride, pad
    (2, 3, 7, 6, 4, 3, 2, (2, 1), (1, 1)),
    (1, 2, 9, 9, 3, 3, 3, (1, 1), (1, 1)),
    (2, 4, 8, 5, 5, 3, 3, (2, 2), (0, 1)),
    (1, 1, 6, 7, 2, 1, 1, (1, 1), (0, 0)),
]


def _bwd_case(orc, case, seed):
    N, C, H, W, K, R, S, st, pd = case
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((N, C, H, W)).astype(F32)
    wt = rng.choice(np.array([-2, -1, 1, 2], dtype=np.int8), size=(K, C, R, S))
    al = rng.random(K) + 0.25
    y, _ = orc.conv2d_nchw(x, wt, al, st, pd)
    dy = rng.standard_normal(y.shape).astype(F32)
    return x, wt, al, y, dy


def pin_bwd_adjoint(orc):
    """<conv(x, W^), dy> = <x, dx> = <W^, dW^>: both gradients are the
    adjoints of the (pinned) forward convolution, which is linear in x and
    in W^ = alpha W~."""
    for i, case in enumerate(BWD_CASES):
        x, wt, al, y, dy = _bwd_case(orc, case, 40 + i)
        st, pd = case[7], case[8]
        dx, bx = orc.conv2d_bwd_data(dy, wt, al, x.shape[2:], st, pd)
        dw, bw = orc.conv2d_bwd_filter(x, dy, wt.shape[2:], st, pd)
        w_hat = al[:, None, None, None] * wt
        ref = float((y * dy).sum())
        scale = float((np.abs(y) * np.abs(dy)).sum())
        assert abs(float((x.astype(np.float64) * dx).sum()) - ref) <= 1e-12 * scale
        assert abs(float((w_hat * dw).sum()) - ref) <= 1e-12 * scale
        assert np.all(bx >= np.abs(dx) - 1e-12) and np.all(bw >= np.abs(dw) - 1e-12)


def pin_bwd_vs_torch(orc):
    """torch's fp64 conv2d_input / conv2d_weight (autograd's routines) give
    the same gradients."""
    for i, case in enumerate(BWD_CASES):
        x, wt, al, y, dy = _bwd_case(orc, case, 50 + i)
        st, pd = case[7], case[8]
        dx, _ = orc.conv2d_bwd_data(dy, wt, al, x.shape[2:], st, pd)
        dw, _ = orc.conv2d_bwd_filter(x, dy, wt.shape[2:], st, pd)
        w_hat = torch.from_numpy(al[:, None, None, None] * wt.astype(np.float64))
        g = torch.from_numpy(dy.astype(np.float64))
        xt = torch.from_numpy(x.astype(np.float64))
        dx_t = torch.nn.grad.conv2d_input(xt.shape, w_hat, g, stride=st, padding=pd)
        dw_t = torch.nn.grad.conv2d_weight(xt, w_hat.shape, g, stride=st, padding=pd)
        assert np.allclose(dx, dx_t.numpy(), rtol=1e-12, atol=1e-12)
        assert np.allclose(dw, dw_t.numpy(), rtol=1e-12, atol=1e-12)


def pin_all_zero_filter(orc):
    # Eq. 5 with every W_i = 0: numerator 0, denominator n -> alpha = 0 (the
    # paper asks alpha > 0; the formula's value is kept), codes all -1.
    W = np.zeros((1, 20), dtype=F32)
    wt, al = orc.quantize(W)
    assert np.all(wt == -1) and al[0] == 0.0


PINS = [pin_quantize_worked_example, pin_discretize_boundaries,
        pin_alpha_is_least_squares_optimum, pin_alpha_minimizes_J, pin_eq4_closed_form,
        pin_bruteforce_tiny, pin_exact_special_case, pin_pack_bit_layout, pin_pack_roundtrip,
        pin_dequantized_values, pin_conv_worked_example, pin_conv_vs_torch,
        pin_conv_vs_im2col, pin_conv_sites, pin_box_filter, pin_linear, pin_glue,
        pin_all_zero_filter, pin_bwd_adjoint, pin_bwd_vs_torch, pin_canonical_layout,
        pin_maxpool_padding, pin_dense_layers]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_oracle_pin(pin):
    pin(oracle.default())


# Plausible mistakes, one per copy of the oracle source: (description,
# original text, replacement).  Each must make at least one pin fail.
MUTANTS = [
    ("strict lower interval of Eq. 3", "if (-1.0 <= w && w <= 0.0)", "if (-1.0 < w && w <= 0.0)"),
    ("zero mapped to +1", "if (-1.0 <= w && w <= 0.0)", "if (-1.0 <= w && w < 0.0)"),
    ("one mapped to +2", "if (0.0 < w && w <= 1.0)", "if (0.0 < w && w < 1.0)"),
    ("B1 uses strict inequality", "if (a <= 1.0) {", "if (a < 1.0) {"),
    ("dropped factor 2 in Eq. 5 numerator", "sum_b1 + 2.0 * sum_b2", "sum_b1 + sum_b2"),
    ("factor 2 instead of 4 in Eq. 5 denominator", "(double)size_b1 + 4.0 * (double)size_b2",
     "(double)size_b1 + 2.0 * (double)size_b2"),
    ("sign/magnitude bits swapped", "case 2:  *field = 1u; return 0;\n    case -1: *field = 2u;",
     "case 2:  *field = 2u; return 0;\n    case -1: *field = 1u;"),
    ("codes 0-7 in the low half-word instead of even/odd halves",
     "return (int)(16 * (l % 2) + l / 2);", "return (int)(16 * (l / 8) + l % 8);"),
    ("sign bit next to the magnitude bit", "return magnitude_bit(i) + 8;",
     "return magnitude_bit(i) + 1;"),
    ("padding ignored in the row index", "int64_t h = p * sh - ph + r;", "int64_t h = p * sh + r;"),
    ("convolution instead of cross-correlation",
     "double wv = (double)wt[((k * C + c) * R + r) * S + s];",
     "double wv = (double)wt[((k * C + c) * R + (R - 1 - r)) * S + (S - 1 - s)];"),
    ("alpha not applied", "*y_out = alpha[k] * acc;", "*y_out = acc;"),
    ("transposed linear operand", "acc += xv * (double)wt[k * Kin + j];",
     "acc += xv * (double)wt[(j % Kout) * Kin + (k % Kin)];"),
    ("input gradient without alpha",
     "double wv = alpha[k] * (double)wt[((k * C + c) * R + r) * S + s];",
     "double wv = (double)wt[((k * C + c) * R + r) * S + s];"),
    ("input gradient with the filter taps mirrored", "dx[o] += g * wv;",
     "dx[o] += g * alpha[k] * (double)wt[((k * C + c) * R + (R - 1 - r)) * S + (S - 1 - s)];"),
    ("filter gradient ignores the stride in the row index", "int64_t h = r + p * sh - ph;",
     "int64_t h = r + p - ph;"),
    ("filter gradient sums magnitudes", "acc += t;", "acc += fabs(t);"),
    ("bound without abs", "acc += xv * wv;\n                abs_sum += fabs(xv);",
     "acc += xv * wv;\n                abs_sum += xv;"),
    ("canonical layout with the sign bit low", "words[k * wpf + i / 16] |= f << (2 * (i % 16));",
     "words[k * wpf + i / 16] |= ((f >> 1) | ((f & 1u) << 1)) << (2 * (i % 16));"),
    ("canonical layout codes in reverse order within a word",
     "return (w >> (2 * (i % 16))) & 3u;", "return (w >> (2 * (15 - i % 16))) & 3u;"),
    ("max pool padding not subtracted", "int64_t h = i * sh - ph + u, w = j * sw - pw + v;",
     "int64_t h = i * sh + u, w = j * sw + v;"),
    ("max pool padding counted as zero", "continue; /* padding never wins the max */",
     "{ if (0.0 > m) m = 0.0; continue; }"),
    ("dense convolution ignores the column stride", "int64_t w_in = q * sw - pw + s;",
     "int64_t w_in = q - pw + s;"),
    ("dense convolution bound without abs", "mag += fabs(xw);", "mag += xw;"),
    ("average over H only", "y[b * C + c] = acc / (double)(H * W);",
     "y[b * C + c] = acc / (double)H;"),
    ("dense linear transposed weight", "(double)w[k * Kin + j];",
     "(double)w[(j % Kout) * Kin + (k % Kin)];"),
]


@pytest.mark.parametrize("desc,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistakes_are_caught(tmp_path, desc, old, new):
    src = oracle.source_text()
    assert src.count(old) == 1, desc
    path = oracle.build_variant(src.replace(old, new), str(tmp_path / "mutant.so"))
    mutant = oracle.Oracle(path)
    failed = []
    for pin in PINS:
        try:
            pin(mutant)
        except (AssertionError, ValueError):
            failed.append(pin.__name__)
    assert failed, "no pin caught: " + desc
