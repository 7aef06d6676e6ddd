"""Pins of the oracle's dual-axis codec (Sec. 4.3, App. C.1, App. C.3) and of the
uniform INT-b baseline (App. B.5).

What the paper fixes and these tests check:
 * Eq. uniform_quantization: codes lie in [-q_b, q_b], q_b = 2^(b-1) - 1, and each
   is the nearest level (brute force over all levels); the error bound is half a
   quantization step for every unclipped element.
 * X_hat = r_i c_j z_ij with z = 2^(8-b) q for KDA rows (App. C.1): the normalised
   codebook reconstructs exactly what the plain codebook does.
 * r_i = m_i^(1/2) w_i^(-1/2): scaling a row by 16 quadruples r_i; scaling
   w_i by 16 divides r_i by 4.
 * The fixed-code column update is the minimiser of the w^2-weighted objective
   (checked by a 1-D search, independent of the closed form).
 * FP16 pivots equal numpy's float16 conversion.
 * The packed bit layout decodes with an independent numpy bit unpacker.
"""
import numpy as np
import pytest

D = 128
HEAD, ROW, PIV = 0, 1, 16


def _state(rng, scale=1.0):
    base = rng.standard_normal((D, D))
    return (scale * base * np.exp(rng.normal(size=(D, 1))) * np.exp(rng.normal(size=(1, D)))
            ).astype(np.float32)


def _w(rng):
    return np.exp(rng.normal(0, 0.3, D)).astype(np.float32)


def _f16(u16):
    return np.asarray(u16, np.uint16).view(np.float16).astype(np.float64)


def _widths(rng, unit, b=None):
    if unit == HEAD:
        return np.full(D, b, np.int8)
    rb = rng.choice([2, 4, 6, 8], size=D).astype(np.int8)
    rb[rng.choice(D, 9, replace=False)] = PIV
    return rb


def _head_streams(codes, b):
    """The 256 per-lane streams (8b bytes each) of a head's code region, ordered
    [column group w][lane l = 8 cg + g]: piece k (16 bytes) of lane l of group w
    sits at w * 256 b + k * 512 + 16 l."""
    return (np.asarray(codes).reshape(8, b // 2, 32, 16).transpose(0, 2, 1, 3)
            .reshape(8, 32, 8 * b))


def _check_nearest_levels(oracle, X, unit, rb, page):
    r16, c16, codes, piv = oracle.unpack_head(page, unit, rb)
    r, c = _f16(r16), _f16(c16)
    Xd = X.astype(np.float64)
    for i in range(D):
        b = int(rb[i])
        if b == PIV:
            assert np.array_equal(_f16(piv[i]), np.float16(X[i]).astype(np.float64))
            continue
        qm = 2 ** (b - 1) - 1
        zs = 2.0 ** (8 - b) if unit == ROW else 1.0
        step = r[i] * c * zs                         # [128] quantization step of row i
        q = codes[i].astype(np.float64)
        assert np.all(np.abs(q) <= qm)
        levels = np.arange(-qm, qm + 1, dtype=np.float64)
        errs = np.abs(Xd[i][:, None] - step[:, None] * levels[None, :])
        best = errs.min(axis=1)
        mine = np.abs(Xd[i] - step * q)
        # nearest level, up to fp32 rounding of the scaled value at exact ties
        assert np.all(mine <= best + 2e-6 * step * (qm + 1)), i
        inside = np.abs(Xd[i]) <= step * qm
        assert np.all(mine[inside] <= step[inside] * (0.5 + 1e-5)), i
        # clipping only beyond the largest level
        clipped = np.abs(q) == qm
        assert np.all(np.abs(Xd[i][~clipped]) <= step[~clipped] * (qm + 0.5 + 1e-5))


@pytest.mark.parametrize("unit,b", [(HEAD, 2), (HEAD, 4), (HEAD, 6), (HEAD, 8), (ROW, None)])
def test_codes_are_nearest_levels(oracle, rng, unit, b):
    for fit_iters in (1, 3):
        X = _state(rng)
        rb = _widths(rng, unit, b)
        page = oracle.encode_head(X, unit, rb, _w(rng), fit_iters)
        _check_nearest_levels(oracle, X, unit, rb, page)


def test_pivot_head_is_fp16(oracle, rng):
    X = _state(rng, 100.0)
    X[0, 0] = 1e6
    X[1, 1] = 3e-7            # binary16 subnormal
    rb = np.full(D, PIV, np.int8)
    page = oracle.encode_head(X, HEAD, rb, _w(rng))
    assert page.size == D * D * 2
    vals = _head_streams(page, 16).view(np.float16).reshape(8, 4, 8, 4, 16)   # [w][cg][g][c][r]
    vals = vals.transpose(2, 4, 0, 1, 3).reshape(D, D)
    ref = np.float16(np.clip(X, -65504, 65504))
    assert np.array_equal(vals.astype(np.float64), ref.astype(np.float64))


@pytest.mark.parametrize("b", [2, 4, 6, 8])
def test_bit_layout_with_independent_unpacker(oracle, rng, b):
    """Head units: offset-binary codes u = q + 2^(b-1), LSB-first, in chunks of
    the 16 codes of one band of rows (16g..16g+15) in one column; the four chunks
    of a band in 4 adjacent columns form one stream, stored as 16-byte pieces
    interleaved over the 32 streams of each group of 16 columns."""
    X = _state(rng)
    rb = np.full(D, b, np.int8)
    page = oracle.encode_head(X, HEAD, rb, _w(rng))
    assert page.size == 512 + 16 * b * D
    r16, c16, codes, _ = oracle.unpack_head(page, HEAD, rb)
    assert np.array_equal(page[:256].view(np.uint16), r16)
    assert np.array_equal(page[256:512].view(np.uint16), c16)
    bits = np.unpackbits(_head_streams(page[512:], b), axis=-1, bitorder="little")
    u = (bits.reshape(8, 4, 8, 4, 16, b) * (1 << np.arange(b))).sum(-1)   # [w][cg][g][c][r]
    u = u.transpose(2, 4, 0, 1, 3).reshape(D, D)
    assert np.array_equal(u - 2 ** (b - 1), codes.astype(np.int64))
    assert u.min() >= 1


def test_row_unit_layout_with_independent_unpacker(oracle, rng):
    """Row units: r | c | row i holds its 128 codes (b_i bits, LSB-first), FP16 rows
    for pivots; rows are stored by decreasing width, equal widths in index order."""
    X = _state(rng)
    rb = _widths(rng, ROW)
    page = oracle.encode_head(X, ROW, rb, _w(rng))
    assert page.size == 512 + 16 * int(np.sum(rb.astype(np.int64)))
    _, _, codes, piv = oracle.unpack_head(page, ROW, rb)
    order = sorted(range(D), key=lambda i: (-int(rb[i]), i))
    assert len(set(rb.tolist())) > 2                # the order is not trivial
    off = 512
    for i in order:
        b = int(rb[i])
        row = page[off:off + 16 * b]
        if b == PIV:
            assert np.array_equal(row.view(np.uint16), piv[i])
        else:
            bits = np.unpackbits(row, bitorder="little").reshape(D, b)
            u = (bits * (1 << np.arange(b))).sum(-1)
            assert np.array_equal(u - 2 ** (b - 1), codes[i].astype(np.int64))
        off += 16 * b


def test_zero_state(oracle, rng):
    X = np.zeros((D, D), np.float32)
    rb = _widths(rng, ROW)
    page = oracle.encode_head(X, ROW, rb, _w(rng))
    r16, c16, codes, piv = oracle.unpack_head(page, ROW, rb)
    nonpiv = rb != PIV
    assert np.all(_f16(r16)[nonpiv] == 2.0 ** -14) and np.all(_f16(r16)[~nonpiv] == 0)
    assert np.all(_f16(c16) == 2.0 ** -14)
    assert not codes.any() and not piv.any()


@pytest.mark.parametrize("unit", [HEAD, ROW])
def test_power_of_two_equivariance(oracle, rng, unit):
    """r_i ~ m_i^(1/2): X -> 16X gives r -> 4r, c -> 4c and identical codes;
    w -> 16w gives r -> r/4, c -> 4c (the common factor of w^2 cancels in the fit)."""
    X = _state(rng, 0.5)
    rb = _widths(rng, unit, 6)
    w = _w(rng)
    r0, c0, z0, p0 = oracle.unpack_head(oracle.encode_head(X, unit, rb, w), unit, rb)
    r1, c1, z1, _ = oracle.unpack_head(oracle.encode_head(16 * X, unit, rb, w), unit, rb)
    r2, c2, z2, _ = oracle.unpack_head(oracle.encode_head(X, unit, rb, 16 * w), unit, rb)
    nonpiv = rb != PIV
    assert np.array_equal(_f16(r1)[nonpiv], 4 * _f16(r0)[nonpiv])
    assert np.array_equal(_f16(c1), 4 * _f16(c0))
    assert np.array_equal(z1, z0)
    assert np.array_equal(_f16(r2)[nonpiv], _f16(r0)[nonpiv] / 4)
    assert np.array_equal(_f16(c2), 4 * _f16(c0))
    assert np.array_equal(z2, z0)


def test_single_row_scaling_moves_only_its_factor(oracle, rng):
    X = _state(rng, 0.5)
    rb = np.full(D, 8, np.int8)
    w = _w(rng)
    r0, _, _, _ = oracle.unpack_head(oracle.encode_head(X, HEAD, rb, w), HEAD, rb)
    X2 = X.copy()
    X2[17] *= 16
    r1, _, _, _ = oracle.unpack_head(oracle.encode_head(X2, HEAD, rb, w), HEAD, rb)
    assert _f16(r1)[17] == 4 * _f16(r0)[17]
    others = np.arange(D) != 17
    assert np.array_equal(r1[others], r0[others])


@pytest.mark.parametrize("b", [2, 4, 6, 8])
def test_normalised_codebook_reconstructs_like_plain(oracle, rng, b):
    """App. C.1: storing q with z = 2^(8-b) q only rescales the shared column vector."""
    X = _state(rng)
    w = _w(rng)
    rb = np.full(D, b, np.int8)
    ph = oracle.encode_head(X, HEAD, rb, w)
    pr = oracle.encode_head(X, ROW, rb, w)
    rh, ch, zh, _ = oracle.unpack_head(ph, HEAD, rb)
    rr, cr, zr, _ = oracle.unpack_head(pr, ROW, rb)
    assert np.array_equal(rh, rr) and np.array_equal(zh, zr)
    assert np.array_equal(_f16(cr) * 2.0 ** (8 - b), _f16(ch))
    assert np.array_equal(oracle.decode_head(ph, HEAD, rb), oracle.decode_head(pr, ROW, rb))


@pytest.mark.parametrize("unit", [HEAD, ROW])
def test_column_update_minimises_weighted_error(oracle, rng, unit):
    """Sec. 4.3 column factors: for the codes it was computed from, c_j minimises
    sum_i w_i^2 (X_ij - r_i c z_ij)^2 (found here by a 1-D golden-section search)."""
    X = _state(rng)
    rb = _widths(rng, unit, 4)
    w = _w(rng)
    r, c, z = oracle.fit_debug(X, unit, rb, w, 1)
    nonpiv = rb != PIV
    zs = np.where(rb == PIV, 0, 2.0 ** (8 - rb.astype(np.float64))) if unit == ROW else np.ones(D)
    Xd = X.astype(np.float64)
    gr = (np.sqrt(5) - 1) / 2
    for j in rng.choice(D, 12, replace=False):
        v = r * zs * z[:, j]

        def f(cc):
            return np.sum((w[nonpiv].astype(np.float64) ** 2) * (Xd[nonpiv, j] - cc * v[nonpiv]) ** 2)

        lo, hi = 0.0, 4.0 * float(c[j])
        for _ in range(200):
            a, bb = hi - gr * (hi - lo), lo + gr * (hi - lo)
            if f(a) < f(bb):
                hi = bb
            else:
                lo = a
        assert abs(0.5 * (lo + hi) - c[j]) <= 1e-5 * c[j]


@pytest.mark.parametrize("unit", [HEAD, ROW])
def test_fit_starts_clip_free_and_takes_one_update(oracle, rng, unit):
    """App. C.1: the column start is the smallest scale at which no integer row
    clips, c0_j = max_i |X_ij| / (r_i zs_i qmax_i); one fixed-code update then
    uses the nearest codes at c0 (clipped to +-qmax, which the start makes
    unnecessary)."""
    X = _state(rng)
    rb = _widths(rng, unit, 6)
    w = _w(rng)
    nonpiv = rb != PIV
    b = np.where(nonpiv, rb, 8).astype(np.float64)
    zs = 2.0 ** (8 - b) if unit == ROW else np.ones(D)
    qm = 2.0 ** (b - 1) - 1
    r, c0, _ = oracle.fit_debug(X, unit, rb, w, 0)
    Xd = X.astype(np.float64)
    start = (np.abs(Xd[nonpiv]) / (r * zs * qm)[nonpiv, None]).max(axis=0)
    assert np.allclose(c0, np.clip(start, 2.0 ** -14, 65504.0), rtol=1e-6)
    # the smallest such scale: slightly below it some integer row of every
    # column needs a code beyond qmax
    below = Xd[nonpiv] / (r * zs)[nonpiv, None] / (c0.astype(np.float64) * (1 - 1e-5))[None, :]
    inside = c0 > 2.0 ** -14
    assert np.all((np.abs(below) > qm[nonpiv, None]).any(axis=0)[inside])
    r1, c1, z1 = oracle.fit_debug(X, unit, rb, w, 1)
    assert np.array_equal(r1, r)
    t = Xd[nonpiv] / (r * zs)[nonpiv, None] / c0.astype(np.float64)[None, :]
    zref = np.clip(np.rint(t), -qm[nonpiv, None], qm[nonpiv, None])
    assert np.mean(z1[nonpiv] != zref) <= 1e-4
    assert np.all(np.abs(t) <= qm[nonpiv, None] * (1 + 1e-6))


@pytest.mark.parametrize("bits", [4, 6, 8])
def test_intb_baseline(oracle, rng, bits):
    """App. B.5: per key row s_i = fp16(absmax/q_b) in [2^-14, 65504], nearest codes."""
    X = _state(rng)
    page = oracle.intb_encode_head(X, bits)
    assert page.size == 256 + 16 * bits * D
    s = page[:256].view(np.float16).astype(np.float64)
    qm = 2 ** (bits - 1) - 1
    amax = np.abs(X.astype(np.float64)).max(axis=1)
    assert np.array_equal(s, np.float16(np.clip(amax / qm, 2 ** -14, 65504)).astype(np.float64))
    R = oracle.intb_decode_head(page, bits)
    q = np.rint(R / s[:, None])
    assert np.all(np.abs(q) <= qm)
    arg = np.abs(X).argmax(axis=1)
    assert np.all(np.abs(q[np.arange(D), arg]) == qm)
    assert np.all(np.abs(R - X) <= s[:, None] * (0.5 + 1e-5) + (np.abs(q) == qm) * np.abs(X))


@pytest.mark.parametrize("bits", [4, 6, 8])
def test_temporal_uniform_widths_is_intb(oracle, rng, bits):
    """"Temporal only" (Sec. 5.4) at one width without pivots is the uniform
    rowwise baseline of App. B.5, byte for byte."""
    X = _state(rng)
    rb = np.full(D, bits, np.int8)
    page = oracle.temporal_encode_head(X, rb)
    assert np.array_equal(page, oracle.intb_encode_head(X, bits))
    assert np.array_equal(oracle.temporal_decode_head(page, rb), oracle.intb_decode_head(page, bits))


def test_temporal_mixed_widths_and_pivots(oracle, rng):
    """Mixed row widths with FP16 pivot rows: every row follows App. B.5 at its
    own width (numpy scale, absmax at +-q_b, half-step bound), pivots are numpy
    float16, and rows sit in index order (independent numpy unpacker)."""
    X = _state(rng)
    rb = rng.choice([2, 4, 6, 8, PIV], size=D, p=[0.15, 0.3, 0.3, 0.2, 0.05]).astype(np.int8)
    rb[:2] = (PIV, 2)
    page = oracle.temporal_encode_head(X, rb)
    assert page.size == 256 + 16 * int(rb.astype(np.int64).sum())
    R = oracle.temporal_decode_head(page, rb)
    s = page[:256].view(np.float16).astype(np.float64)
    bits = np.unpackbits(page, bitorder="little")
    off = 256
    for i in range(D):
        b = int(rb[i])
        x = X[i].astype(np.float64)
        if b == PIV:
            assert s[i] == 0
            vals = page[off:off + 256].view(np.float16).astype(np.float64)
            assert np.array_equal(vals, np.float16(X[i]).astype(np.float64))
            assert np.array_equal(R[i], vals)
        else:
            qm = 2 ** (b - 1) - 1
            assert s[i] == np.float16(np.clip(np.abs(x).max() / qm, 2 ** -14, 65504))
            u = bits[8 * off:8 * off + b * D].reshape(D, b) @ (1 << np.arange(b))
            q = u.astype(np.int64) - (1 << (b - 1))
            assert np.all(np.abs(q) <= qm) and abs(q[np.abs(x).argmax()]) == qm
            assert np.array_equal(R[i], s[i] * q)
            assert np.all(np.abs(R[i] - x) <= s[i] * (0.5 + 1e-5) + (np.abs(q) == qm) * np.abs(x))
        off += 16 * b
    assert off == page.size


def test_code_ties_go_to_even(oracle):
    """Sec. 4.3 quantizes X_ij / (r_i c_j) to the nearest level; an exact tie
    (the quotient a half-integer) goes to the even level. Rows with mean |X| = 1
    and w = 1 get r_i = 1, and a column whose largest entry is qmax = 127 gets
    the clip-free start c0 = 1, so the first fixed-code pass quantizes X_i0
    itself."""
    X = np.zeros((D, D), np.float32)
    X[0, 0], X[0, 1] = 127.0, 1.0
    ties = [0.5, 1.5, 2.5, 3.5, -0.5, -1.5, -2.5, 126.5]
    for i, x in enumerate(ties, start=1):
        X[i, 0] = x
        X[i, 1] = 128.0 - abs(x)                   # mean |X_i| = 1
    rb = np.full(D, 8, np.int8)
    r, c0, _ = oracle.fit_debug(X, HEAD, rb, np.ones(D, np.float32), 0)
    assert np.all(r[:len(ties) + 1] == 1.0) and c0[0] == 1.0
    _, _, z = oracle.fit_debug(X, HEAD, rb, np.ones(D, np.float32), 1)
    assert z[0, 0] == 127
    assert [int(z[i, 0]) for i in range(1, len(ties) + 1)] == [0, 2, 2, 4, 0, -2, -2, 126]
