"""Pins of the oracle's noise generator (Philox4x32-10 + Box-Muller with its own log and sin/cos).

The paper models mini-batch gradient noise only as "a randomly selected
mini-batch" (Sec. II-A, Eq. eg); the surrogate draws it from a counter-based
generator.  Each piece is pinned to something other than the oracle itself:
published known-answer vectors, libm in fp64, Gaussian moments and a KS test,
and torch's own fp32 -> bf16 rounding.
"""
import os

import numpy as np
import pytest

from oracle import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            w = [int(t, 16) for t in line.split()]
            rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,expect", _kat_rows())
def test_philox_known_answers(ctr, key, expect):
    out = O.philox4x32_10(ctr, key)
    assert [int(v) for v in out] == expect


def test_philox_counter_based_and_avalanche():
    # Same (counter, key) -> same block; one flipped counter bit flips about half the output bits.
    base = O.philox4x32_10([5, 6, 7, 8], [9, 10])
    assert np.array_equal(base, O.philox4x32_10([5, 6, 7, 8], [9, 10]))
    flips = []
    for word in range(4):
        for bit in range(32):
            ctr = [5, 6, 7, 8]
            ctr[word] ^= 1 << bit
            out = O.philox4x32_10(ctr, [9, 10])
            flips.append(sum(bin(int(a) ^ int(b)).count("1") for a, b in zip(out, base)))
    flips = np.array(flips)
    assert 56 < flips.mean() < 72  # 64 expected out of 128 bits


def test_noise_stream_layout():
    # Word r of block q belongs to element 4q + r; replica, step and tag each change the stream.
    w = O.philox_words(seed=77, tag=0, i=3, k=11, q0=5, nq=2)
    key = [77, 0]
    assert np.array_equal(w[0], O.philox4x32_10([5, 3, 11, 0], key))
    assert np.array_equal(w[1], O.philox4x32_10([6, 3, 11, 0], key))
    seed = (0xABCDEF01 << 32) | 0x12345678
    w = O.philox_words(seed=seed, tag=1, i=0, k=0, q0=0, nq=1)
    assert np.array_equal(w[0], O.philox4x32_10([0, 0, 0, 1], [0x12345678, 0xABCDEF01]))


def _ulp_err(got, ref):
    ref32 = np.abs(ref).astype(np.float32)
    ulp = np.spacing(ref32).astype(np.float64)
    return np.abs(got.astype(np.float64) - ref) / ulp


def test_ln_exhaustive_on_the_uniform_grid():
    # Every radius input the generator can produce: u = 1 - m 2^-23, m = 0 .. 2^23 - 1.
    m = np.arange(1 << 23, dtype=np.float64)
    u = (1.0 - m * 2.0 ** -23).astype(np.float32)
    got = O.ln(u)
    ref = np.log(u.astype(np.float64))
    assert got[0] == 0.0  # ln 1
    err = _ulp_err(got[1:], ref[1:])
    assert err.max() <= 2.0, err.max()


def test_ln_other_binades():
    rng = np.random.default_rng(1)
    u = rng.uniform(1e-30, 1e30, 200000).astype(np.float32)
    u = np.concatenate([u, np.float32(2.0) ** np.arange(-120, 120, dtype=np.float32)])
    got = O.ln(u)
    ref = np.log(u.astype(np.float64))
    nz = ref != 0
    assert _ulp_err(got[nz], ref[nz]).max() <= 2.0


def test_sincos_exhaustive_on_the_angle_grid():
    m = np.arange(1 << 23, dtype=np.float64)
    u = (m * 2.0 ** -23).astype(np.float32)
    s, c = O.sincos_turn(u)
    th = 2.0 * np.pi * u.astype(np.float64)
    rs, rc = np.sin(th), np.cos(th)
    assert np.abs(s - rs).max() <= 1.2e-7
    assert np.abs(c - rc).max() <= 1.2e-7
    big_s, big_c = np.abs(rs) > 1e-3, np.abs(rc) > 1e-3
    assert _ulp_err(s[big_s], rs[big_s]).max() <= 2.0
    assert _ulp_err(c[big_c], rc[big_c]).max() <= 2.0
    # quarter turns are exact
    q = u[[0, 1 << 21, 1 << 22, 3 << 21]]
    s, c = O.sincos_turn(q)
    assert list(s) == [0.0, 1.0, 0.0, -1.0] and list(c) == [1.0, 0.0, -1.0, 0.0]


def test_box_muller_is_standard_normal():
    from scipy import stats
    N = 1 << 22
    z = O.normals(seed=2024, tag=0, i=1, k=3, j0=0, m=N).astype(np.float64)
    se = 1.0 / np.sqrt(N)
    assert abs(z.mean()) < 5 * se
    assert abs(z.var() - 1.0) < 5 * np.sqrt(2.0 / N)
    kurt = ((z - z.mean()) ** 4).mean() / z.var() ** 2
    assert abs(kurt - 3.0) < 5 * np.sqrt(24.0 / N)
    assert np.abs(z).max() < np.sqrt(-2.0 * np.log(2.0 ** -23)) + 1e-5  # truncation of the radius
    assert stats.kstest(z[: 1 << 20], "norm").pvalue > 1e-4
    # the two normals of a pair are uncorrelated
    pair0, pair1 = z[0::4], z[1::4]
    assert abs(np.corrcoef(pair0, pair1)[0, 1]) < 5 / np.sqrt(pair0.size)


def test_streams_are_independent_across_replica_step_tag():
    a = O.normals(9, 0, 0, 0, 0, 1 << 16).astype(np.float64)
    for other in (O.normals(9, 0, 1, 0, 0, 1 << 16), O.normals(9, 0, 0, 1, 0, 1 << 16),
                  O.normals(9, 1, 0, 0, 0, 1 << 16), O.normals(10, 0, 0, 0, 0, 1 << 16)):
        assert abs(np.corrcoef(a, other.astype(np.float64))[0, 1]) < 5 / 256


def test_normals_offset_window():
    full = O.normals(5, 0, 2, 7, 0, 64)
    part = O.normals(5, 0, 2, 7, 13, 30)
    assert np.array_equal(full[13:43], part)


def test_bf16_noise_tensor_matches_torch_rounding():
    torch = pytest.importorskip("torch")
    n, P = 3, 1027
    t = O.noise_bf16(31, n, P)
    for i in range(n):
        z = O.normals(31, 1, i, 0, 0, P)
        ref = torch.from_numpy(z).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        assert np.array_equal(t[i], ref)


@pytest.mark.parametrize("kexp", [1, 2, 5, 13, 23])
@pytest.mark.parametrize("angle_num,angle_den", [(1, 16), (3, 16), (5, 8), (0, 1)])
def test_box_muller_special_words(kexp, angle_num, angle_den):
    # Words chosen so that u1 = 2^-kexp and u2 = angle_num / angle_den exactly:
    # z0 = sqrt(2 kexp ln 2) cos(2 pi u2), z1 = sqrt(2 kexp ln 2) sin(2 pi u2).
    w_radius = ((1 << 23) - (1 << (23 - kexp))) << 9
    w_angle = (angle_num * (1 << 23) // angle_den) << 9
    z0, z1 = O.box_muller_words(w_radius, w_angle)
    r = np.sqrt(2.0 * kexp * np.log(2.0))
    th = 2.0 * np.pi * angle_num / angle_den
    assert z0 == pytest.approx(r * np.cos(th), abs=4e-7 * r)
    assert z1 == pytest.approx(r * np.sin(th), abs=4e-7 * r)
    # the low 9 bits of a word do not matter
    assert O.box_muller_words(w_radius | 0x1FF, w_angle | 0x1FF) == (z0, z1)


def test_word_to_element_layout():
    # Element 4q + r of replica i at step k: pair (w0, w1) -> elements 0, 1 and (w2, w3) -> 2, 3,
    # with u1 = 1 - (w >> 9) 2^-23 and u2 = (w >> 9) 2^-23 (fp64 evaluation of Box-Muller).
    seed, i, k, q = 0x1234_5678_9ABC_DEF0, 5, 9, 1000
    w = O.philox4x32_10([q, i, k, 0], [seed & 0xFFFFFFFF, seed >> 32]).astype(np.int64)
    u1 = 1.0 - (w[[0, 2]] >> 9) * 2.0 ** -23
    u2 = (w[[1, 3]] >> 9) * 2.0 ** -23
    r = np.sqrt(-2.0 * np.log(u1))
    expect = np.array([r[0] * np.cos(2 * np.pi * u2[0]), r[0] * np.sin(2 * np.pi * u2[0]),
                       r[1] * np.cos(2 * np.pi * u2[1]), r[1] * np.sin(2 * np.pi * u2[1])])
    z = O.normals(seed, 0, i, k, 4 * q, 4)
    assert np.allclose(z, expect, rtol=0, atol=1e-6)


def test_bf16_rounding_ties_to_even():
    torch = pytest.importorskip("torch")
    bits = np.array([0x3F808000, 0x3F818000, 0xBF808000, 0x3F807FFF, 0x3F808001, 0x00008000,
                     0x7F7F8000 - 0x10000, 0x3F800000], dtype=np.uint32)
    rng = np.random.default_rng(0)
    bits = np.concatenate([bits, (rng.integers(0, 1 << 31, 4096, dtype=np.uint32) & 0xFFFF0000) | 0x8000])
    bits = bits[((bits >> 23) & 0xFF) != 0xFF]  # finite values only
    x = bits.view(np.float32)
    ref = torch.from_numpy(x.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(O.to_bf16(x), ref)
