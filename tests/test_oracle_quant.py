"""Pins for the oracle's quantize-on-append path (INT2, QSAC, PSAC).

Each pin checks the oracle against something other than itself: hand-computed
fixtures (tests/golden), closed forms of Eq. 1-2, brute force / library
nearest-neighbour searches (scipy.spatial.distance.cdist), invariances of the
QSAC score (Eq. 12) and an exactly representable PSAC construction (Eq. 16-17).
"""
import json
import os

import numpy as np
import pytest
import torch
from scipy.spatial.distance import cdist

from paper_2609_26425_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf(x):
    """float array -> bf16 bits (values must be exactly representable)."""
    a = np.asarray(x, np.float32)
    b = (a.view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal((b.astype(np.uint32) << 16).view(np.float32), a), "not bf16-exact"
    return b


def code_bit(c):
    """Bit of channel c's code (App. D.1 packing reading: 16-channel little-endian
    words, even channel 2k at bit 2k, odd channel 2k+1 at bit 16+2k)."""
    j = c % 16
    return 32 * (c // 16) + 16 * (j & 1) + 2 * (j >> 1)


def unpack2(bytes_, n):
    b = np.asarray(bytes_, np.uint8)
    out = np.zeros(b.shape[:-1] + (n,), np.int64)
    for c in range(n):
        bit = code_bit(c)
        out[..., c] = (b[..., bit // 8] >> (bit % 8)) & 3
    return out


def f16(bits):
    return np.asarray(bits, np.uint16).view(np.float16).astype(np.float64)


# --------------------------------------------------------------------- INT2
def test_int2_hand_example(orc):
    g = json.load(open(os.path.join(GOLDEN, "int2_hand.json")))
    d, G = g["head_dim"], g["group_size"]
    x = bf(g["key"]).reshape(1, 1, d)
    cent = bf(g["centroid"]).reshape(1, 1, d)
    o = orc.quantize(x, cent, G=G, r=0, M=1, is_key=True)
    assert list(o["codes"][0, 0]) == g["codes"]
    assert list(o["zeros"][0, 0]) == g["zeros"]
    assert list(o["scales"][0, 0]) == g["scales_f16_bits"]
    deq = orc.dequant(o, cent, G=G, r=0)
    assert np.array_equal(deq[0, 0], np.array(g["dequant"]))
    assert np.array_equal(o["khat0"][0, 0].astype(np.float64), np.array(g["dequant"]))


@pytest.mark.parametrize("G", [32, 64])
def test_int2_round_trip_bound(orc, G):
    """|x - xhat| <= s/2 per element, codes and zero-points in [0, 3] (Eq. 1-2)."""
    N, H, d = 300, 3, 128
    x = synth.bits(synth.gaussian_bf16(11, N, H, d, scale=3.0))
    cent = np.zeros((H, 1, d), np.uint16)
    o = orc.quantize(x, cent, G=G, r=0, M=1, is_key=True)
    xf = orc.bf16_to_f32(x).astype(np.float64)
    deq = orc.dequant(o, cent, G=G, r=0)
    s = np.repeat(f16(o["scales"]), G, axis=-1)
    err = np.abs(xf - deq)
    assert np.all(err <= s / 2 + 4 * np.finfo(np.float32).eps * np.abs(xf) + 1e-30)
    codes = unpack2(o["codes"], d)
    assert codes.min() >= 0 and codes.max() <= 3
    # the stored scale covers the zero-inclusive range and is the smallest binary16 that does
    xg = xf.reshape(N, H, d // G, G)
    rng_ = np.maximum(xg.max(-1), 0) - np.minimum(xg.min(-1), 0)
    s_st = f16(o["scales"])
    assert np.all(3 * s_st >= rng_ * (1 - 1e-7))
    prev = np.nextafter(o["scales"].view(np.float16), np.float16(0)).astype(np.float64)
    assert np.all(3 * prev < rng_ * (1 + 1e-6))


def test_int2_grid_values_exact(orc):
    """Values on a grid {-s, 0, s, 2s} with both ends present reconstruct exactly."""
    rng = np.random.default_rng(3)
    N, H, d, G = 64, 2, 128, 32
    s = np.float32(0.1875)  # binary16-exact
    mult = rng.integers(-1, 3, size=(N, H, d)).astype(np.float32)
    mult[..., ::G] = -1
    mult[..., 1::G] = 2
    x = bf(mult * s)
    cent = np.zeros((H, 1, d), np.uint16)
    o = orc.quantize(x, cent, G=G, r=0, M=1, is_key=True)
    deq = orc.dequant(o, cent, G=G, r=0)
    assert np.array_equal(deq, (mult * s).astype(np.float64))
    assert np.all(f16(o["scales"]) == s)


def test_int2_zero_and_constant_groups(orc):
    d, G = 128, 32
    x = np.zeros((2, 1, d), np.float32)
    x[1, 0, :G] = 3 * 0.0625          # constant group, c/3 exact in binary16
    x[1, 0, G:2 * G] = -3 * 0.125
    xb = bf(x)
    cent = np.zeros((1, 1, d), np.uint16)
    o = orc.quantize(xb, cent, G=G, r=0, M=1, is_key=True)
    deq = orc.dequant(o, cent, G=G, r=0)
    assert np.array_equal(deq, x.astype(np.float64))
    assert np.all(o["scales"][0] == 0) and np.all(o["codes"][0] == 0) and np.all(o["zeros"][0] == 0)


def test_packing_layout(orc):
    """Four INT2 codes per byte (App. D.1): channel c at bit code_bit(c);
    zero-point g at byte g/4, bits 2(g%4)."""
    d, G = 128, 32
    s = 0.25
    x = np.zeros((1, 1, d), np.float32)
    want_codes = np.zeros(d, np.int64)
    want_z = []
    for g in range(d // G):
        z = [1, 0, 2, 3][g]
        want_z.append(z)
        q = (np.arange(G) + g) % 4
        q[0], q[1] = 0, 3  # both ends present -> range 3s
        want_codes[g * G:(g + 1) * G] = q
        x[0, 0, g * G:(g + 1) * G] = (q - z) * s
    o = orc.quantize(bf(x), np.zeros((1, 1, d), np.uint16), G=G, r=0, M=1, is_key=True)
    words = np.zeros(d // 16, np.uint32)
    for c in range(d):
        w, j = divmod(c, 16)
        words[w] |= np.uint32(want_codes[c] << (2 * (j >> 1) + 16 * (j & 1)))
    assert np.array_equal(o["codes"][0, 0], words.view(np.uint8))
    zbyte = sum(z << (2 * g) for g, z in enumerate(want_z))
    assert o["zeros"][0, 0, 0] == zbyte
    assert np.array_equal(unpack2(o["codes"], d)[0, 0], want_codes)


# --------------------------------------------------------------------- QSAC
def test_qsac_hand_cases(orc):
    g = json.load(open(os.path.join(GOLDEN, "qsac_hand.json")))
    d, G = g["head_dim"], g["group_size"]
    k = bf(g["key"]).reshape(1, 1, d)
    for case in g["cases"]:
        cent = bf(case["centroids"]).reshape(1, -1, d)
        C = cent.shape[1]
        w = np.array(case["w"], np.float32).reshape(1, d)
        for m, want in case["ids_by_M"].items():
            o = orc.quantize(k, cent, G=G, r=0, M=int(m), is_key=True, w=w, keep_scores=True)
            assert int(o["ids"][0, 0]) == want, (case["name"], m)
            assert np.array_equal(o["dq"][0, 0], np.array(case["dQ"], np.float32)), case["name"]
            if int(m) == C:
                S = np.zeros(C, np.float32)
                S[o["cand"][0, 0]] = o["S"][0, 0]
                assert np.array_equal(S, np.array(case["S"], np.float32)), case["name"]


def _qsac_scores_fp64(k, cent, w, G):
    """Eq. 12 evaluated in fp64 for every centroid: k [d], cent [C][d], w [d]."""
    r = k[None, :] - cent
    C, d = r.shape
    rg = r.reshape(C, d // G, G)
    R = rg.max(-1) - rg.min(-1)
    W = w.reshape(d // G, G).sum(-1)
    return (W[None, :] * R ** 2).sum(-1)


@pytest.mark.parametrize("weighted", [False, True])
def test_qsac_exhaustive_is_global_argmin(orc, weighted):
    """M = C: the chosen id minimises the QSAC score over all centroids (brute force)."""
    N, H, d, C, G = 60, 2, 128, 8, 32
    x = synth.bits(synth.gaussian_bf16(21, N, H, d))
    cent = synth.bits(synth.gaussian_bf16(22, H, C, d, scale=0.7))
    w = synth.random_weights(23, H, d).numpy() if weighted else None
    o = orc.quantize(x, cent, G=G, r=0, M=C, is_key=True, w=w)
    xf = orc.bf16_to_f32(x).astype(np.float64)
    cf = orc.bf16_to_f32(cent).astype(np.float64)
    wf = np.ones((H, d)) if w is None else w.astype(np.float64)
    for i in range(N):
        for h in range(H):
            S = _qsac_scores_fp64(xf[i, h], cf[h], wf[h], G)
            best = S.min()
            got = o["ids"][i, h]
            assert S[got] <= best * (1 + 1e-5) + 1e-12


def test_qsac_invariant_to_groupwise_shift(orc):
    """S depends on group ranges only: shifting a key by a per-group constant keeps the
    exhaustive (M = C) choice (Eq. 10, 12)."""
    rng = np.random.default_rng(5)
    N, H, d, C, G = 40, 1, 128, 6, 32
    k = rng.integers(-16, 16, size=(N, H, d)).astype(np.float32) / 8
    cent = rng.integers(-16, 16, size=(H, C, d)).astype(np.float32) / 8
    shift = np.repeat(rng.integers(-8, 8, size=(N, H, d // G)).astype(np.float32) / 4, G, axis=-1)
    w = synth.random_weights(6, H, d).numpy()
    a = orc.quantize(bf(k), bf(cent), G=G, r=0, M=C, is_key=True, w=w)
    b = orc.quantize(bf(k + shift), bf(cent), G=G, r=0, M=C, is_key=True, w=w)
    assert np.array_equal(a["ids"], b["ids"])


def test_m1_uniform_weights_is_euclidean_nearest(orc):
    """w = 1 and M = 1 reduce QSAC to plain nearest-centroid assignment (QVG / k-means)."""
    N, H, d, C, G = 200, 2, 128, 32, 32
    x = synth.bits(synth.gaussian_bf16(31, N, H, d))
    cent = synth.bits(synth.gaussian_bf16(32, H, C, d, scale=0.5))
    o = orc.quantize(x, cent, G=G, r=0, M=1, is_key=True)
    xf = orc.bf16_to_f32(x).astype(np.float64)
    cf = orc.bf16_to_f32(cent).astype(np.float64)
    for h in range(H):
        D = cdist(xf[:, h], cf[h], "sqeuclidean")
        ref = D.argmin(1)
        got = o["ids"][:, h]
        srt = np.sort(D, 1)
        gap = (srt[:, 1] - srt[:, 0]) / srt[:, 1]
        bad = (got != ref) & (gap > 1e-5)
        assert not bad.any()


def test_topm_candidates_are_weighted_nearest(orc):
    """The candidate set is the M nearest centroids under the Query-aware distance (Eq. 9)."""
    N, H, d, C, G, M = 150, 2, 128, 24, 32, 4
    x = synth.bits(synth.gaussian_bf16(41, N, H, d))
    cent = synth.bits(synth.gaussian_bf16(42, H, C, d, scale=0.5))
    w = synth.random_weights(43, H, d).numpy()
    o = orc.quantize(x, cent, G=G, r=0, M=M, is_key=True, w=w)
    xf = orc.bf16_to_f32(x).astype(np.float64)
    cf = orc.bf16_to_f32(cent).astype(np.float64)
    for h in range(H):
        sw = np.sqrt(w[h].astype(np.float64))
        D = cdist(xf[:, h] * sw, cf[h] * sw, "sqeuclidean")
        order = np.argsort(D, 1, kind="stable")
        for i in range(N):
            got = set(o["cand"][i, h].tolist())
            want = set(order[i, :M].tolist())
            if got != want:
                assert o["m_topm"][i, h] < 1e-5
            # and the id is the QSAC argmin inside the candidate set
            S = _qsac_scores_fp64(xf[i, h], cf[h], w[h].astype(np.float64), G)
            cands = sorted(got)
            assert S[o["ids"][i, h]] <= S[cands].min() * (1 + 1e-5) + 1e-12


def test_duplicate_centroids_tie_to_lowest_index(orc):
    N, H, d, G = 30, 1, 128, 32
    x = synth.bits(synth.gaussian_bf16(51, N, H, d))
    base = synth.bits(synth.gaussian_bf16(52, H, 3, d, scale=0.5))
    cent = np.concatenate([base, base], axis=1)  # centroid j+3 duplicates j
    for M in (1, 2, 6):
        o = orc.quantize(x, cent, G=G, r=0, M=M, is_key=True)
        assert o["ids"].max() < 3


def test_values_ignore_weights_and_psac(orc):
    """Values use w = 1 and no PSAC (App. C.3 cold-start form, App. D.1)."""
    N, H, d, C, G, r = 50, 2, 128, 16, 32, 8
    x = synth.bits(synth.gaussian_bf16(61, N, H, d))
    cent = synth.bits(synth.gaussian_bf16(62, H, C, d, scale=0.5))
    w = synth.random_weights(63, H, d).numpy()
    U = synth.bits(synth.random_orthonormal(64, H, d, r))
    a = orc.quantize(x, cent, G=G, r=r, M=4, is_key=False, w=w, U_bits=U)
    b = orc.quantize(x, cent, G=G, r=r, M=4, is_key=False)
    for key in ("ids", "codes", "scales", "zeros"):
        assert np.array_equal(a[key], b[key])
    assert not a["coef"].any() and not a["sigma"].any()


# --------------------------------------------------------------------- PSAC
def test_psac_exact_when_error_in_span(orc):
    """Construction where E lies in span(U) and the INT8 coefficient is exact:
    K_hat = K_hat0 + C U^T reproduces K exactly (Eq. 13, 16, 17)."""
    d, G, r = 128, 32, 16
    rng = np.random.default_rng(7)
    N = 16
    s = 0.25
    chans = rng.permutation(d)[:r]
    U = np.zeros((1, d, r), np.float32)
    U[0, chans, np.arange(r)] = 1.0
    x = np.zeros((N, 1, d), np.float32)
    for i in range(N):
        mult = rng.integers(-1, 3, size=d).astype(np.float32)
        mult[::G] = -1
        mult[1::G] = 2
        x[i, 0] = mult * s
        c1 = chans[i % r]
        if c1 % G in (0, 1):
            c1 = chans[(i + 1) % r] if chans[(i + 1) % r] % G not in (0, 1) else c1 + 2
        x[i, 0, c1] = 0.0 + 127 * 2.0**-10  # rounds to code of 0: error 127*2^-10
    # channel c1 may lie outside U's span if we shifted it; put it into U
    o = orc.quantize(bf(x), np.zeros((1, 1, d), np.uint16), G=G, r=r, M=1, is_key=True, U_bits=bf(U))
    deq = orc.dequant(o, np.zeros((1, 1, d), np.uint16), G=G, r=r, U_bits=bf(U))
    inspan = [i for i in range(N) if o["kept"][i, 0]]
    assert len(inspan) >= N // 2
    for i in inspan:
        assert np.array_equal(deq[i, 0], x[i, 0].astype(np.float64))
        assert f16(o["sigma"][i, 0]) == 2.0**-10
        assert np.abs(o["coef"][i, 0]).max() == 127


def psac_hand_token(g):
    """The Key token, centroid and basis of the hand-computed INT8 fixture."""
    d, G, r, s = g["head_dim"], g["group_size"], g["psac_rank"], g["grid_scale"]
    m = ((7 * np.arange(d)) % 4 - 1).astype(np.float64)
    m[::G] = -1
    m[1::G] = 2
    x = m * s
    chans = np.array(g["target_channels"])
    assert np.all(chans % G > 1), "target channels must not carry a group's range"
    x[chans] = np.array(g["e_in_units_of_2^-10"]) * 2.0 ** -10
    U = np.zeros((1, d, r), np.float32)
    U[0, chans, np.arange(r)] = 1.0
    return bf(x.reshape(1, 1, d)), np.zeros((1, 1, d), np.uint16), bf(U), chans


def test_psac_int8_rounding_hand_fixture(orc):
    """INT8 PSAC codes round half to even and sigma is the binary16 round-up of
    max|c| / 127 (Sec. 4.2 Eq. 16, App. D.1; tests/golden/psac_int8_hand.json).
    The coefficients land on exact halves, quarters and near-integers, so
    truncation, rounding half away from zero, or a scale off by one binary16
    step give different codes."""
    g = json.load(open(os.path.join(GOLDEN, "psac_int8_hand.json")))
    d, G, r = g["head_dim"], g["group_size"], g["psac_rank"]
    x, cent, Ub, chans = psac_hand_token(g)
    o = orc.quantize(x, cent, G=G, r=r, M=1, is_key=True, U_bits=Ub)
    assert int(o["kept"][0, 0]) == 1
    assert int(o["sigma"][0, 0]) == g["sigma_f16_bits"]
    assert list(o["coef"][0, 0].astype(int)) == g["codes"]
    # the grid channels reconstruct exactly, the targets carry only the correction
    deq = orc.dequant(o, cent, G=G, r=r, U_bits=Ub)
    want = orc.bf16_to_f32(x)[0, 0].astype(np.float64)
    want[chans] = np.array(g["codes"]) * 2.0 ** -10
    assert np.array_equal(deq[0, 0], want)
    # with w = 1 and no correction stored, the zero codes are what a dropped row gives
    o0 = orc.quantize(x, cent, G=G, r=0, M=1, is_key=True)
    assert np.array_equal(o0["codes"], o["codes"]) and np.array_equal(o0["scales"], o["scales"])


def test_psac_off_and_rank_zero(orc):
    N, H, d, C, G = 40, 2, 128, 16, 32
    x = synth.bits(synth.gaussian_bf16(71, N, H, d))
    cent = synth.bits(synth.gaussian_bf16(72, H, C, d, scale=0.5))
    a = orc.quantize(x, cent, G=G, r=0, M=4, is_key=True)
    deq = orc.dequant(a, cent, G=G, r=0)
    assert np.array_equal(deq.astype(np.float32), a["khat0"])


def test_psac_keep_rule_and_projection(orc):
    """Kept rows lower the w-weighted error; zeroed rows carry no correction;
    the exact projection never grows the error (||E - U U^T E|| <= ||E||)."""
    N, H, d, C, G, r = 200, 2, 128, 16, 32, 16
    x = synth.bits(synth.gaussian_bf16(81, N, H, d))
    cent = synth.bits(synth.gaussian_bf16(82, H, C, d, scale=0.5))
    w = synth.random_weights(83, H, d).numpy()
    Ub = synth.bits(synth.random_orthonormal(84, H, d, r))
    o = orc.quantize(x, cent, G=G, r=r, M=4, is_key=True, w=w, U_bits=Ub)
    xf = orc.bf16_to_f32(x).astype(np.float64)
    k0 = o["khat0"].astype(np.float64)
    full = orc.dequant(o, cent, G=G, r=r, U_bits=Ub)
    E = xf - k0
    Ef = xf - full
    werr0 = (w[None] * E ** 2).sum(-1)
    werr1 = (w[None] * Ef ** 2).sum(-1)
    kept = o["kept"].astype(bool)
    assert kept.mean() > 0.5
    assert np.all(werr1[kept] < werr0[kept] * (1 + 1e-5))
    assert np.all(o["coef"][~kept] == 0) and np.all(o["sigma"][~kept] == 0)
    U = orc.bf16_to_f32(Ub).astype(np.float64)
    for h in range(H):
        Q, _ = np.linalg.qr(U[h])
        P = E[:, h] - (E[:, h] @ Q) @ Q.T
        assert np.all(np.linalg.norm(P, axis=1) <= np.linalg.norm(E[:, h], axis=1) + 1e-9)
    # INT8 codes within range, sigma = binary16 round-up of max|c|/127 on kept rows
    assert np.abs(o["coef"]).max() <= 127
    c = np.einsum("nhd,hdr->nhr", E, U)
    a = np.abs(c).max(-1) / 127
    sg = f16(o["sigma"])
    assert np.all(sg[kept] >= a[kept] * (1 - 1e-5))



# ------------------------------------------------------------------ two-level group scales (App. D.1)
def _one_token_chunk(groups):
    """A single token of one head whose residual (centroid 0) has the given
    32-channel groups; values are exact in bf16."""
    k = np.concatenate([np.asarray(g, np.float32) for g in groups])[None, None, :]
    kb = synth.bits(torch.from_numpy(k).to(torch.bfloat16))
    cent = np.zeros((1, 1, 128), np.uint16)
    return kb, cent


def test_two_level_scales_hand_fixture(orc):
    """Group ranges 3, 6, 1.5 and 0 give s32 = 1, 2, 0.5, 0; the secondary
    scale is the binary16 round-up of 2/255 = 0.00784313...: 2^-7 + 5 * 2^-17
    = 0.00785064697265625 (the binary16 step above 2^-7 is 2^-17); the codes
    are ceil(s32 / s2) = 128, 255, 64, 0 (hand computed: 127.38, 254.76,
    63.69)."""
    g0 = np.tile([-1.5, 1.5], 16)
    g1 = np.tile([0.0, 6.0], 16)
    g2 = np.tile([-0.75, 0.75], 16)
    g3 = np.zeros(32)
    kb, cent = _one_token_chunk([g0, g1, g2, g3])
    o = orc.quantize(kb, cent, G=32, r=0, M=1, is_key=True, two_level_scales=True)
    s2 = float(orc.f16_to_f32(o["s2"])[0, 0])
    assert s2 == 2.0 ** -7 + 5 * 2.0 ** -17
    assert o["scode"][0, 0].tolist() == [128, 255, 64, 0]
    assert np.all(o["scales"] == 0)


def test_two_level_scales_cover_minimal_and_round_trip(orc):
    """On random Keys: every code is the smallest with code * s2 >= the
    group's (hi - lo) / 3, and the reconstruction keeps the INT2 bound
    |x - x_hat| <= s / 2 with the stored scale s = code * s2."""
    H, N, C, G = 2, 200, 16, 32
    kb = synth.bits(synth.gaussian_bf16(41, N, H, 128, scale=2.0))
    cent = synth.bits(synth.gaussian_bf16(42, H, C, 128))
    o = orc.quantize(kb, cent, G=G, r=0, M=2, is_key=True, two_level_scales=True)
    x = orc.bf16_to_f32(kb).astype(np.float64)
    mu = orc.bf16_to_f32(cent).astype(np.float64)
    s2 = orc.f16_to_f32(o["s2"]).astype(np.float64)
    khat = orc.dequant(o, cent, G=G, r=0)
    for i in range(N):
        for h in range(H):
            res = x[i, h] - mu[h, o["ids"][i, h]]
            for g in range(128 // G):
                rg = res[g * G:(g + 1) * G]
                s32 = np.float32((np.float32(max(rg.max(), 0.0)) - np.float32(min(rg.min(), 0.0))) / np.float32(3.0))
                c = int(o["scode"][i, h, g])
                assert c * s2[i, h] >= s32 and (c == 0 or (c - 1) * s2[i, h] < s32)
                step = c * s2[i, h]
                assert np.all(np.abs(khat[i, h, g * G:(g + 1) * G] - x[i, h, g * G:(g + 1) * G]) <= step / 2 + 1e-12)


def test_two_level_scales_zero_token_and_psac_layout(orc):
    kb, cent = _one_token_chunk([np.zeros(32)] * 4)
    o = orc.quantize(kb, cent, G=32, r=0, M=1, is_key=True, two_level_scales=True)
    assert o["s2"][0, 0] == 0 and np.all(o["scode"] == 0) and np.all(o["codes"] == 0)
    # App. D.1 layout choice, reading: dense N (r + 2) bytes, sparse K (r + 4) + 4
    kept = np.zeros(100, bool)
    kept[:10] = True
    assert orc.psac_layout_bytes(kept, 8) == (1000, 124, 124)
    kept[:] = True
    assert orc.psac_layout_bytes(kept, 8) == (1000, 1204, 1000)


def test_psac_tile_layout_hand_cases(orc):
    """Per-tile layout choice (App. D.1, reading: dense n_t (r + 2) bytes,
    sparse 16-byte keep mask + K_t (r + 2)): hand-counted boundary cases."""
    k = np.zeros(128, bool)
    k[:10] = True                                    # 10 kept of 128, r = 16
    sp, nb = orc.psac_tile_layout(k, 16)
    assert list(sp) == [True] and list(nb) == [16 + 10 * 18]
    k[:] = True                                      # all kept: the mask only adds
    assert orc.psac_tile_layout(k, 16)[0].tolist() == [False]
    assert orc.psac_tile_layout(k, 16)[1].tolist() == [128 * 18]
    k[5] = False                                     # 127 kept: 16 + 127*18 = 2302 < 2304
    assert orc.psac_tile_layout(k, 16)[0].tolist() == [True]
    assert orc.psac_tile_layout(k, 16)[1].tolist() == [2302]
    assert orc.psac_tile_layout(k, 8)[0].tolist() == [False]   # r = 8: 16 + 127*10 = 1286 > 1280
    k[6] = False                                                # 126 kept, r = 8: 1276 < 1280
    assert orc.psac_tile_layout(k, 8)[1].tolist() == [1276]
    # two tiles and a ragged tail of 72 tokens, all kept in the tail: dense there
    k3 = np.zeros(328, bool)
    k3[:64] = True
    k3[256:] = True
    sp, nb = orc.psac_tile_layout(k3, 16)
    assert sp.tolist() == [True, True, False]
    assert nb.tolist() == [16 + 64 * 18, 16, 72 * 18]



# ------------------------------------------------------------------ full-matrix distance (App. C.4 ablation)
def test_full_matrix_distance_reduces_to_diagonal_and_matches_fp64(orc):
    """With M = diag(w) the full quadratic form is Eq. 9's diagonal distance:
    same candidates and ids wherever the decision margins are clear.  With a
    dense symmetric positive M, the candidates are the M smallest fp64 values
    of (k - mu)^T M (k - mu) (brute force) wherever the margin is clear."""
    H, N, C, G, Mc = 2, 60, 16, 32, 4
    kb = synth.bits(synth.gaussian_bf16(51, N, H, 128))
    cent = synth.bits(synth.gaussian_bf16(52, H, C, 128))
    w = synth.random_weights(53, H, 128).numpy()
    Md = np.stack([np.diag(w[h]) for h in range(H)]).astype(np.float32)
    a = orc.quantize(kb, cent, G=G, r=0, M=Mc, is_key=True, w=w)
    b = orc.quantize(kb, cent, G=G, r=0, M=Mc, is_key=True, w=w, M_full=Md)
    clear = (a["m_topm"] > 1e-5) & (b["m_topm"] > 1e-5) & (a["m_sel"] > 1e-5)
    assert clear.mean() > 0.9
    assert np.array_equal(np.sort(a["cand"], -1)[clear], np.sort(b["cand"], -1)[clear])
    assert np.array_equal(a["ids"][clear], b["ids"][clear])
    rng = np.random.default_rng(54)
    R = rng.standard_normal((H, 128, 128))
    Mf = (np.einsum("hij,hkj->hik", R, R) / 128).astype(np.float32)
    c = orc.quantize(kb, cent, G=G, r=0, M=Mc, is_key=True, w=w, M_full=Mf)
    x = orc.bf16_to_f32(kb).astype(np.float64)
    mu = orc.bf16_to_f32(cent).astype(np.float64)
    for i in range(N):
        for h in range(H):
            e = x[i, h][None, :] - mu[h]
            dfull = np.einsum("jc,cd,jd->j", e, Mf[h].astype(np.float64), e)
            order = np.argsort(dfull, kind="stable")
            gap = (dfull[order[Mc]] - dfull[order[Mc - 1]]) / abs(dfull[order[Mc]])
            if gap > 1e-4:
                assert set(c["cand"][i, h]) == set(order[:Mc])
