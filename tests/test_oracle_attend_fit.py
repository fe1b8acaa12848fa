"""Pins for the oracle's attention, k-means fitting and Query statistics.

Attention (Sec. 3.3 Eq. 5 logits, softmax) is checked against closed forms
(one key, equal logits) and torch's scaled_dot_product_attention in fp64.
k-means (Sec. 2, QVG convention) is checked against closed forms (one
cluster = mean), Lloyd invariants (non-increasing objective, fixed points) and
scikit-learn's Lloyd k-means.  Query statistics (Eq. 6, 7, 8, 15) are checked
against the identity of Eq. 7 and the eigen-decomposition.
"""
import numpy as np
import pytest
import torch

from paper_2609_26425_gb300 import synth


# ------------------------------------------------------------------ attention
def test_attend_single_key_returns_value(orc):
    q = synth.bits(synth.gaussian_bf16(1, 5, 2, 128))
    k = np.random.default_rng(1).standard_normal((1, 2, 128))
    v = np.random.default_rng(2).standard_normal((1, 2, 128))
    out, lse = orc.attend(q, k, v, 1 / np.sqrt(128))
    assert np.allclose(out, np.broadcast_to(v, out.shape), rtol=0, atol=1e-15)


def test_attend_equal_logits_is_mean(orc):
    q = synth.bits(synth.gaussian_bf16(3, 4, 1, 128))
    k = np.broadcast_to(np.random.default_rng(3).standard_normal((1, 1, 128)), (37, 1, 128)).copy()
    v = np.random.default_rng(4).standard_normal((37, 1, 128))
    out, lse = orc.attend(q, k, v, 0.1)
    assert np.allclose(out, np.broadcast_to(v.mean(0), out.shape), rtol=0, atol=1e-13)


def test_attend_matches_torch_sdpa(orc):
    Nq, Nk, H, d = 33, 301, 3, 128
    qb = synth.bits(synth.gaussian_bf16(5, Nq, H, d))
    rng = np.random.default_rng(5)
    k = rng.standard_normal((Nk, H, d)) * 1.5
    v = rng.standard_normal((Nk, H, d))
    scale = 1 / np.sqrt(d)
    out, lse = orc.attend(qb, k, v, scale)
    qf = torch.from_numpy(orc.bf16_to_f32(qb).astype(np.float64)).permute(1, 0, 2)
    kt = torch.from_numpy(k).permute(1, 0, 2)
    vt = torch.from_numpy(v).permute(1, 0, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(qf, kt, vt, scale=scale).permute(1, 0, 2)
    assert np.allclose(out, ref.numpy(), rtol=1e-12, atol=1e-12)
    lref = torch.logsumexp(torch.einsum("hqd,hkd->hqk", qf, kt) * scale, -1).numpy()
    assert np.allclose(lse, lref, rtol=1e-12, atol=1e-12)
    # row subset returns the same rows
    rows = np.array([0, 7, 32], np.int64)
    o2, l2 = orc.attend(qb, k, v, scale, rows=rows)
    assert np.array_equal(o2, out[rows]) and np.array_equal(l2, lse[:, rows])


# ------------------------------------------------------------------ k-means
def test_fit_one_cluster_is_mean(orc):
    N, H, d = 257, 2, 128
    x = synth.bits(synth.gaussian_bf16(11, N, H, d))
    o = orc.fit_centroids(x, C=1, iters=2)
    xf = orc.bf16_to_f32(x).astype(np.float64)
    mean = xf.mean(0)  # [H][d]
    ref = torch.from_numpy(mean.astype(np.float32)).to(torch.bfloat16)
    assert np.array_equal(o["centroids"][:, 0], synth.bits(ref))


def test_fit_objective_non_increasing_and_fixed_point(orc):
    N, H, d, C = 600, 2, 128, 16
    x = synth.bits(synth.gaussian_bf16(12, N, H, d))
    o = orc.fit_centroids(x, C=C, iters=8)
    obj = o["objective"]
    assert np.all(obj[1:] <= obj[:-1] * (1 + 1e-6))
    # well separated clusters: Lloyd reaches its fixed point and stays there
    rng = np.random.default_rng(13)
    centers = rng.standard_normal((C, d)) * 20
    lab = np.arange(N) % C
    xs = centers[lab][:, None, :] + rng.standard_normal((N, 1, d)) * 0.1
    xb = synth.bits(torch.from_numpy(xs.astype(np.float32)).to(torch.bfloat16))
    a = orc.fit_centroids(xb, C=C, iters=6)
    b = orc.fit_centroids(xb, C=C, iters=9)
    assert np.array_equal(a["centroids"], b["centroids"])
    assert np.array_equal(a["assign"], b["assign"])


def test_fit_init_is_strided_tokens(orc):
    N, H, d, C = 100, 1, 128, 7
    x = synth.bits(synth.gaussian_bf16(14, N, H, d))
    o = orc.fit_centroids(x, C=C, iters=0)
    idx = (np.arange(C) * N) // C
    assert np.array_equal(o["centroids"][0], x[idx, 0])


def tokens(rows, d=128):
    """bf16 bits [N][1][d] of tokens given by their first channels."""
    x = np.zeros((len(rows), 1, d), np.float32)
    for i, row in enumerate(rows):
        x[i, 0, : len(row)] = row
    return synth.bits(torch.from_numpy(x).to(torch.bfloat16))


def first_channels(bits, n):
    return orc_f32(bits)[..., :n]


def orc_f32(bits):
    return (np.asarray(bits, np.uint32) << 16).view(np.float32)


def test_fit_tie_goes_to_lower_index(orc):
    """A token at exactly the same distance from two centroids joins the one
    with the lower index (the assignment convention of k-means in Sec. 2).
    Tokens (2, 0), (-2, 0), (0, 1); initial centroids are tokens 0 and 1
    (token floor(j N / C)); token 2 is at distance 5 from both, so it joins
    cluster 0: after one step the centroids are (1, 0.5) and (-2, 0) -- the
    other choice would give (2, 0) and (-1, 0.5)."""
    x = tokens([(2.0, 0.0), (-2.0, 0.0), (0.0, 1.0)])
    o = orc.fit_centroids(x, C=2, iters=1)
    c = first_channels(o["centroids"][0], 3)
    assert np.array_equal(c, np.array([[1.0, 0.5, 0.0], [-2.0, 0.0, 0.0]], np.float32))
    assert not orc_f32(o["centroids"][0])[:, 3:].any()
    assert list(o["assign"][:, 0]) == [0, 1, 0]


def test_fit_empty_cluster_keeps_its_centroid(orc):
    """An empty cluster keeps its previous centroid (Sec. 2 k-means; Lloyd's
    update has no mean for it).  Tokens (1, 0), (1, 0.5), (1, 0), (1, 1.5);
    the initial centroids are tokens 0 and 2, which are equal, so every token
    is equally far from both and joins cluster 0 (lower index): cluster 1 is
    empty after the first step and stays at (1, 0) while cluster 0 moves to
    the mean (1, 0.5).  The second step splits the tokens: (1, 0) and (1, 0)
    go to cluster 1, the others to cluster 0, whose mean is (1, 1)."""
    x = tokens([(1.0, 0.0), (1.0, 0.5), (1.0, 0.0), (1.0, 1.5)])
    o1 = orc.fit_centroids(x, C=2, iters=1)
    assert np.array_equal(first_channels(o1["centroids"][0], 2), np.array([[1.0, 0.5], [1.0, 0.0]], np.float32))
    o2 = orc.fit_centroids(x, C=2, iters=2)
    assert np.array_equal(first_channels(o2["centroids"][0], 2), np.array([[1.0, 1.0], [1.0, 0.0]], np.float32))
    assert list(o2["assign"][:, 0]) == [1, 0, 1, 0]


def test_fit_matches_sklearn_lloyd(orc):
    sk = pytest.importorskip("sklearn.cluster")
    N, H, d, C, iters = 800, 1, 128, 12, 6
    x = synth.bits(synth.gaussian_bf16(15, N, H, d))
    o = orc.fit_centroids(x, C=C, iters=iters)
    xf = orc.bf16_to_f32(x)[:, 0].astype(np.float64)
    init = xf[(np.arange(C) * N) // C]
    km = sk.KMeans(n_clusters=C, init=init, n_init=1, max_iter=iters, tol=0.0, algorithm="lloyd")
    km.fit(xf)
    assert np.allclose(o["cent_f32"][0], km.cluster_centers_, rtol=1e-5, atol=1e-5)


# ------------------------------------------------------------------ Query statistics
def test_query_stats_identities(orc):
    N, H, d, r = 900, 2, 128, 8
    src = synth.ChunkSource(synth.WORKLOADS["single_layer_h4"])
    q, _, _ = src.chunk(0, tokens=N)
    qb = synth.bits(q[:, :H])
    M, w, U, lam = orc.query_stats(qb, r)
    qf = orc.bf16_to_f32(qb).astype(np.float64)
    e = np.random.default_rng(16).standard_normal((H, d))
    # Eq. 7: mean over the queries of (q^T e)^2 equals e^T M e
    lhs = np.einsum("nhd,hd->nh", qf, e) ** 2
    rhs = np.einsum("hd,hde,he->h", e, M, e)
    assert np.allclose(lhs.mean(0), rhs, rtol=1e-10)
    # Eq. 8: weights are the diagonal normalised to mean one
    assert np.allclose(w.mean(-1), 1.0, rtol=1e-6)
    # Eq. 15: U orthonormal eigenvectors, eigenvalues sorted decreasing
    for h in range(H):
        assert np.allclose(U[h].T @ U[h], np.eye(r), atol=1e-10)
        assert np.allclose(M[h] @ U[h], U[h] * lam[h, :r], atol=1e-8)
        assert np.all(np.diff(lam[h]) <= 1e-12)


def test_query_stats_hadamard_closed_form(orc):
    """Queries s_n * had_n along orthogonal +-1 rows (N = d = 128): by Eq. 6,
    M = (1/N) sum_n s_n^2 had_n had_n^T, whose eigenvectors are the rows
    had_n / sqrt(d) with eigenvalues s_n^2 (had_n^T had_n = d = N), and whose
    diagonal is the constant mean(s^2), so Eq. 8 gives w = 1 exactly."""
    H, d, r = 2, 128, 16
    q = synth.hadamard_queries(H, d)
    had = q[:, 0].float() / (torch.arange(d, dtype=torch.float32) + 1)[:, None]
    M, w, U, lam = orc.query_stats(synth.bits(q), r)
    assert np.all(w == 1.0)
    for h in range(H):
        s = np.arange(1, d + 1, dtype=np.float64) if h % 2 == 0 else np.arange(d, 0, -1, dtype=np.float64)
        assert np.allclose(lam[h], np.sort(s ** 2)[::-1], rtol=1e-12)
        top = np.argsort(-s, kind="stable")[:r]
        for j in range(r):
            ref = had[top[j]].double().numpy() / np.sqrt(d)
            assert abs(abs(np.dot(U[h][:, j], ref)) - 1.0) < 1e-10


def test_query_stats_diagonal_weights(orc):
    """Query n = v_n e_n (one channel each): M = diag(v^2) / N, so Eq. 8 gives
    w_c = v_c^2 / mean(v^2) and the eigenvectors are the unit channels in
    decreasing v.  Values v_n = 1 + n/128 are exact in bf16."""
    d, r = 128, 8
    v = 1.0 + np.arange(d) / 128.0
    q = np.zeros((d, 1, d), np.float32)
    q[np.arange(d), 0, np.arange(d)] = v
    qb = synth.bits(torch.from_numpy(q).to(torch.bfloat16))
    M, w, U, lam = orc.query_stats(qb, r)
    assert np.allclose(M[0], np.diag(v ** 2) / d, rtol=0, atol=1e-15)
    assert np.allclose(w[0], v ** 2 / np.mean(v ** 2), rtol=1e-6)
    for j in range(r):
        assert abs(abs(U[0][d - 1 - j, j]) - 1.0) < 1e-12


def test_query_stats_cold_start_and_zero_queries(orc):
    """No Query seen: w = 1, U = 0 (App. C.3).  Only zero Queries: Eq. 8 is
    0/0 and the head keeps the cold-start weights w = 1."""
    H, d, r = 3, 128, 8
    M, w, U, lam = orc.query_stats(np.zeros((0, H, d), np.uint16), r)
    assert np.all(w == 1.0) and np.all(U == 0.0) and np.all(M == 0.0)
    M, w, U, lam = orc.query_stats(np.zeros((5, H, d), np.uint16), r)
    assert np.all(w == 1.0) and np.all(lam == 0.0)


# ------------------------------------------------------------------ token selection (top-1 key)
def test_top1_brute_force_and_ties(orc):
    """Pure-Python loops on a small case; a duplicated best key goes to the
    lower index; a single key has margin inf."""
    rng = np.random.default_rng(21)
    Nq, Nk, H, d = 6, 9, 2, 128
    qb = synth.bits(torch.from_numpy(rng.standard_normal((Nq, H, d)).astype(np.float32)).to(torch.bfloat16))
    k = rng.standard_normal((Nk, H, d))
    k[7] = k[2]                                   # a duplicate of key 2
    idx, margin, _ = orc.top1(qb, k)
    qf = orc.bf16_to_f32(qb).astype(np.float64)
    for h in range(H):
        for n in range(Nq):
            logits = [sum(qf[n, h, c] * k[j, h, c] for c in range(d)) for j in range(Nk)]
            best = max(logits)
            first = min(j for j in range(Nk) if logits[j] == best)
            assert idx[h, n] == first
            assert idx[h, n] != 7                 # the duplicate never wins over key 2
            srt = sorted(logits, reverse=True)
            assert abs(margin[h, n] - (srt[0] - srt[1])) <= 1e-9 * abs(srt[0])
    idx1, m1, _ = orc.top1(qb, k[:1])
    assert np.all(idx1 == 0) and np.all(np.isinf(m1))


def test_top1_closed_form_and_shift_ratio(orc):
    """Keys along the unit channels with weights 1..d: query e_c picks the key
    of channel c; swapping two keys changes exactly the queries that picked
    them, so the shift ratio is 2/d."""
    d = 128
    k = np.zeros((d, 1, d))
    k[np.arange(d), 0, np.arange(d)] = 1.0 + np.arange(d)
    q = np.zeros((d, 1, d), np.float32)
    q[np.arange(d), 0, np.arange(d)] = 1.0
    qb = synth.bits(torch.from_numpy(q).to(torch.bfloat16))
    idx, _, _ = orc.top1(qb, k)
    assert np.array_equal(idx[0], np.arange(d))
    k2 = k.copy()
    k2[[3, 40]] = k2[[40, 3]]
    idx2, _, _ = orc.top1(qb, k2)
    assert orc.top1_shift(idx, idx) == 0.0
    assert orc.top1_shift(idx, idx2) == 2.0 / d
