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
