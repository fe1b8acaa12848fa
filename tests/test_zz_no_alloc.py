"""The allocation-free k-means entry point (qwm_fit_centroids_noalloc).

It serves callers that cannot give the library device scratch (a plain C host
program holding only its input/output tensors, or an engine whose memory pool
forbids cudaMalloc mid-generation); its scratch is a static device array
shared by every call.  This file is collected last so that a run stopping at
its first failure has already run every other test.
"""
import numpy as np
import pytest
import torch

import paper_2609_26425_gb300 as qwm
from paper_2609_26425_gb300 import synth

pytestmark = pytest.mark.gpu


def test_noalloc_fit_matches_workspace_fit_on_consecutive_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    # two different calls in a row, then the first again: each must match the
    # workspace entry point exactly, whatever the previous call left behind
    cases = [(4, 880, 64, 10, 1), (40, 1000, 256, 3, 2), (4, 880, 64, 10, 1)]
    for H, N, C, iters, seed in cases:
        cfg = qwm.config(H, C, kmeans_iters=iters)
        x = synth.gaussian_bf16(seed, N, H, 128).cuda()
        ref = qwm.qwm_fit_centroids(cfg, x)
        got = qwm.qwm_fit_centroids_noalloc(cfg, x)
        torch.cuda.synchronize()
        assert torch.equal(got, ref), (H, N, C)


def test_noalloc_fit_rejects_sizes_beyond_the_static_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cfg = qwm.config(64, 256, kmeans_iters=1)  # centroids 8 MiB + operand images 8 MiB + more > 16 MiB
    x = synth.gaussian_bf16(3, 300, 64, 128).cuda()
    with pytest.raises(qwm.QwmError) as e:
        qwm.qwm_fit_centroids_noalloc(cfg, x)
    assert e.value.status == 3
