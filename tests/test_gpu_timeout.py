"""GPU: the timeout path of the bounded waits, without a GPU fault.

Every wait between the roles of the attention kernel is bounded; when one
runs out the role leaves its loop, the kernel ends on its own and
QWM_ERR_TIMEOUT is recorded in the cache's status word.  The test makes a wait
run out the allowed way: a 1 ms wait limit and the test hook that leaves the
V-rebuild role idle, so the MMA warp waits for a tile that never comes.  It
then checks the status and that the next ordinary call is exact.
"""
import math

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_26425_gb300 import synth
import paper_2609_26425_gb300 as qwm

from parity import compare_attention, oracle_append, oracle_kv, strided_centroids

pytestmark = pytest.mark.gpu
TIMEOUT = 5


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qwm.lib()


def dev(t):
    return t.to("cuda").contiguous()


def test_attend_wait_that_runs_out_records_timeout_and_next_call_is_exact():
    H, N, C, G, r, M = 2, 300, 16, 32, 16, 4
    q = synth.gaussian_bf16(51, N, H, 128)
    k = synth.gaussian_bf16(52, N, H, 128)
    v = synth.gaussian_bf16(53, N, H, 128)
    kb, vb = synth.bits(k), synth.bits(v)
    kc, vc = strided_centroids(kb, C), strided_centroids(vb, C)
    Ub = synth.bits(synth.random_orthonormal(54, H, 128, r))
    cfg = qwm.config(H, C, group_size=G, psac_rank=r, candidates=M)
    cache = qwm.Cache(cfg, N, 1)
    qwm.qwm_quantize_append(cfg, cache, dev(k), dev(v), dev(synth.from_bits(kc)), dev(synth.from_bits(vc)),
                            U=dev(synth.from_bits(Ub)))
    assert cache.status() == 0
    qd = dev(q)
    cache.set_wait_limit(1_000_000)            # 1 ms
    cache.set_idle_role(qwm.QWM_ROLE_V_REBUILD)
    qwm.qwm_attend(cfg, cache, qd, dev(k[:100]), dev(v[:100]))
    torch.cuda.synchronize()                   # the kernel ends by itself
    assert cache.status() == TIMEOUT
    cache.set_idle_role(0)
    cache.set_wait_limit(2_000_000_000)
    out = qwm.qwm_attend(cfg, cache, qd, dev(k[:100]), dev(v[:100]))
    assert cache.status() == 0
    ko, vo = oracle_append(kb, vb, kc, vc, G=G, r=r, M=M, U_bits=Ub)
    K, V = oracle_kv(ko, vo, kc, vc, G=G, r=r, U_bits=Ub)
    K = np.concatenate([K, orc.bf16_to_f32(kb[:100]).astype(np.float64)])
    V = np.concatenate([V, orc.bf16_to_f32(vb[:100]).astype(np.float64)])
    ref, _ = orc.attend(synth.bits(q), K, V, 1 / math.sqrt(128))
    compare_attention(out.float().cpu().numpy(), ref)
