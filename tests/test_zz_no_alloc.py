"""w8a8_act_stats_noalloc: the statistics of one batch with the library's
static scratch give the same results as the caller-accumulator path
(w8a8_act_stats_update + w8a8_act_stats_finalize), on two calls in a row
(the second must not see the first's sums), and reject K beyond the scratch."""

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _reference(w8, X, shift):
    T, K = X.shape
    sums = torch.zeros(4, K, dtype=torch.float64, device=X.device)
    absmax = torch.zeros(K, dtype=torch.float32, device=X.device)
    w8.act_stats_update(X, sums, absmax, shift=shift)
    return w8.act_stats_finalize(sums, absmax, T, shift=shift)


def test_noalloc_stats_two_calls_match_accumulator_path():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12280_gb300 import w8a8
    w8a8.lib()
    dev = "cuda"
    for T, K, seed in ((300, 528, 1), (129, 4096, 2)):
        X = torch.from_numpy(wl.random_bf16((T, K), seed=seed, scale=1.0 + seed).view(np.int16)) \
            .view(torch.bfloat16).to(dev)
        shift = torch.full((K,), 0.25, dtype=torch.float32, device=dev)
        for sh in (None, shift):
            chan, tensor = w8a8.act_stats_noalloc(X, shift=sh)
            want_c, want_t = _reference(w8a8, X, sh)
            torch.cuda.synchronize()
            assert torch.equal(chan[0], want_c[0])                      # max-abs exact
            torch.testing.assert_close(chan, want_c, rtol=1e-6, atol=1e-7)
            torch.testing.assert_close(tensor, want_t, rtol=1e-6, atol=1e-7)
    assert w8a8.device_status() == 0


def test_noalloc_stats_limits():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12280_gb300 import w8a8
    K = w8a8.NOALLOC_STATS_MAX_K
    X = torch.randn(3, K, device="cuda").to(torch.bfloat16)
    chan, tensor = w8a8.act_stats_noalloc(X)                          # the largest K works
    want_c, want_t = _reference(w8a8, X, None)
    torch.testing.assert_close(chan, want_c, rtol=1e-6, atol=1e-7)
    big = torch.zeros(2, K + 16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(w8a8.W8A8Error):
        w8a8.act_stats_noalloc(big)
