"""The window queries' log-sum-exp (the input of the given-LSE entry point):
the oracle against torch.logsumexp and against the oracle's own softmax."""
import numpy as np
import torch

import oracle


def test_window_lse_matches_torch_logsumexp_and_softmax_rows():
    rng = np.random.default_rng(4)
    lens = [23, 9, 4]
    W, Hq, Hkv, d = 6, 4, 2, 16
    cu = np.concatenate([[0], np.cumsum(lens)])
    q = rng.normal(size=(3, Hq, W, d))
    k = rng.normal(size=(int(cu[-1]), Hkv, d))
    lse = oracle.window_lse(q, k, cu, W, scale=0.3)
    for s, L in enumerate(lens):
        for h in range(Hq):
            ku = torch.tensor(k[cu[s]:cu[s + 1], h // 2])
            for w in range(W):
                p = L - W + w
                if p < 0:
                    assert lse[s, h, w] == 0.0
                    continue
                z = 0.3 * (ku[:p + 1] @ torch.tensor(q[s, h, w]))
                assert abs(lse[s, h, w] - torch.logsumexp(z, 0).item()) < 1e-12
    # exp(z - lse) is the oracle's softmax row
    A = oracle.window_attention(q[0, 1], k[:23, 0], 0.3)
    for w in range(W):
        p = 23 - W + w
        z = 0.3 * (k[:p + 1, 0] @ q[0, 1, w])
        np.testing.assert_allclose(np.exp(z - lse[0, 1, w]), A[w, :p + 1], rtol=1e-12)
