"""GPU parity of the brute-force grid top-m (Eq. 5, or Eq. 2 with product
keys) against the oracle's uo_exact_topm, and the recall of the two-phase
search measured with it."""
import numpy as np
import pytest
import torch

import oracle
from paper_2411_12364_gb300 import binding, workloads
from tests import parity

pytestmark = pytest.mark.gpu


def _layer(cfg, B, w=None):
    w = workloads.make_weights(cfg, device="cuda") if w is None else w
    x = workloads.make_tokens(cfg, B, device="cuda")
    t = parity.numpy_inputs(cfg, w, x)
    layer = binding.UltraMemLayer(
        cfg, dict(w, u=torch.from_numpy(t["u"]), t=torch.from_numpy(t["t"])), B)
    return layer, w, x, t


def _full_grid(cfg, t, b, h):
    s_row, s_col = oracle.row_col_scores(cfg, t, b, h)
    return parity.grid(cfg, t, h, s_row, s_col).ravel()


def _compare_exact(cfg, t, tokens, g_idx, g_w, o_idx, o_w):
    """Sets equal, weights within 1e-4 of the head's largest; a differing
    head needs a near-tie at the m-th grid score and valid slots."""
    H, m = int(cfg["heads"]), int(cfg["topm"])
    excused = 0
    for e, b in enumerate(tokens):
        for h in range(H):
            gi, oi = g_idx[b, h], o_idx[e, h]
            if np.array_equal(gi, oi):
                lim = parity.W_TOL * max(np.abs(o_w[e, h]).max(), 1e-30)
                assert np.abs(g_w[b, h] - o_w[e, h]).max() <= lim
                continue
            G = _full_grid(cfg, t, b, h)
            assert parity._gap_is_tie(G, m) or np.array_equal(np.sort(gi), np.sort(oi)), \
                f"exact top-m differs at token {b} head {h} without a near-tie"
            ref = np.sort(G)[::-1][m - 1]
            assert G[gi].min() >= ref - 10 * parity.TIE_REL * np.abs(G).max()
            excused += 1
    return excused


EXACT = [
    dict(dtype=1),
    dict(dtype=0),
    dict(dtype=0, rank=3, d_k=48, heads=3),
    dict(dtype=1, cores=2),
    dict(dtype=1, rank=1, score_mode=1),
    dict(dtype=0, rank=1, score_mode=1, act=1),
    dict(dtype=1, conv_k=3, query_ln=1, ln_eps=1e-5),
    dict(dtype=1, topk=16, topm=200),
]


@pytest.mark.parametrize("case", range(len(EXACT)))
def test_exact_topm_small_layers(case, gpu_lib):
    cfg = workloads.small_config(**EXACT[case])
    B = 9
    layer, w, x, t = _layer(cfg, B)
    g_idx, g_w = layer.retrieve_exact(x)
    torch.cuda.synchronize()
    assert layer.check() == 0
    assert layer.last_launches() >= 2
    o_idx, o_w = oracle.exact_topm(cfg, t, B)
    _compare_exact(cfg, t, range(B), g_idx.cpu().numpy(), g_w.cpu().numpy(), o_idx, o_w)


def test_exact_topm_with_tied_scores(gpu_lib):
    """Every key row equal: every grid score ties, and the top m are the m
    smallest addresses, on both sides (the threshold-tie passes)."""
    cfg = workloads.small_config(dtype=1, topm=40)
    w = workloads.make_weights(cfg, device="cuda")
    w["k_row"][:] = w["k_row"][:, :1]
    w["k_col"][:] = w["k_col"][:, :1]
    layer, w, x, t = _layer(cfg, 5, w)
    g_idx, _ = layer.retrieve_exact(x)
    o_idx, _ = oracle.exact_topm(cfg, t, 5)
    np.testing.assert_array_equal(g_idx.cpu().numpy(), o_idx)
    np.testing.assert_array_equal(o_idx[0, 0], np.arange(40))


def test_exact_topm_decode_1m_and_recall(gpu_lib):
    """The decode-shaped layer: the GPU's exact top-m on a sample of tokens
    against the oracle's brute force, and the recall of the two-phase search
    (forward) against it, which the oracle reproduces on the same tokens."""
    cfg = workloads.layer_config("decode_1m")
    B = 64
    layer, w, x, t = _layer(cfg, B)
    g_idx, g_w = layer.retrieve_exact(x)
    _, a_idx, _ = layer.forward(x, with_slots=True)
    torch.cuda.synchronize()
    assert layer.check() == 0
    g_idx, g_w, a_idx = g_idx.cpu().numpy(), g_w.cpu().numpy(), a_idx.cpu().numpy()
    sample = np.array([0, 13, 31, 63])
    o_idx, o_w = oracle.exact_topm(cfg, t, B, tokens=sample)
    _compare_exact(cfg, t, sample, g_idx, g_w, o_idx, o_w)
    m = cfg["topm"]
    rec = np.array([[len(set(a_idx[b, h]) & set(g_idx[b, h])) / m for h in range(cfg["heads"])]
                    for b in range(B)])
    _, oa_idx, _ = oracle.forward(cfg, t, B, tokens=sample)
    o_rec = np.array([[len(set(oa_idx[e, h]) & set(o_idx[e, h])) / m
                       for h in range(cfg["heads"])] for e in range(len(sample))])
    assert np.abs(rec[sample] - o_rec).max() <= 1.0 / m   # at most one near-tie swap
    assert 0.5 < rec.mean() <= 1.0


def test_product_keys_recall_is_one(gpu_lib):
    """The product-key two-phase search is exact (k >= m): the forward's
    slots are the brute force's."""
    cfg = workloads.layer_config("decode_1m", rank=1, score_mode=1)
    layer, w, x, t = _layer(cfg, 32)
    g_idx, _ = layer.retrieve_exact(x)
    _, a_idx, _ = layer.forward(x, with_slots=True)
    torch.cuda.synchronize()
    g, a = g_idx.cpu().numpy(), a_idx.cpu().numpy()
    same = np.mean([np.array_equal(np.sort(g[b, h]), np.sort(a[b, h]))
                    for b in range(32) for h in range(cfg["heads"])])
    assert same >= 0.99
