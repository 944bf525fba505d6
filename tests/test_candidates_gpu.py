"""The scoring's two forms on the tensor-core path (Eq. 6-9): every rank-1
key written and ranked by the selection, or two scoring passes that leave
per-axis candidate lists (the keys at or above tau, a bound at most the k-th
largest maximum of the axis' groups of 16 keys); by default the lists serve
long grids and every key the others.  Both rank the same fp32
keys by (score, smaller index), so the selected slots, their weights and
the output must be identical bit for bit; the lists are also checked against
the oracle directly.  Tied keys fill a list past the selection's 1024-entry
buffer (then an exact radix select over the list's composites replaces it)
or past its sorting size (then it is tightened first)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2411_12364_gb300 import binding, workloads
from tests import parity

pytestmark = pytest.mark.gpu

EVERY_KEY, LISTS, AUTO = 0, 1, 2


def _layer(cfg, w, B):
    x = workloads.make_tokens(cfg, B, 0, device="cuda")
    t = parity.numpy_inputs(cfg, w, x)
    lw = dict(w, u=torch.from_numpy(t["u"]), t=torch.from_numpy(t["t"]))
    return binding.UltraMemLayer(cfg, lw, B), x, t


def _forward(layer, x, mode):
    layer.candidates(mode)
    out, idx, wt = layer.forward(x, with_slots=True)
    torch.cuda.synchronize()
    assert layer.check() == 0
    return out.cpu(), idx.cpu(), wt.cpu(), layer.last_launches()


def _tied(cfg, rows):
    w = workloads.make_weights(cfg, device="cuda")
    for name in ("k_row", "k_col"):
        k = w[name].clone()
        k[:, :rows, :] = k[:, :1, :]
        w[name] = k
    return w


CASES = [
    # (overrides, tokens, keys tied per axis)
    (dict(dtype=1, n=600, topk=16, topm=32), 37, 0),
    (dict(dtype=1, n=601, topk=64, topm=64), 9, 0),        # K = 1202: a partial last group
    (dict(dtype=1, n=600, topk=75, topm=64), 9, 0),        # k = G = 75 groups
    (dict(dtype=1, n=600, topk=16, topm=32, cores=2), 21, 0),   # MCS
    (dict(dtype=1, n=600, rank=1, score_mode=1, topk=16, topm=16), 21, 0),   # product keys
    (dict(dtype=1, n=600, topk=16, topm=32, share_query=0), 13, 0),
    (dict(dtype=1, n=600, topk=16, topm=32, rank=3, d_k=48), 13, 0),
    (dict(dtype=1, n=600, topk=16, topm=32), 17, 1200),    # all tied: 1200 > 1024 listed
    (dict(dtype=1, n=600, topk=16, topm=32), 17, 500),     # 500 tied: tightened first
    (dict(dtype=1, n=2400, topk=64, topm=64), 5, 0),       # K = 4800
    # more tiles than SMs: the passes keep each token block's query terms
    # resident and change block inside a CTA's share of the tiles
    (dict(dtype=1, n=2400, topk=64, topm=64), 300, 0),
    (dict(dtype=1, n=1000, topk=32, topm=32, heads=3), 260, 0),
]


@pytest.mark.parametrize("over,B,tied", CASES, ids=[str(i) for i in range(len(CASES))])
def test_lists_select_what_every_key_selects(over, B, tied, gpu_lib):
    cfg = workloads.small_config(**over)
    w = _tied(cfg, tied) if tied else workloads.make_weights(cfg, device="cuda")
    layer, x, t = _layer(cfg, w, B)
    o1, i1, w1, n1 = _forward(layer, x, EVERY_KEY)
    o2, i2, w2, n2 = _forward(layer, x, LISTS)
    assert n2 == n1 + 2   # the group-maxima pass and the bound
    assert torch.equal(i1, i2)
    assert torch.equal(w1, w2)
    assert torch.equal(o1, o2)
    # and against the oracle
    o_out, o_idx, o_w = oracle.forward(cfg, t, B)
    parity.compare(cfg, t, np.arange(B), o2.float().numpy(), i2.numpy(), w2.numpy(), o_out,
                   o_idx, o_w)
    layer.close()


def test_lists_at_the_decode_workload(gpu_lib):
    """decode_1m (2048 keys an axis, k = 32) with the lists forced: the same
    selection as every key."""
    cfg = workloads.layer_config("decode_1m")
    layer, x, t = _layer(cfg, workloads.make_weights(cfg, device="cuda"), 64)
    o1, i1, w1, _ = _forward(layer, x, EVERY_KEY)
    o2, i2, w2, _ = _forward(layer, x, LISTS)
    assert torch.equal(i1, i2) and torch.equal(w1, w2) and torch.equal(o1, o2)
    layer.close()


def test_lists_at_a_long_grid(gpu_lib):
    """mid_4m with 2048 tokens (4096 keys an axis, 4 heads: 2048 tiles a
    pass) with the lists forced: the same selection as every key."""
    cfg = workloads.layer_config("mid_4m")
    layer, x, _ = _layer(cfg, workloads.make_weights(cfg, device="cuda"), 2048)
    o1, i1, w1, _ = _forward(layer, x, EVERY_KEY)
    o2, i2, w2, _ = _forward(layer, x, LISTS)
    assert torch.equal(i1, i2) and torch.equal(w1, w2) and torch.equal(o1, o2)
    layer.close()


def test_default_form_by_grid(gpu_lib):
    """The default writes every key (one scoring launch) while the list
    passes would have fewer than 3.5 tiles of 128 tokens x 256 keys per SM,
    and takes the lists (three launches) from there on; either form can be
    forced, with the same result."""
    cfg = workloads.small_config(dtype=1, n=600, topk=16, topm=32)
    w = workloads.make_weights(cfg, device="cuda")
    layer = binding.UltraMemLayer(cfg, w, 4096)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    for B in (100, 300, 4096):
        tiles = 5 * ((B + 127) // 128) * 2 * cfg["heads"]   # K = 1200: 5 tiles of 256 keys
        x = workloads.make_tokens(cfg, B, 0, device="cuda")
        out = layer.forward(x)
        assert layer.check() == 0
        assert layer.last_launches() == (7 if 2 * tiles >= 7 * sms else 5)
    assert layer.last_launches() == 7   # 640 tiles
    o_auto, i_auto, w_auto, _ = _forward(layer, x, AUTO)
    o1, i1, w1, n1 = _forward(layer, x, EVERY_KEY)
    assert n1 == 5
    assert torch.equal(i1, i_auto) and torch.equal(w1, w_auto) and torch.equal(o1, o_auto)
    o2, i2, w2, n2 = _forward(layer, x, LISTS)
    assert n2 == 7
    layer.candidates(AUTO)
    layer.forward(x[:100])
    assert layer.last_launches() == 5
    layer.close()


def test_candidate_hook_arguments(gpu_lib):
    cfg = workloads.small_config(dtype=1, n=600, topk=16, topm=32)
    layer = binding.UltraMemLayer(cfg, workloads.make_weights(cfg, device="cuda"), 8)
    for bad in (-1, 3):
        with pytest.raises(binding.UltraMemError):
            layer.candidates(bad)
    layer.close()
    # fp32 storage runs on CUDA cores: no lists
    cfg32 = workloads.small_config(dtype=0, n=600, topk=16, topm=32)
    layer32 = binding.UltraMemLayer(cfg32, workloads.make_weights(cfg32, device="cuda"), 8)
    with pytest.raises(binding.UltraMemError):
        layer32.candidates(LISTS)
    layer32.candidates(EVERY_KEY)
    layer32.candidates(AUTO)    # the default: every key where lists cannot run
    layer32.close()
