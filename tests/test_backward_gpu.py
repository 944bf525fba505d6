"""GPU parity of the lookup-reduce backward (S7-S9; App. D's fused operator)
against the oracle's uo_lookup_reduce_backward: dL/dV (accumulated), dL/dw
per slot and value slice, dL/dW_p."""
import numpy as np
import pytest
import torch

import oracle
from paper_2411_12364_gb300 import binding, workloads
from tests import parity

pytestmark = pytest.mark.gpu

# The rule of the outputs, element-wise with a floor, at the storage's
# tolerance (1e-4 fp32, 2e-2 bf16); and, for every storage, the normwise
# error of each gradient within 1e-4 of its largest entry.
NORM_TOL = 1e-4


def _check(got, want, what, cfg):
    """max_e |got - want| / max(|want_e|, 1e-3 max |want|) over the whole
    gradient, and max_e |got - want| / max |want|."""
    got = np.asarray(got, np.float64).reshape(1, -1)
    want = np.asarray(want, np.float64).reshape(1, -1)
    err, norm = parity.output_errors(got, want)
    tol = parity.out_tol(cfg)
    assert err.max() <= tol, f"{what}: element-wise {err.max():.3g} > {tol}"
    assert norm.max() <= NORM_TOL, f"{what}: normwise {norm.max():.3g} > {NORM_TOL}"


def _run(cfg, B, repeat=False, bad=False):
    w = workloads.make_weights(cfg, device="cuda")
    x = workloads.make_tokens(cfg, B, device="cuda")
    t = parity.numpy_inputs(cfg, w, x)
    layer = binding.UltraMemLayer(
        cfg, dict(w, u=torch.from_numpy(t["u"]), t=torch.from_numpy(t["t"])), B)
    _, idx, wt = layer.forward(x, with_slots=True)
    torch.cuda.synchronize()
    if repeat:   # a row gathered by several tokens and heads accumulates
        idx[1:, 0, 0] = idx[0, 0, 0]
    if bad:
        idx[B - 1, 0, 1] = -5
    gen = torch.Generator(device="cpu").manual_seed(7)
    g = torch.randn((B, cfg["d_out"]), generator=gen).to(layer.dtype).cuda()
    dv, dw, dwp = layer.lookup_reduce_backward(idx, wt, g)
    torch.cuda.synchronize()
    st = layer.check()
    idx_n, w_n = idx.cpu().numpy(), wt.cpu().numpy().astype(np.float64)
    if bad:
        assert st == binding.EDEVICE
        assert (dw[B - 1, 0, 1] == 0).all()
        idx_n = idx_n.copy()
        w_n = w_n.copy()
        idx_n[B - 1, 0, 1] = 0
        w_n[B - 1, 0, 1] = 0.0   # a skipped slot contributes nothing
    else:
        assert st == 0
    o_dv, o_dw, o_dwp = oracle.lookup_reduce_backward(cfg, t, idx_n, w_n,
                                                      workloads.stored_numpy(g))
    _check(dv.cpu().numpy(), o_dv, "dV", cfg)
    if bad:   # the skipped slot's dw is 0 on the GPU
        o_dw[B - 1, 0, 1] = 0.0
    _check(dw.cpu().numpy(), o_dw, "dw", cfg)
    if dwp is not None:
        _check(dwp.cpu().numpy(), o_dwp, "dW_p", cfg)
    return layer


CASES = [
    dict(dtype=1),
    dict(dtype=0),
    dict(dtype=1, cores=2),
    dict(dtype=0, expand_e=1, has_proj=0, d_out=64, n=40),
    dict(dtype=1, expand_e=9, n=11, d_out=72, heads=3),
]


@pytest.mark.parametrize("case", range(len(CASES)))
def test_backward_small_layers(case, gpu_lib):
    cfg = workloads.small_config(**CASES[case])
    _run(cfg, 37)


def test_backward_repeated_rows(gpu_lib):
    _run(workloads.small_config(dtype=1), 20, repeat=True)


def test_backward_bad_address_is_skipped(gpu_lib):
    _run(workloads.small_config(dtype=1), 9, bad=True)


def test_backward_decode_1m(gpu_lib):
    """The decode-shaped layer (64 tokens), every gradient: slots, gather
    and the CUDA-core dW_p over few tokens, then the tensor-core dacc and
    the rows kernel."""
    layer = _run(workloads.layer_config("decode_1m"), 64)
    assert layer.last_launches() == 5


@pytest.mark.parametrize("B", [256, 260])
def test_backward_many_tokens(B, gpu_lib):
    """256 tokens take the tensor-core dW_p (tokens on K, both operands
    transposed, the pooled rows as two bf16 terms); 260 (not a multiple of
    8) the CUDA-core one."""
    layer = _run(workloads.layer_config("decode_1m"), B)
    assert layer.last_launches() == (8 if B % 8 == 0 else 5)
