"""GPU parity of the query-side extras (Sec. 3.1): Trick 4's causal depthwise
convolution with its conv state, Trick 2's query LayerNorm, and the key
LayerNorm helper, through the C ABI against the CPU oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2411_12364_gb300 import binding, workloads
from tests import parity

pytestmark = pytest.mark.gpu


def _run_seq(cfg, n_seq, L, gpu_lib, with_state=True, batch_index=0, w=None, layer=None):
    w = workloads.make_weights(cfg, device="cuda") if w is None else w
    B = n_seq * L
    x = workloads.make_tokens(cfg, B, batch_index, device="cuda")
    kc = int(cfg.get("conv_k", 0))
    st_in = st_out = None
    if kc > 1 and with_state:
        st_in = workloads.make_conv_state(cfg, n_seq, batch_index, device="cuda")
    if kc > 1:
        st_out = torch.full((n_seq, kc - 1, cfg["d_in"]), float("nan"),
                            dtype=workloads.torch_dtype(cfg), device="cuda")
    t = parity.numpy_inputs(cfg, w, x)
    t["seq_len"] = L
    if st_in is not None:
        t["conv_state"] = workloads.stored_numpy(st_in)
    if layer is None:
        layer = binding.UltraMemLayer(
            cfg, dict(w, u=torch.from_numpy(t["u"]), t=torch.from_numpy(t["t"])), B)
    out, idx, wt = layer.forward_seq(x, n_seq, st_in, st_out, with_slots=True)
    torch.cuda.synchronize()
    assert layer.check() == 0
    o_out, o_idx, o_w = oracle.forward(cfg, t, B)
    res = parity.compare(cfg, t, np.arange(B), out.float().cpu().numpy(), idx.cpu().numpy(),
                         wt.cpu().numpy(), o_out, o_idx, o_w)
    if kc > 1:
        want = oracle.conv_state(cfg, t, B)
        got = st_out.float().cpu().numpy().astype(np.float64)
        np.testing.assert_array_equal(got, want)
    return layer, (w, x, t, st_out), (out, idx, wt), res


CASES = [
    # (overrides, n_seq, seq_len)
    (dict(dtype=1, conv_k=4), 8, 1),                      # decode: one token a sequence
    (dict(dtype=1, conv_k=4, query_ln=1), 37, 1),
    (dict(dtype=1, conv_k=4, query_ln=1), 3, 30),         # tensor-core query (90 tokens)
    (dict(dtype=1, conv_k=2, query_ln=1, share_query=0), 5, 20),
    (dict(dtype=1, query_ln=1), 7, 1),                    # LayerNorm alone, small query
    (dict(dtype=1, query_ln=1), 2, 50),                   # LayerNorm alone, tensor-core query
    (dict(dtype=1, conv_k=1), 4, 5),                      # one tap: no state
    (dict(dtype=1, conv_k=6, query_ln=1), 6, 2),          # sequences shorter than the state
    (dict(dtype=0, conv_k=4, query_ln=1), 4, 9),          # fp32 storage (CUDA-core query)
    (dict(dtype=0, conv_k=3, query_ln=1, share_query=0, rank=3, d_k=48), 3, 5),
    (dict(dtype=1, conv_k=4, query_ln=1, cores=2), 16, 1),   # with Multi-Core Scoring
]


@pytest.mark.parametrize("case", range(len(CASES)))
def test_query_extras_small_layers(case, gpu_lib):
    over, n_seq, L = CASES[case]
    cfg = workloads.small_config(ln_eps=1e-5, **over)
    _run_seq(cfg, n_seq, L, gpu_lib)


def test_fresh_sequences_without_state(gpu_lib):
    """No state in: the convolution reads zeros before each sequence."""
    cfg = workloads.small_config(dtype=1, conv_k=4, query_ln=1, ln_eps=1e-5)
    _run_seq(cfg, 4, 6, gpu_lib, with_state=False)


@pytest.mark.parametrize("n_seq,L", [(64, 1), (4, 32)])
def test_decode_1m_with_query_extras(n_seq, L, gpu_lib):
    """The decode-shaped layer with a 4-tap convolution and the query
    LayerNorm: 64 sequences one token each (the small query) and 4 x 32
    tokens (the tensor-core query with three-term operands)."""
    cfg = workloads.layer_config("decode_1m", conv_k=4, query_ln=1, ln_eps=1e-5)
    _run_seq(cfg, n_seq, L, gpu_lib)


def test_decode_steps_chain_states(gpu_lib):
    """Three decode steps (one token per sequence, each step's state the
    next one's input) give the outputs of one call on the 3-token
    sequences."""
    cfg = workloads.small_config(dtype=1, conv_k=4, query_ln=1, ln_eps=1e-5)
    S, T = 6, 3
    w = workloads.make_weights(cfg, device="cuda")
    x = workloads.make_tokens(cfg, S * T, device="cuda").view(S, T, -1)
    s0 = workloads.make_conv_state(cfg, S, device="cuda")
    layer = binding.UltraMemLayer(cfg, w, S * T)
    whole = layer.forward_seq(x.reshape(S * T, -1), S, s0).float().view(S, T, -1)
    state = s0
    for step in range(T):
        nxt = torch.empty_like(s0)
        o = layer.forward_seq(x[:, step].contiguous(), S, state, nxt).float()
        torch.cuda.synchronize()
        err = (o - whole[:, step]).abs().amax(1) / whole[:, step].abs().amax(1)
        assert err.max().item() <= 1e-2, f"step {step}: {err.max().item()}"
        state = nxt
    assert layer.check() == 0


def test_launch_counts_with_query_extras(gpu_lib):
    """The convolution and the LayerNorm are one kernel each."""
    cfg = workloads.small_config(dtype=1, conv_k=4, query_ln=1, ln_eps=1e-5)
    layer, *_ = _run_seq(cfg, 8, 1, gpu_lib)
    assert layer.last_launches() == 7


def test_overlapping_states_are_rejected(gpu_lib):
    cfg = workloads.small_config(dtype=1, conv_k=4)
    w = workloads.make_weights(cfg, device="cuda")
    layer = binding.UltraMemLayer(cfg, w, 8)
    x = workloads.make_tokens(cfg, 8, device="cuda")
    s = workloads.make_conv_state(cfg, 8, device="cuda")
    with pytest.raises(binding.UltraMemError) as e:
        layer.forward_seq(x, 8, s, s)
    assert e.value.status == binding.EINVAL


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_key_layernorm(dtype, gpu_lib):
    """ultramem_key_ln against the oracle's key LayerNorm: fp32 within 1e-5
    relative, bf16 within one rounding of the result (2^-8 relative)."""
    rng = np.random.default_rng(5)
    keys = torch.from_numpy(rng.standard_normal((3, 700, 128)) * 0.1).to(dtype).cuda()
    g = torch.from_numpy(1 + 0.1 * rng.standard_normal(128)).float().cuda()
    b = torch.from_numpy(0.1 * rng.standard_normal(128)).float().cuda()
    got = binding.key_ln(keys, g, b, eps=1e-5)
    inplace = keys.clone()
    binding.key_ln(inplace, g, b, eps=1e-5, out=inplace)
    torch.cuda.synchronize()
    ref = oracle.key_ln(workloads.stored_numpy(keys), 1 if dtype == torch.bfloat16 else 0,
                        g.cpu().numpy(), b.cpu().numpy(), eps=1e-5)
    tol = 2.0 ** -8 if dtype == torch.bfloat16 else 1e-5
    err = np.abs(got.float().cpu().numpy() - ref) / np.maximum(np.abs(ref), 1e-2)
    assert err.max() <= tol
    assert torch.equal(inplace, got)
