"""GPU parity: the CUDA library against the CPU oracle on the same seeded
inputs, through the C ABI (ctypes binding).  Indices bit-exact up to the
near-tie rule, weights and outputs within the stated tolerances."""
import numpy as np
import pytest
import torch

import oracle
from paper_2411_12364_gb300 import workloads
from tests import parity

pytestmark = pytest.mark.gpu


def _run(cfg, B, gpu_lib, tokens=None, max_tokens=None, batch_index=0, perm=None,
         pass_svd=True):
    from paper_2411_12364_gb300.binding import UltraMemLayer
    w = workloads.make_weights(cfg, device="cuda")
    if perm is not None:
        w["perm"] = perm
    x = workloads.make_tokens(cfg, B, batch_index, device="cuda")
    t = parity.numpy_inputs(cfg, w, x)
    if perm is not None:
        t["perm"] = perm.cpu().numpy().astype(np.int64)
    lw = dict(w)
    if pass_svd:
        lw["u"], lw["t"] = torch.from_numpy(t["u"]), torch.from_numpy(t["t"])
    layer = UltraMemLayer(cfg, lw, max_tokens or B)
    out, idx, wt = layer.forward(x, with_slots=True)
    torch.cuda.synchronize()
    assert layer.check() == 0
    tokens = np.arange(B) if tokens is None else np.asarray(tokens)
    o_out, o_idx, o_w = oracle.forward(cfg, t, B, tokens=tokens)
    res = parity.compare(cfg, t, tokens, out.float().cpu().numpy(), idx.cpu().numpy(),
                         wt.cpu().numpy(), o_out, o_idx, o_w)
    return layer, (w, x, t), (out, idx, wt), res


SMALL = [
    dict(dtype=0),
    dict(dtype=1),
    dict(dtype=0, expand_e=1, has_proj=0, d_out=64, n=40),
    dict(dtype=1, expand_e=9, n=11, d_out=72),
    dict(dtype=0, rank=1, d_k=24),
    dict(dtype=0, rank=3, d_k=48, heads=3),
    dict(dtype=1, share_query=0),
    dict(dtype=0, act=1),
    dict(dtype=0, topk=48, topm=1),          # k = K: no pruning
    dict(dtype=0, n=6, topk=5, topm=25),     # m = k*k
    dict(dtype=1, heads=4, topk=16, topm=40, d_v=128, d_out=40),
    dict(dtype=0, shuffle_seed=0),
    dict(dtype=1, rank=3, d_k=48),           # tensor path, odd rank (folded query)
    dict(dtype=1, rank=5, d_k=40, heads=3),  # tensor path, 8-wide rank chunks
    dict(dtype=0, cores=2),                  # Multi-Core Scoring (Eq. 16-17)
    dict(dtype=1, cores=2),
    dict(dtype=1, cores=4, rank=3, d_k=48),  # four 16-wide value slices
    dict(dtype=0, cores=2, expand_e=1, has_proj=0, d_out=64, n=40),
    dict(dtype=1, cores=8, d_v=128, d_out=40, heads=4, topk=16, topm=40),
    dict(dtype=1, cores=2, heads=4, topk=24, topm=160),   # H*m > 512: per-lane gather
    dict(dtype=1, rank=1, score_mode=1),                  # product keys (Eq. 2), raw
    dict(dtype=0, rank=1, score_mode=1, act=1),           # PKM with its softmax (Eq. 3)
    dict(dtype=1, rank=1, score_mode=1, share_query=0, topk=16, topm=16),
    dict(dtype=1, n=600, topk=128, topm=128),             # k = 128: four S_col columns a lane
]


@pytest.mark.parametrize("B", [1, 7, 37, 70])
@pytest.mark.parametrize("over", SMALL, ids=[str(i) for i in range(len(SMALL))])
def test_small_layers(over, B, gpu_lib):
    cfg = workloads.small_config(**over)
    _run(cfg, B, gpu_lib)


def _no_floor_ties(res):
    """The five workloads: every excused head is a near-tie relative to its
    own boundary scores, none only through the cancellation floor."""
    assert res[3].floor_ties == 0, f"{res[3].floor_ties} heads excused only by the floor"


def test_tiny_fp32_workload(gpu_lib):
    cfg = workloads.layer_config("tiny_fp32")
    _no_floor_ties(_run(cfg, 16, gpu_lib))


def test_decode_1m_workload(gpu_lib):
    cfg = workloads.layer_config("decode_1m")
    _no_floor_ties(_run(cfg, 64, gpu_lib))


@pytest.mark.parametrize("B", [64, 300])
def test_product_key_workload(B, gpu_lib):
    """The decode-shaped layer as a product-key memory (Eq. 2-3): rank 1,
    additive grid scores, PKM's softmax over the m slots."""
    cfg = workloads.layer_config("decode_1m", rank=1, score_mode=1, act=1)
    _run(cfg, B, gpu_lib)


@pytest.mark.parametrize("name,B", [("decode_1m", 64), ("mid_4m", 128)])
def test_multi_core_scoring_workloads(name, B, gpu_lib):
    """The paper's default h = 2 component cores (Sec. 3.2, Eq. 16-17) on the
    decode-shaped layers: top-m on the summed core, two weights per slot,
    each scaling one 128-wide half of the physical value row."""
    cfg = workloads.layer_config(name, cores=2)
    _run(cfg, B, gpu_lib)


@pytest.mark.parametrize("B", [1, 8, 32, 128])
def test_mid_4m_workload(B, gpu_lib):
    cfg = workloads.layer_config("mid_4m")
    _no_floor_ties(_run(cfg, B, gpu_lib))


@pytest.mark.parametrize("B", [1, 64, 256])
def test_large_20m_workload(B, gpu_lib):
    cfg = workloads.layer_config("large_20m")
    _no_floor_ties(_run(cfg, B, gpu_lib))


def test_prefill_16k_sampled(gpu_lib):
    """All 16384 tokens run on the GPU; a seeded sample of 384 (including the
    first and last tile's tokens) is checked against the oracle."""
    cfg = workloads.layer_config("prefill_16k")
    rng = np.random.default_rng(4)
    sample = np.unique(np.concatenate([np.arange(8), np.arange(16384 - 8, 16384),
                                       rng.choice(16384, 368, replace=False)]))
    _no_floor_ties(_run(cfg, 16384, gpu_lib, tokens=sample))


@pytest.mark.parametrize("cores", [0, 2])
def test_lookup_reduce_on_oracle_slots(cores, gpu_lib):
    """S7-S9 alone: the GPU pools the oracle's own (v, w) like the oracle
    (with MCS, h weights per slot, one per value slice)."""
    from paper_2411_12364_gb300.binding import UltraMemLayer
    cfg = workloads.layer_config("decode_1m", cores=cores)
    w = workloads.make_weights(cfg, device="cuda")
    x = workloads.make_tokens(cfg, 16, device="cuda")
    t = parity.numpy_inputs(cfg, w, x)
    layer = UltraMemLayer(cfg, dict(w, u=torch.from_numpy(t["u"]), t=torch.from_numpy(t["t"])), 16)
    o_out, o_idx, o_w = oracle.forward(cfg, t, 16)
    out = layer.lookup_reduce(torch.from_numpy(o_idx).cuda(),
                              torch.from_numpy(o_w.astype(np.float32)).cuda())
    ref = oracle.lookup_reduce(cfg, t, o_idx, o_w.astype(np.float32).astype(np.float64))
    err, _ = parity.output_errors(out.float().cpu().numpy(), ref)
    assert err.max() <= parity.out_tol(cfg), err.max()
    assert layer.check() == 0


def test_retrieve_and_host_forward_agree_with_forward(gpu_lib):
    cfg = workloads.small_config(dtype=1)
    layer, (w, x, t), (out, idx, wt), _ = _run(cfg, 33, gpu_lib)
    i2, w2 = layer.retrieve(x)
    assert torch.equal(i2, idx) and torch.equal(w2, wt)
    xh = x.cpu().pin_memory()
    oh = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    layer.forward_host(xh, oh)              # pinned: copy kernels over the host link
    assert torch.equal(oh, out.cpu())
    xp = x.cpu().clone()
    op = torch.empty(out.shape, dtype=out.dtype)
    layer.forward_host(xp, op)              # pageable: the copy engines
    assert torch.equal(op, out.cpu())


@pytest.mark.parametrize("B", [64, 65])
def test_host_forward_at_decode_shape(B, gpu_lib):
    """The host-buffer call on decode_1m, on both sides of the CUDA-core
    query's batch limit: a copy kernel reads the pinned tokens over the host
    link and the projection writes the pinned output; both calls (captured,
    then replayed) equal the device forward bit for bit."""
    from paper_2411_12364_gb300.binding import UltraMemLayer
    cfg = workloads.layer_config("decode_1m")
    w = workloads.make_weights(cfg, device="cuda")
    layer = UltraMemLayer(cfg, w, 65)
    x = workloads.make_tokens(cfg, B, 3, device="cuda")
    out = layer.forward(x)
    xh = x.cpu().pin_memory()
    oh = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    for _ in range(2):   # captured, then replayed
        oh.zero_()
        layer.forward_host(xh, oh)
        assert layer.check() == 0
        assert torch.equal(oh, out.cpu())
    layer.close()


def test_forward_is_deterministic(gpu_lib):
    cfg = workloads.small_config(dtype=1, heads=3)
    layer, (w, x, t), (out, idx, wt), _ = _run(cfg, 70, gpu_lib)
    for _ in range(3):
        o2, i2, w2 = layer.forward(x, with_slots=True)
        assert torch.equal(o2, out) and torch.equal(i2, idx) and torch.equal(w2, wt)


def test_library_svd_and_explicit_perm(gpu_lib):
    """(u, t) computed by the library at create, and an explicit shuffle
    table, both give the oracle's result."""
    cfg = workloads.small_config(dtype=0, n=10)
    M = cfg["expand_e"] * cfg["n"] ** 2
    perm = torch.from_numpy(np.random.default_rng(3).permutation(M).astype(np.int32)).cuda()
    _run(cfg, 20, gpu_lib, perm=perm, pass_svd=False)


def test_workspace_reuse_across_batch_sizes(gpu_lib):
    """One handle sized for 70 tokens serves smaller batches too: the same
    slots, and the same outputs up to the query's summation order (70 tokens
    take the tensor-core query, 64 and fewer the CUDA-core one)."""
    cfg = workloads.small_config(dtype=1)
    layer, (w, x, t), (out, idx, wt), _ = _run(cfg, 70, gpu_lib)
    for B in (1, 5, 32, 64):
        o2, i2, w2 = layer.forward(x[:B].contiguous(), with_slots=True)
        assert torch.equal(i2, idx[:B])
        torch.testing.assert_close(w2, wt[:B], rtol=1e-5, atol=1e-6)
        ref = out[:B].float()
        err = (o2.float() - ref).abs().amax(1) / ref.abs().amax(1)
        assert err.max().item() <= 2 ** -7   # one bf16 rounding of the output


def test_bad_address_is_reported_not_read(gpu_lib):
    """An out-of-range virtual address given to lookup_reduce is skipped by
    the kernel's own bounds check and reported by ultramem_check."""
    from paper_2411_12364_gb300 import binding
    cfg = workloads.small_config(dtype=1)
    layer, (w, x, t), (out, idx, wt), _ = _run(cfg, 4, gpu_lib)
    bad = idx.clone()
    bad[1, 0, 0] = cfg["expand_e"] * cfg["n"] ** 2 + 5
    bad[2, 1, 3] = -1
    layer.lookup_reduce(bad, wt)
    assert layer.check() == binding.EDEVICE
    assert layer.check() == 0   # the error word is cleared by the read


def test_batch_limits(gpu_lib):
    from paper_2411_12364_gb300 import binding
    cfg = workloads.small_config(dtype=1)
    layer, (w, x, t), _, _ = _run(cfg, 8, gpu_lib)
    lib = binding.load()
    st = lib.ultramem_forward(layer._h, x.data_ptr(), 0, None, None, None, None)
    assert st == binding.OK
    big = torch.zeros((9, cfg["d_in"]), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.UltraMemError):
        layer.forward(big)


MAXIMA = [
    # K = sqrt(16) * 5120 = 20480 keys per axis, k = 128, m = 1024 = the
    # selection's limits (the final list overflows into the radix select),
    # r = 8, E = 16 virtual blocks, 26 M physical rows
    dict(dtype=1, d_in=64, d_k=64, heads=2, rank=8, n=5120, expand_e=16, d_v=16, d_out=32,
         topk=128, topm=1024),
    # the same limits with fp32 storage (CUDA-core path) and eight cores
    dict(dtype=0, d_in=64, d_k=64, heads=1, rank=8, n=5120, expand_e=16, d_v=64, d_out=32,
         topk=128, topm=1024, cores=8),
]


@pytest.mark.parametrize("case", range(len(MAXIMA)))
def test_maximum_sizes(case, gpu_lib):
    """The ABI's upper limits at once, on 6 tokens against the oracle."""
    cfg = workloads.small_config(**MAXIMA[case])
    assert workloads.keys_per_axis(cfg) == 20480
    _run(cfg, 6, gpu_lib)


def _tied_weights(cfg, rows_tied):
    """Weights whose first `rows_tied` keys of each axis are one and the same
    row, so that their rank-1 and exact scores tie exactly."""
    w = workloads.make_weights(cfg, device="cuda")
    for name in ("k_row", "k_col"):
        k = w[name].clone()
        k[:, :rows_tied, :] = k[:, :1, :]
        w[name] = k
    return w


def _run_weights(cfg, w, B, gpu_lib):
    from paper_2411_12364_gb300.binding import UltraMemLayer
    x = workloads.make_tokens(cfg, B, 0, device="cuda")
    t = parity.numpy_inputs(cfg, w, x)
    layer = UltraMemLayer(cfg, dict(w, u=torch.from_numpy(t["u"]), t=torch.from_numpy(t["t"])), B)
    out, idx, wt = layer.forward(x, with_slots=True)
    torch.cuda.synchronize()
    assert layer.check() == 0
    o_out, o_idx, o_w = oracle.forward(cfg, t, B)
    parity.compare(cfg, t, np.arange(B), out.float().cpu().numpy(), idx.cpu().numpy(),
                   wt.cpu().numpy(), o_out, o_idx, o_w)
    return idx


@pytest.mark.parametrize("dtype", [0, 1])
def test_all_keys_tied(dtype, gpu_lib):
    """Every key of both axes is the same row: all K = 1200 rank-1 scores tie
    (more candidates than a list holds, so the exact radix select runs), and
    all k*k = 1600 Tucker scores tie too.  Ties go to the smaller index: the
    slots are the first m pairs of rows 0..k-1 x columns 0..k-1."""
    cfg = workloads.small_config(dtype=dtype, n=600, topk=40, topm=64)
    K = workloads.keys_per_axis(cfg)
    w = _tied_weights(cfg, K)
    idx = _run_weights(cfg, w, 9, gpu_lib).cpu().numpy()
    k, m = cfg["topk"], cfg["topm"]
    pairs = np.array([i * K + j for i in range(k) for j in range(k)])[:m]
    assert (np.sort(idx, axis=-1) == np.sort(pairs)).all()


@pytest.mark.parametrize("dtype", [0, 1])
def test_many_keys_tied(dtype, gpu_lib):
    """500 of the 1200 keys of each axis tie: for tokens whose tied score is
    at the top, the candidate list is long but fits (it is tightened before
    ranking); the others cut through or below the tie."""
    cfg = workloads.small_config(dtype=dtype, n=600, topk=40, topm=64)
    _run_weights(cfg, _tied_weights(cfg, 500), 37, gpu_lib)


def test_last_launches_counts_each_call(gpu_lib):
    """The library's kernel count per call: the tensor path runs one query
    projection per query, score and select (retrieve), then gather and the
    projection (split-K reduced inside its clusters); the CUDA-core path adds
    a reduce after each split-K contraction's partials; lookup_reduce runs
    slots, gather, projection and reduce."""
    cfg = workloads.small_config(dtype=1)
    layer, (w, x, t), (out, idx, wt), _ = _run(cfg, 16, gpu_lib)
    assert layer.last_launches() == 5
    layer.retrieve(x)
    assert layer.last_launches() == 3
    layer.lookup_reduce(idx, wt)
    assert layer.last_launches() == 4
    cfg2 = workloads.small_config(dtype=1, share_query=0)
    layer2, *_ = _run(cfg2, 16, gpu_lib)
    assert layer2.last_launches() == 6
    cfg32 = workloads.small_config(dtype=0)
    layer32, *_ = _run(cfg32, 16, gpu_lib)
    assert layer32.last_launches() == 6


LONG_GRID = [
    dict(dtype=1, topk=48, topm=1),                          # k = K: every key a candidate
    dict(dtype=0, n=6, topk=5, topm=25),                     # m = k*k
    dict(dtype=1, heads=4, topk=16, topm=40, d_v=128, d_out=40),
    dict(dtype=1, topk=24, topm=64),
    dict(dtype=1, topk=24, topm=64, cores=2),                # MCS
    dict(dtype=1, heads=4, topk=24, topm=160, cores=2),      # MCS, per-lane gather
    dict(dtype=1, topk=32, topm=100),
    dict(dtype=0, n=600, topk=100, topm=128),                # axis lists over 128: counted
    dict(dtype=1, n=600, topk=96, topm=64),                  # k = 96: three S_col columns a lane
    dict(dtype=1, n=2400, topk=64, topm=64),                 # K = 4800 > 4096: keys streamed from L2
    dict(dtype=1, n=2049, topk=64, topm=64),                 # K = 4098, not a multiple of 4: staged
]


@pytest.mark.parametrize("over", LONG_GRID, ids=[str(i) for i in range(len(LONG_GRID))])
def test_long_grid_selection(over, gpu_lib):
    """Batches whose selection grid exceeds three CTAs per SM (here 300 tokens
    x H heads) take the long-grid selection, which ranks candidates by
    sorted warp runs instead of counting (longer lists are counted); its
    lists here fill several runs."""
    cfg = workloads.small_config(**over)
    _run(cfg, 300, gpu_lib)


@pytest.mark.parametrize("rows_tied", [1200, 500])
def test_tied_keys_long_grid(rows_tied, gpu_lib):
    """The tie cases above on the long-grid selection (240 tokens x 2 heads)."""
    cfg = workloads.small_config(dtype=1, n=600, topk=40, topm=64)
    _run_weights(cfg, _tied_weights(cfg, rows_tied), 240, gpu_lib)
