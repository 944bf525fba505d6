"""Pins of the CPU oracle against facts fixed outside it: hand-worked
examples, the brute-force definition of Eq. 5, the exactness of the
two-phase search for a rank-1 core (Eq. 6), the PKM reduction at r = 1
(Eq. 2-3), the explicit virtual table (Eq. 13-15), numpy's SVD (Eq. 7),
the published SplitMix64 outputs, plain invariants of top-m and softmax,
and Eq. 16-17 of Multi-Core Scoring (per-core grids by brute force, the
explicit sliced table, the h = 1 and equal-core reductions)."""
import json
import os

import numpy as np
import pytest

import oracle
from paper_2411_12364_gb300 import workloads
from tests import util

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    d = json.load(open(os.path.join(GOLDEN, name)))
    cfg = d["config"]
    t = {}
    for k, v in d["tensors"].items():
        a = np.array(v)
        t[k] = a.astype(np.int64) if k == "perm" else a.astype(np.float32)
    return cfg, t, d["expected"]


@pytest.mark.parametrize("name", ["hand_tucker_ive.json", "hand_pruning_rows.json",
                                  "hand_mcs.json", "hand_conv_ln.json"])
def test_hand_worked_examples(name):
    cfg, t, exp = _golden(name)
    out, idx, w = oracle.forward(cfg, t, B=len(t["x"]))
    np.testing.assert_array_equal(idx, np.array(exp["idx"]))
    np.testing.assert_array_equal(w, np.array(exp["w"], dtype=np.float64))
    np.testing.assert_array_equal(out, np.array(exp["out"], dtype=np.float64))


def _f32_cfg(**kw):
    base = dict(dtype=0, n=6, expand_e=4, d_k=8, d_in=12, heads=2, d_v=8, d_out=10,
                topk=5, topm=6, seed=3, shuffle_seed=77)
    base.update(kw)
    return workloads.small_config(**base)


def test_brute_force_equals_tdqkr_without_pruning():
    """k = K keeps every key (Eq. 8-9 are vacuous), so Eq. 10's top-m is the
    top-m of Eq. 5 over the whole grid."""
    cfg = _f32_cfg()
    K = workloads.keys_per_axis(cfg)
    cfg["topk"] = K
    t = util.numpy_layer(cfg, B=3)
    u, tt = util.numpy_rank1(t["core"])
    t["u"], t["t"] = u.astype(np.float32), tt.astype(np.float32)
    out, idx, w = oracle.forward(cfg, t, B=3)
    for b in range(3):
        for h in range(cfg["heads"]):
            v, g = util.brute_force_grid(cfg, t, b, h, t["core"][h])
            np.testing.assert_array_equal(idx[b, h], v)
            np.testing.assert_allclose(w[b, h], g, rtol=1e-12, atol=1e-12)


def _positive_layer(cfg, B, rank1_core):
    """Keys, queries and singular vectors with positive entries: every
    rank-1 score is positive (Eq. 6)."""
    t = util.numpy_layer(cfg, B=B)
    for k in ("x", "w_q", "k_row", "k_col"):
        t[k] = np.abs(t[k])
    rng = np.random.default_rng(5)
    H, r = cfg["heads"], cfg["rank"]
    core = np.zeros((H, r, r), np.float32)
    for h in range(H):
        if rank1_core:
            uu = rng.uniform(0.2, 1.0, r)
            tt = rng.uniform(0.2, 1.0, r)
            core[h] = 1.7 * np.outer(uu, tt)
        else:
            core[h] = rng.uniform(0.5, 1.5, (r, r))
    t["core"] = core
    return t


@pytest.mark.parametrize("rank", [1, 2, 4])
def test_rank1_core_two_phase_is_exact(rank):
    """Invariant of the method: with C = sigma u t^T and positive scores, the
    grid score is sigma*a_i*b_j, monotone in both factors, so the two-phase
    top-m (Eq. 8-10 with k = m) equals brute force over all K*K slots."""
    cfg = _f32_cfg(rank=rank, d_k=8, topk=6, topm=6, n=8)
    t = _positive_layer(cfg, B=4, rank1_core=True)
    out, idx, w = oracle.forward(cfg, t, B=4)  # (u, t) from the oracle's own SVD
    for b in range(4):
        for h in range(cfg["heads"]):
            v, g = util.brute_force_grid(cfg, t, b, h, t["core"][h])
            np.testing.assert_array_equal(idx[b, h], v)
            np.testing.assert_allclose(w[b, h], g, rtol=1e-9)


def test_rank_one_reduces_to_product_key_memory():
    """Invariant of the method: at r = 1 the core is a positive scalar c and
    g(i,j) = c*S_row[i]*S_col[j]; with positive scores log g = log c +
    log S_row[i] + log S_col[j], the additive product-key score of PKM
    (Eq. 2), whose two-phase top-m is exact.  PKM's retrieval is computed
    here independently in numpy and must select the same slots."""
    cfg = _f32_cfg(rank=1, d_k=6, topk=7, topm=7, n=9, heads=2)
    t = _positive_layer(cfg, B=3, rank1_core=True)
    K = workloads.keys_per_axis(cfg)
    out, idx, w = oracle.forward(cfg, t, B=3)
    for b in range(3):
        for h in range(cfg["heads"]):
            s_row, s_col = util.numpy_scores(cfg, t, b, h)
            lr, lc = np.log(s_row[0]), np.log(s_col[0])
            m = cfg["topm"]
            I = np.argsort(-lr, kind="stable")[:m]  # Eq. 2, row phase
            J = np.argsort(-lc, kind="stable")[:m]  # Eq. 2, column phase
            cand = (lr[I][:, None] + lc[J][None, :]).ravel()
            v = (I[:, None] * K + J[None, :]).ravel()
            order = np.lexsort((v, -cand))[:m]  # Eq. 3's top-m on the grid
            np.testing.assert_array_equal(np.sort(idx[b, h]), np.sort(v[order]))
            np.testing.assert_array_equal(idx[b, h], v[order])


def test_general_core_selection_invariants():
    """For a general core: the per-axis survivors are the top-k of u^T S_row
    and t^T S_col (Eq. 8-9), the selected slots are inside I x J, and every
    selected fp32 score is >= every unselected candidate's (Eq. 10)."""
    cfg = _f32_cfg(n=10, topk=6, topm=9)
    t = util.numpy_layer(cfg, B=4)
    u, tt = util.numpy_rank1(t["core"])
    t["u"], t["t"] = u.astype(np.float32), tt.astype(np.float32)
    K = workloads.keys_per_axis(cfg)
    out, idx, w = oracle.forward(cfg, t, B=4)
    for b in range(4):
        for h in range(cfg["heads"]):
            s_row, s_col = util.numpy_scores(cfg, t, b, h)
            a = t["u"][h].astype(np.float64) @ s_row
            bb = t["t"][h].astype(np.float64) @ s_col
            I = util.topm_desc(a, np.arange(K), cfg["topk"])
            J = util.topm_desc(bb, np.arange(K), cfg["topk"])
            G = s_row.T @ t["core"][h].astype(np.float64) @ s_col
            cand_v = (I[:, None] * K + J[None, :]).ravel()
            cand_g = G[I][:, J].ravel()
            sel = set(idx[b, h].tolist())
            assert sel <= set(cand_v.tolist())
            sel_g = np.array([G[v // K, v % K] for v in idx[b, h]])
            rest = np.array([g for v, g in zip(cand_v, cand_g) if v not in sel])
            assert sel_g.astype(np.float32).min() >= rest.astype(np.float32).max()
            np.testing.assert_allclose(w[b, h], sel_g, rtol=1e-12, atol=1e-14)
            assert np.all(np.diff(w[b, h].astype(np.float32)) <= 0)


def test_explicit_virtual_table_equals_implicit():
    """Invariant of the method: materialising V~_p = V W_p (Eq. 13), scattering
    the weights at the shuffled addresses (Eq. 14) and taking V~^T s^ gives
    the implicit sum_p W_p^T (V^T s^_p) of Eq. 15."""
    cfg = _f32_cfg(n=6, expand_e=4, d_v=8, d_out=11, topk=5, topm=7, heads=3)
    t = util.numpy_layer(cfg, B=5)
    M = cfg["expand_e"] * cfg["n"] ** 2
    t["perm"] = np.random.default_rng(9).permutation(M).astype(np.int64)
    out, idx, w = oracle.forward(cfg, t, B=5)
    ref = util.explicit_ive(cfg, t, idx, w, t["perm"])
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-13)
    # the seeded shuffle, through the oracle's own pi(v), gives the same
    t2 = dict(t)
    t2.pop("perm")
    out2, idx2, w2 = oracle.forward(cfg, t2, B=5)
    perm = oracle.shuffle(cfg, np.arange(M))
    np.testing.assert_allclose(out2, util.explicit_ive(cfg, t2, idx2, w2, perm),
                               rtol=1e-11, atol=1e-13)


def test_no_expansion_is_plain_weighted_pooling():
    """E = 1 without projector: o = sum of w * V[pi(v)] (Eq. 1/3 pooling
    without the softmax, Trick 1)."""
    cfg = _f32_cfg(expand_e=1, has_proj=0, d_out=8, d_v=8, n=12)
    t = util.numpy_layer(cfg, B=3)
    out, idx, w = oracle.forward(cfg, t, B=3)
    V = util.widen(t["values"])
    perm = oracle.shuffle(cfg, np.arange(cfg["n"] ** 2))
    for b in range(3):
        ref = (w[b].ravel()[:, None] * V[perm[idx[b].ravel()]]).sum(0)
        np.testing.assert_allclose(out[b], ref, rtol=1e-12, atol=1e-14)


def test_softmax_weights_sum_to_one():
    """Invariant of the method: with PKM's softmax (Eq. 3) the m weights of a
    head are positive, sum to 1 and keep the score order; without it
    (Trick 1) they are the raw scores."""
    cfg = _f32_cfg(act=1, topm=7)
    t = util.numpy_layer(cfg, B=4)
    out_s, idx_s, w_s = oracle.forward(cfg, t, B=4)
    cfg0 = dict(cfg, act=0)
    out_n, idx_n, w_n = oracle.forward(cfg0, t, B=4)
    np.testing.assert_array_equal(idx_s, idx_n)
    np.testing.assert_allclose(w_s.sum(-1), 1.0, rtol=1e-12)
    assert np.all(w_s > 0)
    ref = np.exp(w_n - w_n.max(-1, keepdims=True))
    ref /= ref.sum(-1, keepdims=True)
    np.testing.assert_allclose(w_s, ref, rtol=1e-12)


def test_heads_are_summed():
    """Multi-head retrieval reads one shared table (Sec. 3.1): the H-head
    output is the sum of H one-head layers built from each head's weights."""
    cfg = _f32_cfg(heads=3)
    t = util.numpy_layer(cfg, B=3)
    out, idx, w = oracle.forward(cfg, t, B=3)
    dk = cfg["d_k"]
    total = np.zeros_like(out)
    for h in range(3):
        c1 = dict(cfg, heads=1)
        t1 = dict(t)
        t1["w_q"] = t["w_q"][h * dk:(h + 1) * dk]
        t1["k_row"] = t["k_row"][h:h + 1]
        t1["k_col"] = t["k_col"][h:h + 1]
        t1["core"] = t["core"][h:h + 1]
        o1, i1, w1 = oracle.forward(c1, t1, B=3)
        np.testing.assert_array_equal(i1[:, 0], idx[:, h])
        total += o1
    np.testing.assert_allclose(out, total, rtol=1e-11, atol=1e-14)


def test_separate_column_query():
    """Without Trick 5 the column keys see their own query W_q_col x."""
    cfg = _f32_cfg(share_query=0, topk=30)
    K = workloads.keys_per_axis(cfg)
    cfg["topk"] = K
    t = util.numpy_layer(cfg, B=2)
    assert t["w_q_col"] is not None
    u, tt = util.numpy_rank1(t["core"])
    t["u"], t["t"] = u.astype(np.float32), tt.astype(np.float32)
    out, idx, w = oracle.forward(cfg, t, B=2)
    for b in range(2):
        for h in range(cfg["heads"]):
            v, g = util.brute_force_grid(cfg, t, b, h, t["core"][h])
            np.testing.assert_array_equal(idx[b, h], v)


def test_scores_match_reshaped_keys():
    """Eq. 4 with keys reshaped to r x n x (D_k/r): rank chunk alpha is the
    alpha-th slice of D_k/r columns of each key and of the query."""
    cfg = _f32_cfg(rank=4, d_k=16, share_query=0)
    t = util.numpy_layer(cfg, B=2)
    for b in range(2):
        for h in range(cfg["heads"]):
            sr, sc = oracle.row_col_scores(cfg, t, b, h)
            nr, nc = util.numpy_scores(cfg, t, b, h)
            np.testing.assert_allclose(sr, nr, rtol=1e-12, atol=1e-14)
            np.testing.assert_allclose(sc, nc, rtol=1e-12, atol=1e-14)


def test_planted_slot_is_found():
    """A key pair aligned with the query dominates the grid: the top slot
    must be v = i* K + j* (Sec. 3.1 addressing) with score ~ the planted one."""
    cfg = _f32_cfg(rank=1, d_k=8, d_in=8, heads=1, n=10, topk=4, topm=4, expand_e=1,
                   has_proj=0, d_out=8, shuffle_seed=0)
    t = util.numpy_layer(cfg, B=1)
    K = workloads.keys_per_axis(cfg)
    t["w_q"] = np.eye(8, dtype=np.float32)
    x = np.zeros((1, 8), np.float32)
    x[0, 2] = 1.0
    t["x"] = x
    t["core"] = np.ones((1, 1, 1), np.float32)
    kr = np.random.default_rng(1).normal(0, 0.01, (1, K, 8)).astype(np.float32)
    kc = np.random.default_rng(2).normal(0, 0.01, (1, K, 8)).astype(np.float32)
    kr[0, 7, 2], kc[0, 3, 2] = 5.0, 4.0
    t["k_row"], t["k_col"] = kr, kc
    out, idx, w = oracle.forward(cfg, t, B=1)
    assert idx[0, 0, 0] == 7 * K + 3
    assert abs(w[0, 0, 0] - 20.0) < 0.5
    V = util.widen(t["values"])
    assert np.abs(out[0] - (w[0, 0][:, None] * V[idx[0, 0]]).sum(0)).max() < 1e-12


def test_ties_go_to_the_smaller_index():
    """All-equal scores: the per-axis survivors are keys 0..k-1 and the m
    selected slots are the m smallest v = i*K + j among them."""
    cfg = _f32_cfg(rank=2, heads=1, n=8, topk=3, topm=5)
    t = util.numpy_layer(cfg, B=1)
    t["x"] = np.zeros_like(t["x"])
    K = workloads.keys_per_axis(cfg)
    out, idx, w = oracle.forward(cfg, t, B=1)
    cand = sorted(i * K + j for i in range(3) for j in range(3))
    np.testing.assert_array_equal(idx[0, 0], cand[:5])
    assert np.all(w == 0) and np.all(out == 0)


def test_bf16_storage_widens_exactly():
    """bf16 values are the top halves of fp32 words: the layer on bf16
    storage equals the layer on the same values stored as fp32."""
    cfg = _f32_cfg(dtype=1)
    t = util.numpy_layer(cfg, B=3)
    out_b, idx_b, w_b = oracle.forward(cfg, t, B=3)
    t32 = {k: (util.widen(v).astype(np.float32) if (v is not None and v.dtype == np.uint16)
               else v) for k, v in t.items()}
    out_f, idx_f, w_f = oracle.forward(dict(cfg, dtype=0), t32, B=3)
    np.testing.assert_array_equal(idx_b, idx_f)
    np.testing.assert_array_equal(out_b, out_f)


def test_token_subset_and_lookup_reduce_agree():
    cfg = _f32_cfg()
    t = util.numpy_layer(cfg, B=6)
    out, idx, w = oracle.forward(cfg, t, B=6)
    sub = np.array([4, 1, 5])
    o2, i2, w2 = oracle.forward(cfg, t, B=6, tokens=sub)
    np.testing.assert_array_equal(i2, idx[sub])
    np.testing.assert_array_equal(o2, out[sub])
    o3 = oracle.lookup_reduce(cfg, t, idx, w)
    np.testing.assert_array_equal(o3, out)


@pytest.mark.parametrize("r", [1, 2, 3, 4, 8])
def test_rank1_against_numpy_svd(r):
    """Eq. 7: (u, t, sigma) is the leading singular triplet; checked against
    numpy's SVD, the defining relations and, for r = 2, the closed form
    sigma_1^2 = (|C|_F^2 + sqrt(|C|_F^4 - 4 det(C)^2)) / 2."""
    rng = np.random.default_rng(100 + r)
    for _ in range(20):
        C = rng.normal(size=(r, r))
        u, t, s = oracle.rank1(C)
        U, S, Vt = np.linalg.svd(C)
        assert abs(s - S[0]) <= 1e-12 * S[0]
        np.testing.assert_allclose(C @ t, s * u, atol=1e-11)
        np.testing.assert_allclose(C.T @ u, s * t, atol=1e-11)
        assert abs(np.linalg.norm(u) - 1) < 1e-12 and abs(np.linalg.norm(t) - 1) < 1e-12
        assert u.sum() > 0
        if S.size > 1 and S[0] - S[1] > 1e-6:
            sgn = np.sign(U[:, 0] @ u)
            np.testing.assert_allclose(u, sgn * U[:, 0], atol=1e-9)
            np.testing.assert_allclose(t, sgn * Vt[0], atol=1e-9)
        if r == 2:
            f2 = (C ** 2).sum()
            closed = np.sqrt((f2 + np.sqrt(f2 ** 2 - 4 * np.linalg.det(C) ** 2)) / 2)
            assert abs(s - closed) < 1e-10 * closed


def test_rank1_rejects_zero_core():
    with pytest.raises(ValueError):
        oracle.rank1(np.zeros((2, 2)))


def test_splitmix64_published_outputs():
    """Outputs 1-5 of SplitMix64 seeded with 1234567 as published with the
    generator (each output advances the state by the golden gamma)."""
    gamma = 0x9E3779B97F4A7C15
    want = [6457827717110365317, 3203168211198807973, 9817491932198370423,
            4593380528125082431, 16408922859458223821]
    s = 1234567
    for w in want:
        assert oracle.splitmix64(s) == w
        s = (s + gamma) % (1 << 64)


@pytest.mark.parametrize("M", [2, 36, 97, 1000, 4 * 1024 * 1024])
def test_shuffle_parameters_from_published_outputs(M):
    """pi's multiplier and offset come from the first two SplitMix64 outputs
    of the seed; for seed 1234567 those are published, so (a, c) follow by
    integer arithmetic alone."""
    import math
    o1, o2 = 6457827717110365317, 3203168211198807973
    a = 1 + o1 % (M - 1)
    while math.gcd(a, M) != 1:
        a = a + 1 if a + 1 < M else 1
    assert oracle.shuffle_params(1234567, M) == (a, o2 % M)


@pytest.mark.parametrize("seed", [0, 1, 77, 2**40 + 3])
@pytest.mark.parametrize("M", [1, 2, 36, 64, 97, 1000])
def test_shuffle_is_a_bijection(seed, M):
    """Eq. 14's shuffle must permute the virtual addresses; seed 0 is the
    identity."""
    cfg = dict(workloads.small_config(), n=1, expand_e=1, shuffle_seed=seed)
    a, c = oracle.shuffle_params(seed, M)
    import math
    assert math.gcd(a, M) == 1
    v = np.arange(M)
    pv = (a * v + c) % M
    assert np.array_equal(np.sort(pv), v)
    if seed == 0:
        assert (a, c) == (1, 0)
    # through uo_shuffle on a grid with E*N = M where M is a square
    if int(round(M ** 0.5)) ** 2 == M:
        cfg = dict(cfg, n=int(round(M ** 0.5)))
        got = oracle.shuffle(cfg, v)
        assert np.array_equal(np.sort(got), v)
        assert np.array_equal(got, pv)


def test_shuffle_honours_explicit_permutation():
    cfg = dict(workloads.small_config(), n=3, expand_e=4)
    perm = np.random.default_rng(0).permutation(36)
    got = oracle.shuffle(cfg, np.arange(36), perm=perm)
    assert np.array_equal(got, perm)


def test_invalid_configs_are_rejected():
    base = _f32_cfg()
    t = util.numpy_layer(base, B=1)
    bad = [dict(rank=3), dict(expand_e=3), dict(topk=10 ** 6), dict(topm=26),
           dict(has_proj=0), dict(act=5), dict(cores=3), dict(cores=2, act=1),
           dict(cores=9), dict(cores=-1), dict(conv_k=-1), dict(conv_k=65),
           dict(conv_k=2), dict(query_ln=2), dict(query_ln=1)]
    for kw in bad:
        with pytest.raises(ValueError):
            oracle.forward(dict(base, **kw), t, B=1)


# ---- Multi-Core Scoring (Sec. 3.2, Eq. 16-17) -------------------------------

def _mcs_layer(cfg, B, seed=21):
    """A layer whose h component cores are multiples of 1/8, so that their
    fp32 sum is exact and a one-core layer can be given the same aggregate."""
    t = util.numpy_layer(cfg, B=B)
    H, h, r = cfg["heads"], cfg["cores"], cfg["rank"]
    rng = np.random.default_rng(seed)
    t["core"] = (rng.integers(-16, 17, (H, h, r, r)) / 8.0).astype(np.float32)
    return t


def test_mcs_selection_uses_the_aggregate_core():
    """Eq. 16: top-m runs on S_row^T (sum_i C^(i)) S_col, so the addresses
    equal those of one core C = sum_i C^(i) (with u, t from its SVD), and the
    h per-core weights of a slot sum to that slot's aggregate score."""
    cfg = _f32_cfg(cores=3, rank=3, d_k=12, d_v=9, d_out=10, topk=6, topm=7)
    t = _mcs_layer(cfg, B=4)
    out, idx, w = oracle.forward(cfg, t, B=4)
    assert w.shape == (4, cfg["heads"], cfg["topm"], 3)
    one = dict(t)
    one["core"] = t["core"].sum(1)
    cfg1 = dict(cfg, cores=0)
    _, idx1, w1 = oracle.forward(cfg1, one, B=4)
    np.testing.assert_array_equal(idx, idx1)
    np.testing.assert_allclose(w.sum(-1), w1, rtol=1e-12, atol=1e-13)


def test_mcs_weights_are_the_per_core_grids():
    """Eq. 16-17 by brute force: with k = K (no pruning) the addresses are
    the top-m of the whole aggregate grid, and weight i of each is the
    individual map S_row^T C^(i) S_col (numpy reshapes, numpy SVD) there."""
    cfg = _f32_cfg(cores=2, d_v=8)
    K = workloads.keys_per_axis(cfg)
    cfg["topk"] = K
    t = _mcs_layer(cfg, B=3)
    out, idx, w = oracle.forward(cfg, t, B=3)
    for b in range(3):
        for h in range(cfg["heads"]):
            agg = t["core"][h].astype(np.float64).sum(0)
            v, g = util.brute_force_grid(cfg, t, b, h, agg)
            np.testing.assert_array_equal(idx[b, h], v)
            s_row, s_col = util.numpy_scores(cfg, t, b, h)
            for i in range(2):
                Gi = s_row.T @ t["core"][h, i].astype(np.float64) @ s_col
                np.testing.assert_allclose(w[b, h, :, i], Gi.ravel()[v], rtol=1e-11,
                                           atol=1e-12)


def test_mcs_explicit_sliced_table():
    """Eq. 17 with IVE (Eq. 15 on the split physical table): o is the sum
    over slices i of the explicit virtual-table output of a table whose
    columns outside slice i are zero, weighted by the i-th scores."""
    cfg = _f32_cfg(cores=4, d_v=8, d_out=11, heads=3, topm=7, expand_e=4)
    t = _mcs_layer(cfg, B=5)
    M = cfg["expand_e"] * cfg["n"] ** 2
    t["perm"] = np.random.default_rng(9).permutation(M).astype(np.int64)
    out, idx, w = oracle.forward(cfg, t, B=5)
    ref = np.zeros_like(out)
    sl = cfg["d_v"] // 4
    for i in range(4):
        ti = dict(t)
        V = util.widen(t["values"]).copy()
        V[:, :i * sl] = 0
        V[:, (i + 1) * sl:] = 0
        ti["values"] = V.astype(np.float32)
        ref += util.explicit_ive(cfg, ti, idx, w[..., i], t["perm"])
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-13)
    # lookup_reduce pools the same (address, weights) pairs the same way
    np.testing.assert_allclose(oracle.lookup_reduce(cfg, t, idx, w), out,
                               rtol=1e-12, atol=1e-14)


def test_mcs_equal_cores_scale_the_output():
    """h equal component cores C/h: every individual score is g/h, so each
    slice gets weight g/h and the output is 1/h of the one-core layer's."""
    cfg = _f32_cfg(cores=2, d_v=8, heads=2)
    t = util.numpy_layer(cfg, B=3)
    t1 = util.numpy_layer(dict(cfg, cores=0), B=3)
    core = t1["core"] * 2
    t["core"] = np.stack([core / 2, core / 2], axis=1).astype(np.float32)
    t1["core"] = core.astype(np.float32)
    out, idx, w = oracle.forward(cfg, t, B=3)
    out1, idx1, w1 = oracle.forward(dict(cfg, cores=0), t1, B=3)
    np.testing.assert_array_equal(idx, idx1)
    np.testing.assert_allclose(w, np.repeat(w1[..., None] / 2, 2, axis=-1), rtol=1e-12)
    np.testing.assert_allclose(out, out1 / 2, rtol=1e-11, atol=1e-14)


def test_mcs_one_core_is_plain():
    """h = 1 is the layer without MCS: same addresses, weights and output."""
    cfg = _f32_cfg()
    t = util.numpy_layer(cfg, B=3)
    a = oracle.forward(cfg, t, B=3)
    b = oracle.forward(dict(cfg, cores=1), dict(t, core=t["core"][:, None]), B=3)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


# ---- query-side extras (Sec. 3.1, Trick 4 convolution, Trick 2 LayerNorm) ----

def _conv_layer(cfg, B, taps=None, bias=None, state_seqs=None):
    t = util.numpy_layer(cfg, B=B)
    if taps is not None:
        t["conv_w"] = np.asarray(taps, np.float32)
        t["conv_b"] = None if bias is None else np.asarray(bias, np.float32)
    if state_seqs:
        t["conv_state"] = workloads.stored_numpy(workloads.make_conv_state(cfg, state_seqs))
    return t


def test_identity_conv_is_no_conv():
    """Taps [1, 0, ..] without bias leave the query input unchanged."""
    cfg = _f32_cfg(conv_k=3)
    taps = np.zeros((3, cfg["d_in"]))
    taps[0] = 1
    t = _conv_layer(cfg, 6, taps)
    plain = oracle.forward(dict(cfg, conv_k=0), t, B=6)
    for a, b in zip(oracle.forward(cfg, t, B=6), plain):
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("lag", [1, 2])
def test_shift_conv_reads_previous_tokens(lag):
    """One tap at lag j makes the query input the token j positions back in
    its own sequence, or the state row before the sequence: the layer then
    equals the plain layer on those shifted rows."""
    cfg = _f32_cfg(conv_k=3)
    S, L = 3, 4
    taps = np.zeros((3, cfg["d_in"]))
    taps[lag] = 1
    t = _conv_layer(cfg, S * L, taps, state_seqs=S)
    t["seq_len"] = L
    x, st = t["x"].reshape(S, L, -1), t["conv_state"]
    shifted = np.concatenate([st, x], axis=1)[:, 2 - lag:2 - lag + L].reshape(S * L, -1)
    t0 = dict(t, x=np.ascontiguousarray(shifted))
    plain = oracle.forward(dict(cfg, conv_k=0), t0, B=S * L)
    for a, b in zip(oracle.forward(cfg, t, B=S * L), plain):
        np.testing.assert_array_equal(a, b)


def test_conv_equals_numpy_convolution():
    """The causal depthwise convolution against numpy's np.convolve per
    channel, on small integers and quarter taps so that every input, product
    and sum is exact in fp32: the layer equals the plain layer on x~."""
    cfg = _f32_cfg(conv_k=4)
    B, rng = 9, np.random.default_rng(3)
    t = util.numpy_layer(cfg, B=B)
    t["x"] = rng.integers(-3, 4, (B, cfg["d_in"])).astype(np.float32)
    t["conv_w"] = (rng.integers(-4, 5, (4, cfg["d_in"])) / 4).astype(np.float32)
    t["conv_b"] = (rng.integers(-2, 3, cfg["d_in"]) / 2).astype(np.float32)
    xt = np.stack([np.convolve(t["x"][:, c], t["conv_w"][:, c])[:B]
                   for c in range(cfg["d_in"])], axis=1) + t["conv_b"]
    plain = oracle.forward(dict(cfg, conv_k=0), dict(t, x=xt.astype(np.float32)), B=B)
    for a, b in zip(oracle.forward(cfg, t, B=B), plain):
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("first", [1, 2, 5])
def test_conv_state_carries_sequences_across_calls(first):
    """Two sequences of 7 tokens in one call equal the same sequences cut
    after `first` tokens, the second call starting from the state the first
    left (decode is the case of one token per call)."""
    cfg = _f32_cfg(conv_k=4, query_ln=1, ln_eps=1e-5)
    S, L = 2, 7
    t = _conv_layer(cfg, S * L, state_seqs=S)
    t["seq_len"] = L
    whole = oracle.forward(cfg, t, B=S * L)
    x = t["x"].reshape(S, L, -1)
    t1 = dict(t, x=np.ascontiguousarray(x[:, :first].reshape(S * first, -1)), seq_len=first)
    part1 = oracle.forward(cfg, t1, B=S * first)
    st = oracle.conv_state(cfg, t1, B=S * first).astype(np.float32)
    rest = L - first
    t2 = dict(t, x=np.ascontiguousarray(x[:, first:].reshape(S * rest, -1)), seq_len=rest,
              conv_state=st)
    part2 = oracle.forward(cfg, t2, B=S * rest)
    for a, p1, p2 in zip(whole, part1, part2):
        a = a.reshape(S, L, *a.shape[1:])
        np.testing.assert_array_equal(a[:, :first], p1.reshape(S, first, *p1.shape[1:]))
        np.testing.assert_array_equal(a[:, first:], p2.reshape(S, rest, *p2.shape[1:]))


def test_conv_state_is_the_last_inputs():
    """The state after a call: the last conv_k - 1 inputs of each sequence,
    reaching into the previous state when a sequence is shorter."""
    cfg = _f32_cfg(conv_k=4)
    t = _conv_layer(cfg, 6, state_seqs=3)
    x = t["x"]
    for L in (3, 2, 1):
        S = 6 // L if L != 1 else 3
        tt = dict(t, x=np.ascontiguousarray(x[:S * L]), seq_len=L)
        got = oracle.conv_state(cfg, tt, B=S * L)
        hist = np.concatenate([t["conv_state"][:S], x[:S * L].reshape(S, L, -1)], axis=1)
        np.testing.assert_array_equal(got, hist[:, -3:])


@pytest.mark.parametrize("share", [1, 0])
def test_query_layernorm_against_torch(share):
    """Trick 2 on each head's query against torch.nn.functional.layer_norm,
    then Eq. 4 by numpy reshapes; a separate column query has its own gain
    and bias."""
    torch = pytest.importorskip("torch")
    cfg = _f32_cfg(query_ln=1, ln_eps=1e-3, share_query=share)
    t = util.numpy_layer(cfg, B=3)
    r, dk, H = cfg["rank"], cfg["d_k"], cfg["heads"]
    K = workloads.keys_per_axis(cfg)
    g = t["ln_g"].astype(np.float64)
    bb = t["ln_b"].astype(np.float64)
    for b in range(3):
        for h in range(H):
            x = util.widen(t["x"])[b]
            qs = []
            for a, w in enumerate([t["w_q"], t["w_q"] if share else t["w_q_col"]]):
                q = util.widen(w)[h * dk:(h + 1) * dk] @ x
                a = 0 if share else a
                q = torch.nn.functional.layer_norm(
                    torch.from_numpy(q), (dk,), torch.from_numpy(g[a, h * dk:(h + 1) * dk]),
                    torch.from_numpy(bb[a, h * dk:(h + 1) * dk]), eps=1e-3).numpy()
                qs.append(q)
            kr = util.widen(t["k_row"])[h].reshape(K, r, dk // r)
            kc = util.widen(t["k_col"])[h].reshape(K, r, dk // r)
            s_row = np.einsum("iac,ac->ai", kr, qs[0].reshape(r, dk // r))
            s_col = np.einsum("jbc,bc->bj", kc, qs[1].reshape(r, dk // r))
            o_row, o_col = oracle.row_col_scores(cfg, t, b, h)
            np.testing.assert_allclose(o_row, s_row, rtol=1e-10, atol=1e-12)
            np.testing.assert_allclose(o_col, s_col, rtol=1e-10, atol=1e-12)


def test_query_layernorm_is_scale_invariant():
    """With eps = 0, LayerNorm removes any positive scale of the query:
    W_q scaled by 4 (exact in fp32) leaves the layer unchanged."""
    cfg = _f32_cfg(query_ln=1, ln_eps=0.0, conv_k=2)
    t = util.numpy_layer(cfg, B=4)
    base = oracle.forward(cfg, t, B=4)
    scaled = oracle.forward(cfg, dict(t, w_q=t["w_q"] * np.float32(4)), B=4)
    for a, b in zip(base, scaled):
        np.testing.assert_array_equal(a, b)


def test_key_layernorm_against_torch():
    """Trick 2 for keys: each stored key row layer-normalised like
    torch.nn.functional.layer_norm."""
    torch = pytest.importorskip("torch")
    cfg = _f32_cfg(dtype=1)
    t = util.numpy_layer(cfg, B=1)
    dk = cfg["d_k"]
    rng = np.random.default_rng(8)
    g = (1 + 0.1 * rng.standard_normal(dk)).astype(np.float32)
    bb = (0.1 * rng.standard_normal(dk)).astype(np.float32)
    got = oracle.key_ln(t["k_row"], 1, g, bb, eps=1e-5)
    ref = torch.nn.functional.layer_norm(
        torch.from_numpy(util.widen(t["k_row"])), (dk,), torch.from_numpy(g.astype(np.float64)),
        torch.from_numpy(bb.astype(np.float64)), eps=1e-5).numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-10, atol=1e-12)


# ---- product-key scoring (Eq. 2-3) and the exact grid top-m (Eq. 5) ----------

def _pkm_cfg(**kw):
    return _f32_cfg(rank=1, score_mode=1, **kw)


def test_exact_topm_is_the_brute_force_grid():
    """uo_exact_topm against numpy's grid S_row^T C S_col (Eq. 5) over every
    slot, with the summed core under Multi-Core Scoring."""
    for cfg in (_f32_cfg(), _f32_cfg(cores=2, d_v=8), _f32_cfg(rank=3, d_k=12)):
        t = _mcs_layer(cfg, B=3) if cfg.get("cores") else util.numpy_layer(cfg, B=3)
        idx, w = oracle.exact_topm(cfg, t, 3)
        core = parity_core(cfg, t)
        for b in range(3):
            for h in range(cfg["heads"]):
                v, g = util.brute_force_grid(cfg, t, b, h, core[h])
                np.testing.assert_array_equal(idx[b, h], v)
                np.testing.assert_allclose(w[b, h], g, rtol=1e-12, atol=1e-13)


def parity_core(cfg, t):
    c = np.asarray(t["core"], np.float64)
    return c.sum(axis=1) if int(cfg.get("cores", 0)) > 1 else c


def test_exact_topm_equals_search_without_pruning():
    """With k = K the two-phase search keeps every key and is exact."""
    cfg = _f32_cfg()
    cfg["topk"] = workloads.keys_per_axis(cfg)
    t = util.numpy_layer(cfg, B=4)
    _, idx, w = oracle.forward(cfg, t, 4)
    ei, ew = oracle.exact_topm(cfg, t, 4)
    np.testing.assert_array_equal(idx, ei)
    np.testing.assert_array_equal(w, ew)


def test_pkm_scores_are_additive():
    """Eq. 2: with product keys the grid score is s_row[i] + s_col[j]
    (numpy reshapes, rank 1), searched over every slot when k = K."""
    cfg = _pkm_cfg()
    K = workloads.keys_per_axis(cfg)
    cfg["topk"] = K
    t = util.numpy_layer(cfg, B=3)
    t.pop("core")
    _, idx, w = oracle.forward(cfg, t, 3)
    for b in range(3):
        for h in range(cfg["heads"]):
            s_row, s_col = util.numpy_scores(cfg, t, b, h)
            G = (s_row[0][:, None] + s_col[0][None, :]).ravel()
            v = np.arange(K * K)
            pos = util.topm_desc(G, v, cfg["topm"])
            np.testing.assert_array_equal(idx[b, h], v[pos])
            np.testing.assert_allclose(w[b, h], G[pos], rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("act", [0, 1])
def test_pkm_two_phase_is_exact(act):
    """Product keys' two-phase top-m is exact once k >= m: a slot of the
    grid's top m has its row among the top m rows (else m rows would beat
    it in its own column), and its column likewise (Sec. 3.1)."""
    cfg = _pkm_cfg(topk=6, topm=6, act=act)
    t = util.numpy_layer(cfg, B=5)
    t.pop("core")
    _, idx, w = oracle.forward(cfg, t, 5)
    ei, ew = oracle.exact_topm(cfg, t, 5)
    np.testing.assert_array_equal(idx, ei)
    if act == 0:
        np.testing.assert_array_equal(w, ew)
    else:
        np.testing.assert_allclose(w.sum(-1), 1.0, rtol=1e-12)


def test_pkm_needs_rank_one():
    cfg = dict(_pkm_cfg(), rank=2)
    t = util.numpy_layer(_f32_cfg(), B=1)
    with pytest.raises(ValueError):
        oracle.forward(cfg, t, 1)


# ---- backward of the lookup-reduce (Eq. 14-15, App. D) ----------------------

def _torch_lookup_reduce(cfg, t, idx, w, perm):
    """Eq. 14-15 restated in torch (float64, autograd on V, w and W_p)."""
    torch = pytest.importorskip("torch")
    N = cfg["n"] ** 2
    E, dv, do = cfg["expand_e"], cfg["d_v"], cfg["d_out"]
    h = max(1, int(cfg.get("cores", 0)))
    V = torch.tensor(util.widen(t["values"]), requires_grad=True)
    W = torch.tensor(util.widen(t["w_proj"]).reshape(E, dv, do), requires_grad=True) \
        if cfg["has_proj"] else None
    wt = torch.tensor(np.asarray(w, np.float64).reshape(idx.shape + (h,)), requires_grad=True)
    vs = torch.from_numpy(perm[idx.ravel()]).reshape(idx.shape)
    p, row = vs // N, vs % N
    rows = V[row]                                                  # [n, H, m, dv]
    wexp = wt.repeat_interleave(dv // h, dim=-1)                   # slice weights per column
    contrib = wexp * rows
    acc = torch.zeros(idx.shape[0], E, dv, dtype=torch.float64)
    for b in range(idx.shape[0]):
        acc[b] = acc[b].index_add(0, p[b].ravel(), contrib[b].reshape(-1, dv))
    out = torch.einsum("bpc,pco->bo", acc, W) if W is not None else acc[:, 0]
    return out, V, wt, W


@pytest.mark.parametrize("over", [dict(), dict(cores=2, d_v=8), dict(expand_e=1, has_proj=0,
                                                                     d_out=8, d_v=8, n=12)])
def test_lookup_reduce_backward_against_autograd(over):
    """The backward against torch's autograd of the lookup-reduce restated
    in torch (the forward itself checked against the oracle's)."""
    torch = pytest.importorskip("torch")
    cfg = _f32_cfg(**over)
    t = _mcs_layer(cfg, B=4) if cfg.get("cores") else util.numpy_layer(cfg, B=4)
    _, idx, w = oracle.forward(cfg, t, 4)
    # one slot of token 1 repeats one of token 0's: its row gradient accumulates twice
    idx[1, 0, 0] = idx[0, 1, 2]
    M = cfg["expand_e"] * cfg["n"] ** 2
    perm = oracle.shuffle(cfg, np.arange(M))
    out, V, wt, W = _torch_lookup_reduce(cfg, t, idx, w, perm)
    np.testing.assert_allclose(out.detach().numpy(), oracle.lookup_reduce(cfg, t, idx, w),
                               rtol=1e-12, atol=1e-14)
    g = np.random.default_rng(4).standard_normal(out.shape).astype(np.float32)
    (out * torch.from_numpy(g.astype(np.float64))).sum().backward()
    dv, dw, dwp = oracle.lookup_reduce_backward(cfg, t, idx, w, g)
    np.testing.assert_allclose(dv, V.grad.numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(dw.reshape(wt.grad.shape), wt.grad.numpy(), rtol=1e-12,
                               atol=1e-14)
    if W is not None:
        np.testing.assert_allclose(dwp, W.grad.numpy(), rtol=1e-12, atol=1e-14)


def test_lookup_reduce_backward_finite_differences():
    """The loss sum(g * o) is linear in each of V, w and W_p, so a change of
    one stored entry by d changes it by exactly d times that entry's
    gradient (up to fp64 rounding): checked through the oracle's forward."""
    cfg = _f32_cfg()
    t = util.numpy_layer(cfg, B=3)
    _, idx, w = oracle.forward(cfg, t, 3)
    g = np.random.default_rng(6).standard_normal((3, cfg["d_out"])).astype(np.float32)
    dv, dw, dwp = oracle.lookup_reduce_backward(cfg, t, idx, w, g)
    base = (oracle.lookup_reduce(cfg, t, idx, w) * g).sum()
    perm = oracle.shuffle(cfg, np.arange(cfg["expand_e"] * cfg["n"] ** 2))
    row = int(perm[idx[2, 1, 3]] % cfg["n"] ** 2)
    for c in (0, 5):
        V = t["values"].copy()
        V[row, c] = np.float32(V[row, c] + 2.0 ** -10)
        d = float(V[row, c]) - float(t["values"][row, c])
        got = (oracle.lookup_reduce(cfg, dict(t, values=V), idx, w) * g).sum() - base
        np.testing.assert_allclose(got, d * dv[row, c], rtol=1e-9, atol=1e-15)
    w2 = w.copy()
    w2[2, 1, 3] += 0.125
    got = (oracle.lookup_reduce(cfg, t, idx, w2) * g).sum() - base
    np.testing.assert_allclose(got, 0.125 * dw[2, 1, 3], rtol=1e-9, atol=1e-15)
    Wp = t["w_proj"].copy()
    Wp[1, 3, 4] = np.float32(Wp[1, 3, 4] + 2.0 ** -8)
    d = float(Wp[1, 3, 4]) - float(t["w_proj"][1, 3, 4])
    got = (oracle.lookup_reduce(cfg, dict(t, w_proj=Wp), idx, w) * g).sum() - base
    np.testing.assert_allclose(got, d * dwp[1, 3, 4], rtol=1e-9, atol=1e-15)
