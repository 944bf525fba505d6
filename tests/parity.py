"""GPU-vs-oracle comparison rules shared by the parity tests and smoke().

Selected slots must match the oracle exactly (as sets per head; order is
compared by score, so only sets are required to be equal) except for a head
whose oracle scores have a near-tie at a decision boundary: the k-th and
(k+1)-th rank-1 score of an axis, or the m-th and (m+1)-th exact score of
the survivors, closer than ``TIE_REL`` relative.  An excused head must still
select valid slots (each no worse than the oracle's m-th score within the
same tolerance), and the token's output is then compared with the oracle's
lookup-reduce of the GPU's own slots.

Output tolerance: per token, max_e |y - y_ref| / max_e |y_ref| <= 1e-4 in
fp32 mode and 2e-2 in bf16 mode.  Weights: |w - w_ref| <= 1e-4 * max |w_ref|
per head (over all h weights of a slot with Multi-Core Scoring).  With MCS
the selection and the near-tie rule use each head's summed core (Eq. 16).
"""
from __future__ import annotations

import numpy as np

import oracle
from paper_2411_12364_gb300 import workloads
from tests import util

TIE_REL = 1e-5
W_TOL = 1e-4


def out_tol(cfg):
    return 1e-4 if int(cfg["dtype"]) == 0 else 2e-2


def _gap_is_tie(vals, kk):
    if kk >= vals.size:
        return False
    srt = np.sort(vals)[::-1]
    scale = max(abs(srt[kk - 1]), abs(srt[kk]), 1e-3 * np.abs(vals).max(), 1e-30)
    return (srt[kk - 1] - srt[kk]) <= TIE_REL * scale


def tucker_core(cfg, t):
    """[H, r, r] fp64: each head's Tucker core, the sum of its component
    cores when there are h > 1 of them (Eq. 16)."""
    c = np.asarray(t["core"], np.float64)
    return c.sum(axis=1) if int(cfg.get("cores", 0)) > 1 else c


def head_scores(cfg, t, b, h):
    """Oracle's Eq. 4 scores, rank-1 scores and the survivors' exact scores."""
    s_row, s_col = oracle.row_col_scores(cfg, t, b, h)
    u = np.asarray(t["u"], np.float64)[h]
    tt = np.asarray(t["t"], np.float64)[h]
    return s_row, s_col, u @ s_row, tt @ s_col


def near_tie(cfg, t, b, h):
    k, m = int(cfg["topk"]), int(cfg["topm"])
    s_row, s_col, a, bb = head_scores(cfg, t, b, h)
    if _gap_is_tie(a, k) or _gap_is_tie(bb, k):
        return True
    I = np.argsort(-a, kind="stable")[:k]
    J = np.argsort(-bb, kind="stable")[:k]
    G = grid(cfg, t, h, s_row[:, I], s_col[:, J])
    return _gap_is_tie(G.ravel(), m)


def grid(cfg, t, h, s_row, s_col):
    """Grid scores of the given row and column score columns: Eq. 5's
    S_row^T C S_col, or Eq. 2's s_row + s_col with product keys."""
    if int(cfg.get("score_mode", 0)) == 1:
        return s_row[0][:, None] + s_col[0][None, :]
    return s_row.T @ tucker_core(cfg, t)[h] @ s_col


def slot_scores(cfg, t, b, h, v):
    """Exact Eq. 5 score of given virtual addresses v = i*K + j."""
    K = workloads.keys_per_axis(cfg)
    s_row, s_col, _, _ = head_scores(cfg, t, b, h)
    i, j = np.asarray(v) // K, np.asarray(v) % K
    if int(cfg.get("score_mode", 0)) == 1:
        return s_row[0][i] + s_col[0][j]
    C = tucker_core(cfg, t)[h]
    return np.einsum("an,ab,bn->n", s_row[:, i], C, s_col[:, j])


def compare(cfg, t, tokens, gpu_out, gpu_idx, gpu_w, ora_out, ora_idx, ora_w):
    """Asserts parity for the listed tokens.  gpu_* are indexed by token id,
    ora_* by position in ``tokens``.  Returns (excused heads, max out error)."""
    H = int(cfg["heads"])
    excused_pos = []
    n_excused = 0
    for e, b in enumerate(tokens):
        tok_excused = False
        for h in range(H):
            gi, oi = gpu_idx[b, h], ora_idx[e, h]
            if np.array_equal(np.sort(gi), np.sort(oi)):
                gw = gpu_w[b, h][np.argsort(gi)]
                ow = ora_w[e, h][np.argsort(oi)]
                lim = W_TOL * max(np.abs(ow).max(), 1e-30)
                assert np.abs(gw - ow).max() <= lim, \
                    f"weights differ at token {b} head {h}: {np.abs(gw - ow).max()} > {lim}"
                continue
            assert near_tie(cfg, t, b, h), \
                f"selected slots differ at token {b} head {h} without a near-tie"
            ref = np.sort(slot_scores(cfg, t, b, h, oi))[::-1]
            got = slot_scores(cfg, t, b, h, gi)
            assert len(set(gi.tolist())) == gi.size, "duplicate slot selected"
            scale = max(np.abs(ref).max(), 1e-30)
            assert got.min() >= ref[-1] - 10 * TIE_REL * scale, \
                f"invalid slot at token {b} head {h}"
            tok_excused = True
            n_excused += 1
        if tok_excused:
            excused_pos.append(e)
    ref = np.array(ora_out, dtype=np.float64, copy=True)
    if excused_pos:
        tok = np.asarray(tokens)[excused_pos]
        ref[excused_pos] = oracle.lookup_reduce(cfg, t, gpu_idx[tok], gpu_w[tok].astype(np.float64))
    got = np.asarray(gpu_out, np.float64)[np.asarray(tokens)]
    den = np.maximum(np.abs(ref).max(axis=1), 1e-30)
    err = (np.abs(got - ref).max(axis=1) / den)
    tol = out_tol(cfg)
    worst = int(np.argmax(err))
    assert err.max() <= tol, f"output error {err.max():.3g} > {tol} at token {tokens[worst]}"
    return n_excused, float(err.max())


def numpy_inputs(cfg, weights, x):
    """The oracle's view of device tensors (exact copies), with (u, t) from
    numpy's SVD so that both sides prune with the same singular pair."""
    t = {k: workloads.stored_numpy(v) for k, v in weights.items() if k not in ("u", "t")}
    t["x"] = workloads.stored_numpy(x)
    if int(cfg.get("score_mode", 0)) == 1:   # product keys: the axis scores themselves
        H = int(cfg["heads"])
        t["u"] = t["t"] = np.ones((H, 1), np.float32)
        return t
    u, tt = util.numpy_rank1(tucker_core(cfg, t))
    t["u"], t["t"] = u.astype(np.float32), tt.astype(np.float32)
    return t
