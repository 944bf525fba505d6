"""GPU-vs-oracle comparison rules shared by the parity tests and smoke().

Selected slots must match the oracle exactly (as sets per head; order is
compared by score, so only sets are required to be equal) except for a head
whose oracle scores have a near-tie at a decision boundary: the k-th and
(k+1)-th rank-1 score of an axis, or the m-th and (m+1)-th exact score of
the survivors, closer than ``TIE_REL`` relative.  An excused head must still
select valid slots (each no worse than the oracle's m-th score within the
same tolerance), and the token's output is then compared with the oracle's
lookup-reduce of the GPU's own slots.

Output tolerance, element-wise with a floor: per token,
max_e |y_e - y_ref_e| / max(|y_ref_e|, 1e-3 max_e' |y_ref_e'|) <= 1e-4 in fp32
mode and 2e-2 in bf16 mode (the floor keeps the ratio defined for elements
near 0).  The normwise figure max_e |y - y_ref| / max_e |y_ref| is reported
beside it.  Weights: |w - w_ref| <= 1e-4 * max |w_ref| per head (over all h
weights of a slot with Multi-Core Scoring).  With MCS the selection and the
near-tie rule use each head's summed core (Eq. 16).

A near-tie is a gap of at most 1e-5 relative to the two boundary scores
themselves.  Boundary scores near 0 come from cancellation, where an fp32
result is only accurate to the size of the cancelled terms, so a gap within
1e-5 of 1e-3 times the head's largest score also counts; such heads are
counted separately (``floor_ties``), and the workload tests require none.
"""
from __future__ import annotations

import numpy as np

import oracle
from paper_2411_12364_gb300 import workloads
from tests import util

TIE_REL = 1e-5
W_TOL = 1e-4
OUT_FLOOR = 1e-3     # of the token's largest |y_ref|: the element-wise denominator's floor


def out_tol(cfg):
    return 1e-4 if int(cfg["dtype"]) == 0 else 2e-2


NO_TIE, TIE, FLOOR_TIE = 0, 1, 2


def tie_kind(vals, kk):
    """Whether the kk-th and (kk+1)-th largest of vals are a near-tie: TIE
    when their gap is within TIE_REL of the larger of the two, FLOOR_TIE when
    it is only within TIE_REL of 1e-3 max |vals| (cancellation near 0)."""
    if kk >= vals.size:
        return NO_TIE
    srt = np.sort(vals)[::-1]
    gap = srt[kk - 1] - srt[kk]
    if gap <= TIE_REL * max(abs(srt[kk - 1]), abs(srt[kk]), 1e-30):
        return TIE
    if gap <= TIE_REL * 1e-3 * np.abs(vals).max():
        return FLOOR_TIE
    return NO_TIE


def _gap_is_tie(vals, kk):
    return tie_kind(vals, kk) != NO_TIE


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
    """The kind of near-tie (NO_TIE / TIE / FLOOR_TIE) at the head's decision
    boundaries: either axis' k-th/(k+1)-th rank-1 score, or the survivors'
    m-th/(m+1)-th grid score."""
    k, m = int(cfg["topk"]), int(cfg["topm"])
    s_row, s_col, a, bb = head_scores(cfg, t, b, h)
    kinds = [tie_kind(a, k), tie_kind(bb, k)]
    I = np.argsort(-a, kind="stable")[:k]
    J = np.argsort(-bb, kind="stable")[:k]
    G = grid(cfg, t, h, s_row[:, I], s_col[:, J])
    kinds.append(tie_kind(G.ravel(), m))
    if TIE in kinds:
        return TIE
    return FLOOR_TIE if FLOOR_TIE in kinds else NO_TIE


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


def output_errors(got, ref):
    """Per-token output errors: (element-wise with the floor, normwise)."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    peak = np.abs(ref).max(axis=1, keepdims=True)
    den = np.maximum(np.abs(ref), np.maximum(OUT_FLOOR * peak, 1e-30))
    diff = np.abs(got - ref)
    elem = (diff / den).max(axis=1)
    norm = diff.max(axis=1) / np.maximum(peak[:, 0], 1e-30)
    return elem, norm


class Result(tuple):
    """(excused heads, element-wise output error), with the normwise error
    and the count of heads excused only through the floor as attributes."""

    def __new__(cls, excused, err, err_norm, floor_ties):
        r = super().__new__(cls, (excused, err))
        r.excused, r.err, r.err_norm, r.floor_ties = excused, err, err_norm, floor_ties
        return r


def compare(cfg, t, tokens, gpu_out, gpu_idx, gpu_w, ora_out, ora_idx, ora_w):
    """Asserts parity for the listed tokens.  gpu_* are indexed by token id,
    ora_* by position in ``tokens``.  Returns a Result: (excused heads, max
    element-wise output error), .err_norm, .floor_ties."""
    H = int(cfg["heads"])
    excused_pos = []
    n_excused = 0
    floor_ties = 0
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
            kind = near_tie(cfg, t, b, h)
            assert kind != NO_TIE, f"selected slots differ at token {b} head {h} without a near-tie"
            floor_ties += kind == FLOOR_TIE
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
    err, err_norm = output_errors(got, ref)
    tol = out_tol(cfg)
    worst = int(np.argmax(err))
    assert err.max() <= tol, \
        f"element-wise output error {err.max():.3g} > {tol} at token {tokens[worst]} " \
        f"(normwise {err_norm[worst]:.3g})"
    return Result(n_excused, float(err.max()), float(err_norm.max()), floor_ties)


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
