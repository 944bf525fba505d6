"""Helpers shared by the tests: small seeded layers and independent numpy
restatements used to pin the oracle (brute force over the whole grid, the
explicitly materialised virtual table, numpy's SVD)."""
from __future__ import annotations

import numpy as np

from paper_2411_12364_gb300 import workloads


def numpy_layer(cfg: dict, B: int, batch_index: int = 0) -> dict:
    """Seeded weights and tokens of a layer as the oracle reads them."""
    w = workloads.make_weights(cfg, device="cpu")
    t = {k: workloads.stored_numpy(v) for k, v in w.items()}
    t["x"] = workloads.stored_numpy(workloads.make_tokens(cfg, B, batch_index))
    return t


def widen(a) -> np.ndarray:
    """Stored array (float32 or bf16 bits in uint16) as float64."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def numpy_rank1(core: np.ndarray):
    """Leading singular pair of each head's core from numpy's SVD, with the
    sign rule sum(u) > 0 (first non-zero entry positive if the sum is 0)."""
    H = core.shape[0]
    r = core.shape[1]
    u = np.zeros((H, r))
    t = np.zeros((H, r))
    for h in range(H):
        U, S, Vt = np.linalg.svd(core[h].astype(np.float64))
        uu, tt = U[:, 0], Vt[0]
        s = uu.sum()
        flip = s < 0 or (s == 0 and uu[np.nonzero(uu)[0][0]] < 0)
        if flip:
            uu, tt = -uu, -tt
        u[h], t[h] = uu, tt
    return u, t


def numpy_scores(cfg: dict, t: dict, b: int, h: int):
    """Eq. 4 written with numpy reshapes: S_row, S_col in R^{r x K}."""
    r, dk = cfg["rank"], cfg["d_k"]
    x = widen(t["x"])[b]
    wq = widen(t["w_q"])[h * dk:(h + 1) * dk]
    q_row = wq @ x
    q_col = q_row if cfg["share_query"] else widen(t["w_q_col"])[h * dk:(h + 1) * dk] @ x
    K = workloads.keys_per_axis(cfg)
    kr = widen(t["k_row"])[h].reshape(K, r, dk // r)
    kc = widen(t["k_col"])[h].reshape(K, r, dk // r)
    s_row = np.einsum("iac,ac->ai", kr, q_row.reshape(r, dk // r))
    s_col = np.einsum("jbc,bc->bj", kc, q_col.reshape(r, dk // r))
    return s_row, s_col


def topm_desc(scores: np.ndarray, index: np.ndarray, m: int) -> np.ndarray:
    """Positions of the m largest fp32-rounded scores, ties to the smaller
    index, in (score desc, index asc) order."""
    key = scores.astype(np.float32)
    order = np.lexsort((index, -key.astype(np.float64)))
    return order[:m]


def brute_force_grid(cfg: dict, t: dict, b: int, h: int, core: np.ndarray):
    """Eq. 5 over all K*K slots: returns (v, g) of the top-m in order."""
    s_row, s_col = numpy_scores(cfg, t, b, h)
    G = s_row.T @ core.astype(np.float64) @ s_col  # [K, K]
    K = G.shape[0]
    v = np.arange(K * K, dtype=np.int64)
    pos = topm_desc(G.ravel(), v, cfg["topm"])
    return v[pos], G.ravel()[pos]


def explicit_ive(cfg: dict, t: dict, idx: np.ndarray, w: np.ndarray, perm: np.ndarray):
    """Eq. 13-15 the expensive way: materialise V~ = [V W_0; ...; V W_{E-1}],
    scatter the weights into s^ at the shuffled addresses, o = V~^T s^."""
    V = widen(t["values"])
    E = cfg["expand_e"]
    if cfg["has_proj"]:
        Wp = widen(t["w_proj"])
        Vt = np.concatenate([V @ Wp[p] for p in range(E)], axis=0)
    else:
        Vt = V
    out = np.zeros((idx.shape[0], Vt.shape[1]))
    for b in range(idx.shape[0]):
        s_hat = np.zeros(Vt.shape[0])
        np.add.at(s_hat, perm[idx[b].ravel()], w[b].ravel())
        out[b] = Vt.T @ s_hat
    return out
