"""The candidate lists' bound (the scoring's second form, Eq. 8-9): per
(token, head, axis) the keys are taken in groups of 16, tau is the largest
value with zero low 16 bits that at least k group maxima reach (on the
order-preserving 32-bit keys of the fp32 scores), and the lists keep every
key >= tau.  Whatever the scores, the axis' top k (score descending, then
the smaller index) must lie in the list, and the list holds at least k
keys.  Checked here on the rule itself, in plain numpy, over random,
clustered, tied and padded inputs; the GPU tests check the kernels' lists
against scoring every key bit for bit."""
import numpy as np
import pytest

GROUP = 16


def order_keys(scores):
    """The order-preserving 32-bit key of each fp32 score (-0 and +0 alike)."""
    u = (np.asarray(scores, np.float32) + np.float32(0.0)).view(np.uint32).astype(np.uint64)
    return np.where(u & 0x80000000, (~u) & 0xFFFFFFFF, u | 0x80000000)


def bound(keys, k):
    """Largest T with zero low 16 bits such that k group maxima are >= T."""
    n = len(keys)
    maxima = np.array([keys[g:g + GROUP].max() for g in range(0, n, GROUP)])
    t = 0
    for bit in range(31, 15, -1):
        c = t | (1 << bit)
        if (maxima >= c).sum() >= k:
            t = c
    return t


def top_k(keys, k):
    """Indices of the k largest keys, ties to the smaller index."""
    order = sorted(range(len(keys)), key=lambda i: (-int(keys[i]), i))
    return order[:k]


CASES = [
    ("normal", 2048, 32),
    ("normal", 4096, 64),
    ("normal", 1202, 64),      # a partial last group
    ("clustered", 2048, 32),   # scores within 1e-3 of each other
    ("tied", 1200, 16),        # every score the same
    ("few_levels", 4096, 64),  # scores on a coarse grid: many ties
    ("signs", 2048, 32),       # negative and positive, with zeros
]


@pytest.mark.parametrize("kind,n,k", CASES)
def test_bound_keeps_the_top_k(kind, n, k):
    rng = np.random.default_rng(sum(map(ord, kind)) * 7919 + n + k)   # seeded per case
    for trial in range(20):
        if kind == "normal":
            s = rng.normal(0.0, 1.0, n)
        elif kind == "clustered":
            s = 1.0 + rng.normal(0.0, 1e-3, n)
        elif kind == "tied":
            s = np.full(n, rng.normal())
        elif kind == "few_levels":
            s = np.round(rng.normal(0.0, 1.0, n), 1)
        else:
            s = rng.normal(0.0, 1.0, n)
            s[rng.choice(n, n // 8, replace=False)] = 0.0
            s[rng.choice(n, n // 16, replace=False)] = -0.0
        keys = order_keys(s)
        tau = bound(keys, k)
        assert tau & 0xFFFF == 0
        listed = keys >= tau
        assert listed.sum() >= k
        assert all(listed[i] for i in top_k(keys, k))
        # k distinct groups reach tau, so it is at most the k-th largest maximum
        maxima = np.sort([keys[g:g + GROUP].max() for g in range(0, n, GROUP)])[::-1]
        assert tau <= maxima[k - 1]


def test_order_keys_are_monotone():
    """Larger fp32 scores map to larger keys; -0 and +0 share one key."""
    s = np.array([-np.inf, -3.5, -1e-30, -0.0, 0.0, 1e-30, 2.0, np.inf], np.float32)
    keys = order_keys(s)
    assert keys[3] == keys[4]
    assert all(keys[i] < keys[i + 1] for i in range(len(s) - 1) if i != 3)
