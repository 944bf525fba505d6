"""Host-side checks of the selection kernel's index arithmetic.

The kernel assigns work to threads with closed-form index maps; a map that is
not a bijection would drop or repeat candidates.  These tests evaluate the
same maps on the CPU, exhaustively over the sizes the library accepts
(k <= 128, 256 threads in 8 warps), and check that each covers its range
exactly once.  The fp32 floor division is evaluated in numpy float32, the
precision the kernel computes it in.
"""
import numpy as np
import pytest

THREADS, WARPS = 256, 8
PAIR_MIX = 421            # the kernel's kPairMix: a prime above the largest k
MAX_K = 128


def test_pair_mix_is_prime_above_max_k():
    assert PAIR_MIX > MAX_K
    assert all(PAIR_MIX % d for d in range(2, int(PAIR_MIX ** 0.5) + 1))


@pytest.mark.parametrize("k", range(1, MAX_K + 1))
def test_mixed_pair_order_is_a_bijection(k):
    """Thread t visits p = t, t + 256, ... as pp = p * 421 mod k^2, kept by
    adding (256 * 421) mod k^2 and subtracting k^2 once when it overflows."""
    k2 = k * k
    step = (THREADS * PAIR_MIX) % k2
    seen = np.zeros(k2, dtype=np.int32)
    for t in range(min(THREADS, k2)):
        pp = (t * PAIR_MIX) % k2
        for c in range(t, k2, THREADS):
            assert pp == (c * PAIR_MIX) % k2
            seen[pp] += 1
            pp += step
            if pp >= k2:
                pp -= k2
    assert (seen == 1).all()


@pytest.mark.parametrize("k", range(1, MAX_K + 1))
def test_fp32_floor_division_of_pair_index(k):
    """ii = (int)((pp + 0.5f) * (1.0f / k)) equals pp // k for every pair."""
    pp = np.arange(k * k, dtype=np.int64)
    inv_k = np.float32(1.0) / np.float32(k)
    ii = ((pp.astype(np.float32) + np.float32(0.5)) * inv_k).astype(np.int64)
    assert (ii == pp // k).all()


@pytest.mark.parametrize("k", [32, 64, 96, 128])
def test_diagonal_pair_layout_covers_every_pair_once(k):
    """Lane l of warp w: columns l + 32 h, rows ((w + l) mod 8) + 8 i; every
    warp holds every row and every column of the k x k survivors."""
    owner = np.full((k, k), -1)
    for w in range(WARPS):
        rows_w, cols_w = set(), set()
        for lane in range(32):
            i0 = (w + lane) & 7
            for jj in range(lane, k, 32):
                for ii in range(i0, k, 8):
                    assert owner[ii, jj] == -1
                    owner[ii, jj] = w * 32 + lane
                    rows_w.add(ii)
                    cols_w.add(jj)
        assert rows_w == set(range(k)) and cols_w == set(range(k))
    assert (owner >= 0).all()
    # each thread computes k^2 / 256 pairs
    assert np.bincount(owner.ravel(), minlength=THREADS).tolist() == [k * k // THREADS] * THREADS


@pytest.mark.parametrize("n", [1, 3, 4, 5, 24, 25, 1023, 1024, 1025, 4096, 8960, 16384, 20480])
def test_compaction_groups_cover_the_keys_once(n):
    """A round covers 4 * 256 16-byte groups; lane l of warp w reads groups
    r0 + (q * 8 + w) * 32 + l (q < 4); bit 4q + e of its mask is key
    4 * group + e, kept only below n."""
    n4 = (n + 3) // 4
    seen = np.zeros(n, dtype=np.int32)
    for r0 in range(0, n4, 4 * THREADS):
        for w in range(WARPS):
            for lane in range(32):
                for q in range(4):
                    g = r0 + (q * WARPS + w) * 32 + lane
                    if g >= n4:
                        continue
                    valid = min(4, n - 4 * g)
                    assert valid >= 1
                    for e in range(valid):
                        b = 4 * q + e
                        i = 4 * (r0 + ((b >> 2) * WARPS + w) * 32 + lane) + (b & 3)
                        assert i == 4 * g + e
                        seen[i] += 1
    assert (seen == 1).all()
    # the last group read ends at the 16-byte end of an n-word array
    assert 16 * n4 == ((4 * n + 15) // 16) * 16
