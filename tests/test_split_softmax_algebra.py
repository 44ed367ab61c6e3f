"""The arithmetic behind the attention kernels' key splits, checked in fp64 on the CPU.

Each split walks its 64-key blocks with a lazily moved running maximum (moved only when a
block's maximum exceeds it by more than 8 in log2 units, so probabilities stay below 2^8) and
keeps unnormalised sums; splits are combined as o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s
with M the largest running maximum. That equals softmax(scores) V exactly up to rounding, for
any split of the key blocks, including splits in which a row sees no key at all (state and
context rows see only the prefix)."""

import numpy as np
import pytest

KEYS = 64
RESCALE = 8.0


def _split_pass(s2, v, vis, blocks):
    """One split over key blocks `blocks`: scores in log2 units s2 [rows][keys], values v
    [keys][d], visible-key counts vis [rows]. Returns (m, l, O) and the largest probability."""
    rows, d = s2.shape[0], v.shape[1]
    m = np.full(rows, -np.inf)
    l = np.zeros(rows)
    o = np.zeros((rows, d))
    pmax = 0.0
    for blk in blocks:
        k0, k1 = blk * KEYS, min((blk + 1) * KEYS, s2.shape[1])
        idx = np.arange(k0, k1)
        seen = idx[None, :] < vis[:, None]
        sb = np.where(seen, s2[:, k0:k1], -np.inf)
        mb = sb.max(axis=1)
        move = mb > m + RESCALE
        # Where the maximum moves, mb is finite; a row that had seen nothing drops its (zero) sums.
        m_f, mb_f = np.where(np.isinf(m), 0.0, m), np.where(np.isinf(mb), 0.0, mb)
        alpha = np.where(move, np.where(np.isinf(m), 0.0, np.exp2(m_f - mb_f)), 1.0)
        o *= alpha[:, None]
        l *= alpha
        m = np.where(move, mb, m)
        has = ~np.isinf(m)
        p = np.where(seen & has[:, None], np.exp2(sb - np.where(has, m, 0.0)[:, None]), 0.0)
        pmax = max(pmax, float(p.max(initial=0.0)))
        l += p.sum(axis=1)
        o += p @ v[k0:k1]
    return m, l, o, pmax


def _combine(parts):
    ms = np.stack([p[0] for p in parts])
    M = ms.max(axis=0)
    w = np.where(np.isinf(ms), 0.0, np.exp2(np.where(np.isinf(ms), 0.0, ms - np.where(np.isinf(M), 0.0, M))))
    num = sum(w[i][:, None] * parts[i][2] for i in range(len(parts)))
    den = sum(w[i] * parts[i][1] for i in range(len(parts)))
    return np.where(den[:, None] > 0, num / np.where(den > 0, den, 1.0)[:, None], 0.0)


def _exact(s2, v, vis):
    out = np.zeros((s2.shape[0], v.shape[1]))
    for r in range(s2.shape[0]):
        if vis[r] == 0:
            continue
        e = np.exp2(s2[r, :vis[r]] - s2[r, :vis[r]].max())
        out[r] = (e / e.sum()) @ v[:vis[r]]
    return out


@pytest.mark.parametrize("nk,nsplit,gain", [(866, 1, 1.0), (866, 2, 1.0), (866, 3, 1.0), (866, 4, 1.0),
                                            (866, 4, 40.0), (84, 2, 5.0), (64, 1, 1.0), (2099, 4, 3.0)])
def test_split_combine_equals_softmax(nk, nsplit, gain):
    rng = np.random.default_rng(nk * 10 + nsplit)
    rows, d, prefix = 96, 32, max(1, nk - 51)
    s2 = gain * rng.standard_normal((rows, nk))
    v = rng.standard_normal((nk, d))
    # Rows 0..7 see the prefix only (the state token's heads), one row sees nothing (padding).
    vis = np.full(rows, nk)
    vis[:8] = prefix
    vis[8] = 0
    nb = (nk + KEYS - 1) // KEYS
    parts = []
    for sp in range(nsplit):
        b0, b1 = sp * nb // nsplit, (sp + 1) * nb // nsplit
        m, l, o, pmax = _split_pass(s2, v, vis, range(b0, b1))
        assert pmax <= 2.0 ** RESCALE
        parts.append((m, l, o))
    got = _combine(parts)
    want = _exact(s2, v, vis)
    assert np.abs(got - want).max() <= 1e-12 * max(1.0, np.abs(want).max())
    assert not got[8].any()


def test_a_split_whose_rows_see_no_key_weighs_nothing():
    # Two splits; the second holds only keys past the prefix, invisible to the first 8 rows.
    rng = np.random.default_rng(7)
    nk, rows, d = 256, 16, 8
    s2 = rng.standard_normal((rows, nk))
    v = rng.standard_normal((nk, d))
    vis = np.full(rows, nk)
    vis[:8] = 128
    parts = [_split_pass(s2, v, vis, [0, 1])[:3], _split_pass(s2, v, vis, [2, 3])[:3]]
    assert np.isinf(parts[1][0][:8]).all() and not parts[1][1][:8].any()
    got = _combine(parts)
    assert np.abs(got - _exact(s2, v, vis)).max() <= 1e-12
