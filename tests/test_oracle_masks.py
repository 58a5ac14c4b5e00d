"""Pins of the oracle's Philox generator and mask draw: published
known-answer vectors, the Bernoulli(1 - p) rate of Eq. (layer_dropout_train),
the per-batch special case of the Tensor Granularity subsection, p = 0 / 1,
and resume-at-step invariance of a counter-based draw."""

import math
import os

import numpy as np
import pytest

from oracle import masks as M
from oracle import philox as P
from oracle import schedule as S

KAT = os.path.join(os.path.dirname(__file__), "golden", "philox_kat.txt")


def _kat_rows():
    rows = []
    for line in open(KAT):
        if line.startswith("#") or not line.strip():
            continue
        v = [int(x, 16) for x in line.split()]
        rows.append((tuple(v[:4]), tuple(v[4:6]), tuple(v[6:])))
    return rows


@pytest.mark.parametrize("row", _kat_rows())
def test_philox_known_answers(row):
    ctr, key, out = row
    assert P.philox4x32_10(ctr, key) == out
    got = P.philox4x32_10_np(*[np.array([c], dtype=np.uint64) for c in ctr],
                             np.array([key[0]], dtype=np.uint64), np.array([key[1]], dtype=np.uint64))
    assert tuple(int(g[0]) for g in got) == out


def test_vectorised_matches_scalar():
    rng = np.random.default_rng(0)
    for _ in range(50):
        seed = int(rng.integers(0, 2 ** 63))
        step, layer, b = int(rng.integers(0, 2 ** 40)), int(rng.integers(0, 64)), int(rng.integers(0, 4096))
        assert int(M.words_np(seed, step, layer, b)) == M.mask_word(seed, step, layer, b)


def test_kept_rate_is_bernoulli():
    # 10^6 draws at p = 0.3: kept fraction within 4 sigma of 1 - p.
    n_steps, L, B = 2000, 25, 20
    st, la, bb = np.meshgrid(np.arange(n_steps), np.arange(L), np.arange(B), indexing="ij")
    u = M.words_np(7, st, la, bb)
    thr = S.drop_threshold(0.3)
    kept = (u >= np.uint64(thr)).mean()
    n = u.size
    assert n == 10 ** 6
    sigma = math.sqrt(0.3 * 0.7 / n)
    assert abs(kept - 0.7) < 4 * sigma
    # words are uniform on [0, 2^32): mean and the low/high halves
    uf = u.astype(np.float64) / 2 ** 32
    assert abs(uf.mean() - 0.5) < 4 * math.sqrt(1 / 12 / n)
    # adjacent sequences / layers / steps are uncorrelated
    for ax in range(3):
        a = np.moveaxis(uf, ax, 0)
        r = np.corrcoef(a[:-1].ravel(), a[1:].ravel())[0, 1]
        assert abs(r) < 5 / math.sqrt(a[:-1].size)


def test_expected_executed_layers():
    # E[# executed layers per sequence] = sum_l (1 - thr_l / 2^32), Monte Carlo.
    L, B = 16, 64
    rates = S.layer_rates(dict(dist="ild", p_max=0.6), L, 0)
    thr = [S.drop_threshold(p) for p in rates]
    expect = sum(1 - t / 2 ** 32 for t in thr)
    assert expect == pytest.approx(S.effective_depth(rates), abs=1e-8)
    runs = []
    for step in range(300):
        mk = M.draw_masks(3, step, thr, B)
        runs.append(mk.sum(axis=0))
    runs = np.concatenate(runs)
    var = sum((1 - t / 2 ** 32) * (t / 2 ** 32) for t in thr)
    assert abs(runs.mean() - expect) < 4 * math.sqrt(var / runs.size)


def test_p0_p1_and_per_batch():
    L, B = 6, 9
    thr = [S.drop_threshold(p) for p in (0.0, 1.0, 0.5, 0.5, 0.9, 0.1)]
    for step in (0, 1, 2 ** 33 + 5):
        mk = M.draw_masks(11, step, thr, B)
        assert mk[0].all() and not mk[1].any()
        pb = M.draw_masks(11, step, thr, B, M.PER_BATCH)
        # per batch = the per-sequence draw of sequence 0, broadcast
        for l in range(L):
            assert (pb[l] == mk[l, 0]).all()


def test_resume_invariance():
    # The draw for step t depends on (seed, t, l, b) only: drawing step 37
    # directly equals drawing it after steps 0..36.
    thr = [S.drop_threshold(0.4)] * 5
    seq = [M.draw_masks(5, t, thr, 12) for t in range(38)]
    assert (M.draw_masks(5, 37, thr, 12) == seq[37]).all()
    assert not all((seq[t] == seq[0]).all() for t in range(1, 38))


def test_threshold_semantics_brute_force():
    # drop iff u < thr, checked word by word on a few thousand draws.
    for p in (0.0, 1e-9, 0.25, 0.5, 0.999, 1.0):
        thr = S.drop_threshold(p)
        mk = M.draw_masks(99, 4, [0, 0, thr], 200)
        for b in range(200):
            u = M.mask_word(99, 4, 2, b)
            assert mk[2, b] == (0 if u < thr else 1)


def test_kept_lists():
    mk = np.array([[1, 0, 1, 1, 0], [0, 0, 0, 0, 0], [1, 1, 1, 1, 1]], dtype=np.uint8)
    idx, cnt = M.kept_lists(mk)
    assert list(cnt) == [3, 0, 5]
    assert list(idx[0][:3]) == [0, 2, 3] and (idx[0][3:] == -1).all()
    assert (idx[1] == -1).all()
    assert list(idx[2]) == [0, 1, 2, 3, 4]


def test_tie_at_threshold_keeps():
    # Reading of the draw: dropped iff u < thr (strict), so a word equal to
    # the threshold keeps the layer and thr = u + 1 drops it.
    for b in range(5):
        u = M.mask_word(2024, 9, 0, b)
        assert M.draw_masks(2024, 9, [u], 5)[0, b] == 1
        assert M.draw_masks(2024, 9, [u + 1], 5)[0, b] == 0


def test_sublayer_masks():
    # Sub-layer granularity: M_attn is the layer-granularity mask (word 0),
    # M_ffn an independent Bernoulli(1 - p) draw (word 1); p = 0 / 1 and the
    # per-batch case behave as for one mask; kept lists per block.
    thr = [S.drop_threshold(p) for p in (0.0, 0.3, 0.5, 1.0)]
    for gran in (M.PER_SEQUENCE, M.PER_BATCH):
        pair = M.draw_masks(11, 42, thr, 64, gran, sublayer=True)
        assert pair.shape == (2, 4, 64) and pair.dtype == np.uint8
        assert (pair[0] == M.draw_masks(11, 42, thr, 64, gran)).all()
        assert (pair[:, 0] == 1).all() and (pair[:, 3] == 0).all()
        if gran == M.PER_BATCH:
            assert (pair == pair[:, :, :1]).all()
        idx, cnt = M.kept_lists(pair)
        assert idx.shape == (2, 4, 64) and cnt.shape == (2, 4)
        for w in range(2):
            i1, c1 = M.kept_lists(pair[w])
            assert (idx[w] == i1).all() and (cnt[w] == c1).all()
    # joint frequencies of (attn, ffn) at p = 0.5 over 2 * 10^5 draws: each
    # of the four outcomes within 4 sigma of 1/4
    t2 = [S.drop_threshold(0.5)] * 50
    both = np.stack([M.draw_masks(3, t, t2, 400, sublayer=True) for t in range(10)], axis=1)  # [2, 10, 50, 400]
    a, f = both[0].ravel().astype(np.int64), both[1].ravel().astype(np.int64)
    n = a.size
    sigma = math.sqrt(0.25 * 0.75 / n)
    for va in (0, 1):
        for vf in (0, 1):
            assert abs(((a == va) & (f == vf)).mean() - 0.25) < 4 * sigma
    assert abs(np.corrcoef(a, f)[0, 1]) < 4 / math.sqrt(n)


def test_per_shard_masks():
    # Per-shard draws (per-device batch dropping): a shard's mask is the
    # per-sequence draw of its first global sequence, broadcast over the
    # shard; shard 0 is the per-batch mask; distinct shards draw independently.
    thr = [S.drop_threshold(p) for p in (0.0, 0.4, 0.7, 1.0)]
    B = 8
    for off in (0, 8, 24, 2 ** 31 - 9):
        m = M.draw_masks(3, 17, thr, B, M.PER_SHARD, b_offset=off)
        ref = M.draw_masks(3, 17, thr, 1, M.PER_SEQUENCE, b_offset=off)
        assert (m == ref).all()
    assert (M.draw_masks(3, 17, thr, B, M.PER_SHARD, b_offset=0) == M.draw_masks(3, 17, thr, B, M.PER_BATCH)).all()
    # two shards at p = 0.5 over many (layer, step): they agree on half the draws (independence)
    t2 = [S.drop_threshold(0.5)] * 40
    a = np.stack([M.draw_masks(5, t, t2, 4, M.PER_SHARD, b_offset=0)[:, 0] for t in range(50)]).ravel()
    b = np.stack([M.draw_masks(5, t, t2, 4, M.PER_SHARD, b_offset=4)[:, 0] for t in range(50)]).ravel()
    n = a.size
    assert abs((a == b).mean() - 0.5) < 4 * math.sqrt(0.25 / n)
    assert abs(a.mean() - 0.5) < 4 * math.sqrt(0.25 / n)
