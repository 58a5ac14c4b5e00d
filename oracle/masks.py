"""Layer-dropout masks M^{l,t} and kept-sequence lists.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Follows Eq. (layer_dropout_train): M^{l,t} in {0,1}^B with entries drawn
Bernoulli(1 - p^{l,t}); the Tensor Granularity subsection: per-sequence (one
independent draw per sequence b) or per-batch (one draw per layer and step,
shared by every b); and the "more efficient implementation" paragraph of the
Preliminary section: the layer runs only on {b_i : M[b_i] = 1}.

Reading of the draw (the paper names no generator):
  u = word 0 of Philox4x32-10 with key (seed mod 2^32, seed >> 32) and
      counter (b', l, t mod 2^32, t >> 32), where b' = b per sequence and
      b' = 0 per batch (so a per-batch mask is the per-sequence draw of
      sequence 0, broadcast);
  the layer is dropped for that sequence iff u < thr_l, thr_l = floor(p 2^32).
Per shard (the paper's per-device batch dropping for data parallelism, Tensor
Granularity subsection): b' = b_offset, the shard's first global sequence,
for every sequence of the shard -- one draw per layer and step per shard.
Sub-layer granularity (Model Granularity subsection: M_attn and M_ffn drawn
independently, each Bernoulli(1 - p^{l,t})): the attention mask uses word 0
of the same Philox output and the FFN mask word 1, so the attention mask is
the layer-granularity mask.
Kept lists are in ascending b.

Per token (finer than per sequence; the Tensor Granularity subsection names it
as future work, so the draw and the layer's meaning are this package's
reading): M^{l,t}[b, s] ~ Bernoulli(1 - p^{l,t}) for each token, from word 2
of the Philox output for the counter (g, l, t mod 2^32, t >> 32) with
g = (b_offset + b) S + s the global token index (word 3 for the FFN mask
with sub-layer granularity).  A kept token runs the layer; the kept tokens
of a sequence form a shorter sequence that keeps their original order and
positions, and a dropped token neither changes nor contributes keys and
values at that layer.  Kept token lists hold the row b S + s of each kept
token in ascending order, with per-sequence segment offsets.
"""

import numpy as np

from .philox import philox4x32_10, philox4x32_10_np

PER_SEQUENCE, PER_BATCH, PER_SHARD, PER_TOKEN = "per_sequence", "per_batch", "per_shard", "per_token"


def mask_word(seed, step, layer, b, word=0):
    """The 32-bit uniform word for (seed, step, layer, sequence): output word
    `word` of Philox4x32-10."""
    seed = int(seed)
    step = int(step)
    key = (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    ctr = (b, layer, step & 0xFFFFFFFF, (step >> 32) & 0xFFFFFFFF)
    return philox4x32_10(ctr, key)[word]


def draw_masks(seed, step, thresholds, B, granularity=PER_SEQUENCE, b_offset=0, sublayer=False, S=None):
    """mask[l][b] in {0,1} (1 = keep) for every layer l (uint8, shape [L, B]);
    with ``sublayer`` the pair (M_attn, M_ffn) as uint8 [2, L, B].  The batch
    holds the global sequences b_offset .. b_offset + B - 1.  Per token
    (needs S): mask[l][b][s], shape [L, B, S] (or [2, L, B, S])."""
    if granularity == PER_TOKEN:
        return draw_token_masks(seed, step, thresholds, B, S, b_offset, sublayer)
    L = len(thresholds)
    nw = 2 if sublayer else 1
    mask = np.zeros((nw, L, B), dtype=np.uint8)
    for w in range(nw):
        for layer in range(L):
            for b in range(B):
                if granularity == PER_SEQUENCE:
                    bb = b_offset + b
                elif granularity == PER_SHARD:
                    bb = b_offset
                else:
                    bb = 0
                u = mask_word(seed, step, layer, bb, w)
                mask[w, layer, b] = 0 if u < thresholds[layer] else 1
    return mask if sublayer else mask[0]


def token_word(seed, step, layer, g, word=2):
    """The 32-bit uniform word of global token g: output word `word` of
    Philox4x32-10 for the counter (g, layer, t mod 2^32, t >> 32)."""
    return mask_word(seed, step, layer, g, word)


def draw_token_masks(seed, step, thresholds, B, S, b_offset=0, sublayer=False):
    """Per-token masks, uint8 [L, B, S] (1 = keep), or [2, L, B, S] with
    ``sublayer`` (attention mask from word 2, FFN mask from word 3)."""
    L = len(thresholds)
    nw = 2 if sublayer else 1
    g = (b_offset + np.arange(B, dtype=np.uint64))[:, None] * np.uint64(S) + np.arange(S, dtype=np.uint64)[None, :]
    mask = np.zeros((nw, L, B, S), dtype=np.uint8)
    for w in range(nw):
        for layer in range(L):
            u = words_np(seed, step, layer, g, word=2 + w)
            mask[w, layer] = (u >= np.uint64(thresholds[layer])).astype(np.uint8)
    return mask if sublayer else mask[0]


def kept_token_lists(mask):
    """Per-token kept lists of a mask [L, B, S]: (rows int32 [L, B*S] holding
    b*S + s of every kept token in ascending order, padded with -1; counts
    int32 [L]; segment offsets int32 [L, B+1], the kept tokens of sequence b
    being rows[l][seg[l][b]:seg[l][b+1]]).  A pair [2, L, B, S] gives each
    array with a leading axis of 2."""
    mask = np.asarray(mask)
    if mask.ndim == 4:
        parts = [kept_token_lists(m) for m in mask]
        return tuple(np.stack([p[i] for p in parts]) for i in range(3))
    L, B, S = mask.shape
    rows = np.full((L, B * S), -1, dtype=np.int32)
    cnt = np.zeros(L, dtype=np.int32)
    seg = np.zeros((L, B + 1), dtype=np.int32)
    for layer in range(L):
        flat = [b * S + s for b in range(B) for s in range(S) if mask[layer, b, s] == 1]
        cnt[layer] = len(flat)
        rows[layer, : len(flat)] = flat
        for b in range(B):
            seg[layer, b + 1] = seg[layer, b] + int(mask[layer, b].sum())
    return rows, cnt, seg


def kept_lists(mask):
    """kept_idx[l] = ascending b with mask[l][b] = 1; kept_cnt[l] = its length.

    Returned as (int32 [L, B] padded with -1, int32 [L]); a sub-layer mask
    [2, L, B] gives ([2, L, B], [2, L])."""
    mask = np.asarray(mask)
    if mask.ndim == 3:
        pairs = [kept_lists(m) for m in mask]
        return np.stack([p[0] for p in pairs]), np.stack([p[1] for p in pairs])
    L, B = mask.shape
    idx = np.full((L, B), -1, dtype=np.int32)
    cnt = np.zeros(L, dtype=np.int32)
    for layer in range(L):
        kept = [b for b in range(B) if mask[layer, b] == 1]
        cnt[layer] = len(kept)
        idx[layer, : len(kept)] = kept
    return idx, cnt


def words_np(seed, step, layer, b, word=0):
    """Vectorised ``mask_word`` over numpy arrays of (step, layer, b)."""
    seed = int(seed)
    step = np.asarray(step, dtype=np.uint64)
    z = np.zeros(np.broadcast(step, layer, b).shape, dtype=np.uint64)
    c0 = np.asarray(b, dtype=np.uint64) + z
    c1 = np.asarray(layer, dtype=np.uint64) + z
    c2 = (step & np.uint64(0xFFFFFFFF)) + z
    c3 = (step >> np.uint64(32)) + z
    k0 = np.uint64(seed & 0xFFFFFFFF) + z
    k1 = np.uint64((seed >> 32) & 0xFFFFFFFF) + z
    return philox4x32_10_np(c0, c1, c2, c3, k0, k1)[word]
