"""Host-side properties of the persistent pass kernel's work schedule (no GPU).

Every CTA walks its items in order and an item spins until the items it reads are done, so the
pass cannot deadlock when (1) every item an item reads comes earlier in the topologically
ordered list that is dealt round-robin to the CTAs (CTA k takes items k, k + grid, ...), and
(2) the items that wait for one another -- the K slices of one linear tile, whose reducers read
each other's partial sums, and the splits of one attention head group, which merge together --
sit on distinct CTAs.  The dependencies below restate what each item reads (the residual stream,
the attention inputs, the merged attention, SiLU-up) from the model's data flow, independently
of the kernel's counters.
"""
import numpy as np
import pytest

from paper_2607_12422_gb300 import pbd, synth

OP_EMBED, OP_LINEAR, OP_ATTN, OP_FINAL = 0, 1, 2, 3
TILE = 128


def _decode(items):
    w = items[:, 0]
    return w & 0xFF, (w >> 8) & 0xFF, w >> 16, items[:, 1], items[:, 2], items[:, 3]


def _global_order(off, grid, n):
    g = np.empty(n, np.int64)
    for c in range(grid):
        for p in range(off[c + 1] - off[c]):
            g[off[c] + p] = c + p * grid
    assert np.array_equal(np.sort(g), np.arange(n)), "the dealing is not a permutation of the list"
    return g


def _check(S, items, off, grid, n_layers_run, slice_w):
    n = len(items)
    g = _global_order(off, grid, n)
    op, lin, layer, a, b, c = _decode(items)
    cta = g % grid
    d, grp = S.head_dim, S.n_q_heads // S.n_kv_heads
    qw, kvw = S.n_q_heads * d, S.n_kv_heads * d
    main_tiles = [(S.n_q_heads + 2 * S.n_kv_heads) * d // TILE, S.hidden // TILE, 2 * S.intermediate // TILE,
                  S.hidden // TILE]
    # completion index (the latest global index) of each group of items a consumer reads
    last = {}

    def note(key, gi):
        last[key] = max(last.get(key, -1), gi)

    for i in range(n):
        if op[i] == OP_EMBED:
            note(("embed",), g[i])
        elif op[i] == OP_LINEAR:
            note(("lin", lin[i], layer[i]), g[i])
            note(("tile", lin[i], layer[i], a[i]), g[i])
        elif op[i] == OP_ATTN:
            note(("att", layer[i], a[i], b[i]), g[i])

    def tiles_over(f0, f1):
        return range(f0 // TILE, (f1 - 1) // TILE + 1)

    for i in range(n):
        l, gi = int(layer[i]), g[i]
        need = []
        if op[i] == OP_LINEAR:
            adapter_tile = ("tile", lin[i], l, main_tiles[lin[i]])
            if lin[i] == 0:  # RMSNorm(h): h after the previous layer's down projection (or the embedding)
                need.append(("lin", 3, l - 1) if l > 0 else ("embed",))
            elif lin[i] == 1:  # the merged attention of the slice's heads, every sequence
                heads = range(b[i] * slice_w[1] // d, ((b[i] + 1) * slice_w[1] - 1) // d + 1)
                need += [k for k in last if k[0] == "att" and k[1] == l and k[3] in {h // grp for h in heads}]
            elif lin[i] == 2:  # RMSNorm(h): h after this layer's o projection
                need.append(("lin", 1, l))
            else:  # SiLU(gate) * up of the slice's features: gate|up tiles of 64 features each
                f0 = b[i] * slice_w[3]
                need += [("tile", 2, l, t) for t in range(f0 // 64, (f0 + slice_w[3] - 1) // 64 + 1)]
                if ("tile", 2, l, main_tiles[2]) in last:  # the draft's gate|up adapter tile
                    need.append(("tile", 2, l, main_tiles[2]))
            if a[i] < main_tiles[lin[i]] and adapter_tile in last:  # main reducers sum the adapter tile
                need.append(adapter_tile)
        elif op[i] == OP_ATTN:
            grp_g = int(b[i])
            for f0, f1 in ((grp_g * grp * d, (grp_g + 1) * grp * d), (qw + grp_g * d, qw + (grp_g + 1) * d),
                           (qw + kvw + grp_g * d, qw + kvw + (grp_g + 1) * d)):
                need += [("tile", 0, l, t) for t in tiles_over(f0, f1)]
            if ("tile", 0, l, main_tiles[0]) in last:
                need.append(("tile", 0, l, main_tiles[0]))
        elif op[i] == OP_FINAL:
            assert l == n_layers_run - 1
            need.append(("lin", 3, l))
        for k in need:
            assert k in last, (k, "is read but never produced")
            assert last[k] < gi, ("item", i, "reads", k, "which completes later in the list")

    # items that wait for one another sit on distinct CTAs, consecutively in the list
    groups = {}
    for i in range(n):
        if op[i] == OP_LINEAR:
            groups.setdefault(("tile", lin[i], layer[i], a[i]), []).append(i)
        elif op[i] == OP_ATTN:
            groups.setdefault(("att", layer[i], a[i], b[i]), []).append(i)
    for k, idx in groups.items():
        gs = np.sort(g[idx])
        assert np.array_equal(gs, np.arange(gs[0], gs[0] + len(gs))), (k, "not consecutive")
        if len(idx) <= grid:
            assert len(set(cta[idx])) == len(idx), (k, "shares a CTA")
    assert set(layer[op == OP_LINEAR]) == set(range(n_layers_run))


def _check_counters(items, off, grid):
    """The host-computed waits agree with the releases: every counter an item waits for receives
    exactly its target of releases, all from items earlier in the list.  Attention splits release
    once each after merging when a group's splits sit on distinct CTAs, else only the last one."""
    n = len(items)
    g = _global_order(off, grid, n)
    op, lin, layer, a, b, c = _decode(items)
    w_off, w_tgt, rel = items[:, 4], items[:, 5], items[:, 6:8]
    att_groups = {}
    for i in np.nonzero(op == OP_ATTN)[0]:
        att_groups.setdefault((layer[i], a[i], b[i]), []).append(i)
    count, last = {}, {}
    for i in range(n):
        if op[i] == OP_ATTN:
            continue
        for r in rel[i]:
            if r >= 0:
                count[r] = count.get(r, 0) + 1
                last[r] = max(last.get(r, -1), g[i])
    for idx in att_groups.values():
        r = rel[idx[0], 0]
        assert (rel[idx, 0] == r).all() and (rel[idx, 1] == -1).all()
        count[r] = count.get(r, 0) + (len(idx) if len(idx) <= grid else 1)
        last[r] = max(last.get(r, -1), max(g[idx]))
    waits = 0
    for i in range(n):
        if w_off[i] < 0:
            assert op[i] == OP_EMBED or (op[i] == OP_LINEAR and lin[i] == 3), i  # down polls act words
            continue
        waits += 1
        assert count.get(w_off[i], 0) == w_tgt[i], (i, "waits for", w_tgt[i], "releases of", w_off[i],
                                                    "which receives", count.get(w_off[i], 0))
        assert last[w_off[i]] < g[i], (i, "waits for a release later in the list")
    assert waits > 0


CASES = [
    ("tiny", synth.TINY, 16, [64], 64),
    ("tiny-b4", synth.TINY, 16, [64, 40, 17, 100], 64),
    ("qwen", synth.QWEN3_0_6B, 16, [512], 256),
    ("qwen-4096", synth.QWEN3_0_6B, 16, [4096], 512),
    ("qwen-b8", synth.QWEN3_0_6B, 16, list(synth.WORKLOADS["qwen3-0.6b-b8-d16-p256to2048-g256"].prompt_lens), 256),
    ("qwen-d32", synth.QWEN3_0_6B, 32, [1024], 256),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("kind", [0, 1, 2])
@pytest.mark.parametrize("grid", [152, 37])
def test_schedule_is_deadlock_free(case, kind, grid):
    _, S, D, lens, G = case
    cfg = pbd.make_config(S, D, len(lens), max(lens) + G + 8)
    items, off = pbd.pbd_plan_pass(cfg, kind, lens, G, grid)
    slice_w = [256, 256, 512 if S.hidden % 512 == 0 else 256, 256]
    _check(S, items, off, grid, S.n_layers, slice_w)
    _check_counters(items, off, grid)
    op, lin, layer, a, b, c = _decode(items)
    rows = len(lens) * (1 if kind == 2 else D + 1)
    assert (op == OP_EMBED).sum() == rows
    assert (op == OP_FINAL).sum() == len(lens) * (1 if kind == 2 else (D if kind == 0 else D + 1))
    # the adapter tile exists in the draft only
    main = [(S.n_q_heads + 2 * S.n_kv_heads) * S.head_dim // TILE, S.hidden // TILE, 2 * S.intermediate // TILE,
            S.hidden // TILE]
    has_adapter = any(a[i] >= main[lin[i]] for i in np.nonzero(op == OP_LINEAR)[0])
    assert has_adapter == (kind == 0)


@pytest.mark.parametrize("E", [1, 14])
def test_early_exit_schedule(E):
    S = synth.QWEN3_0_6B
    cfg = pbd.make_config(S, 16, 1, 1024, draft_layers=E)
    items, off = pbd.pbd_plan_pass(cfg, 0, [512], 256, 152)
    _check(S, items, off, 152, E, [256, 256, 512, 256])
    _check_counters(items, off, 152)
    # the verify pass still runs every layer
    items_v, off_v = pbd.pbd_plan_pass(cfg, 1, [512], 256, 152)
    _check(S, items_v, off_v, 152, S.n_layers, [256, 256, 512, 256])


def test_plan_rejects_bad_arguments():
    S = synth.TINY
    cfg = pbd.make_config(S, 16, 1, 128)
    with pytest.raises(pbd.PbdError):
        pbd.pbd_plan_pass(cfg, 3, [64], 32, 152)
    with pytest.raises(pbd.PbdError):
        pbd.pbd_plan_pass(cfg, 1, [120], 32, 152)  # prompt + budget beyond max_seq_len
    with pytest.raises(pbd.PbdError):
        pbd.pbd_plan_pass(cfg, 1, [64], 32, 152, cap=10)


def _redeal(all_items, grid):
    """Deals a list in global order round-robin, as the builder does: (items by CTA, offsets)."""
    n = len(all_items)
    counts = np.bincount(np.arange(n) % grid, minlength=grid)
    off = np.concatenate([[0], np.cumsum(counts)])
    out = np.empty_like(all_items)
    fill = off[:-1].copy()
    for i in range(n):
        out[fill[i % grid]] = all_items[i]
        fill[i % grid] += 1
    return out, off


@pytest.mark.parametrize("mistake", ["target-low", "release-dropped", "wrong-counter"])
def test_counter_check_catches_planted_mistakes(mistake):
    S = synth.QWEN3_0_6B
    cfg = pbd.make_config(S, 16, 1, 1024)
    items, off = pbd.pbd_plan_pass(cfg, 1, [512], 256, 152)
    _check_counters(items, off, 152)
    bad = items.copy()
    op, lin, layer, a, b, c = _decode(bad)
    if mistake == "target-low":  # an o slice that would start one merge early
        i = int(np.nonzero((op == OP_LINEAR) & (lin == 1) & (layer == 3))[0][0])
        bad[i, 5] -= 1
    elif mistake == "release-dropped":  # a q|k|v reduction that never counts
        i = int(np.nonzero((op == OP_LINEAR) & (lin == 0) & (layer == 2) & (a == 0))[0][0])
        bad[i, 6] = -1
    else:  # a down reduction counting on the o counter
        i = int(np.nonzero((op == OP_LINEAR) & (lin == 3) & (layer == 5))[0][0])
        j = int(np.nonzero((op == OP_LINEAR) & (lin == 1) & (layer == 5))[0][0])
        bad[i, 6] = bad[j, 6]
    with pytest.raises(AssertionError):
        _check_counters(bad, off, 152)


@pytest.mark.parametrize("mistake", ["attention-before-qkv", "down-before-gate-up", "slices-apart"])
def test_check_catches_planted_mistakes(mistake):
    S = synth.TINY
    grid = 37
    cfg = pbd.make_config(S, 16, 1, 160)
    items, off = pbd.pbd_plan_pass(cfg, 1, [64], 32, grid)
    g = _global_order(off, grid, len(items))
    all_items = np.empty_like(items)
    all_items[g] = items
    _check(S, *_redeal(all_items, grid), grid, S.n_layers, [256, 256, 256, 256])  # the list as built passes
    op, lin, layer, a, b, c = _decode(all_items)
    bad = all_items.copy()
    if mistake == "attention-before-qkv":
        i = int(np.nonzero((op == OP_ATTN) & (layer == 1))[0][0])
        j = int(np.nonzero((op == OP_LINEAR) & (lin == 0) & (layer == 1))[0][-1])
        bad[[i, j]] = bad[[j, i]]
    elif mistake == "down-before-gate-up":
        i = int(np.nonzero((op == OP_LINEAR) & (lin == 3) & (layer == 0))[0][0])
        j = int(np.nonzero((op == OP_LINEAR) & (lin == 2) & (layer == 0))[0][-1])
        bad[[i, j]] = bad[[j, i]]
    else:  # the second K slice of a down tile moved to the end of its layer
        i = int(np.nonzero((op == OP_LINEAR) & (lin == 3) & (layer == 0) & (b == 1))[0][0])
        j = int(np.nonzero((op == OP_LINEAR) & (lin == 3) & (layer == 0))[0][-1])
        bad = np.concatenate([bad[:i], bad[i + 1:j + 1], bad[i:i + 1], bad[j + 1:]])
    with pytest.raises(AssertionError):
        _check(S, *_redeal(bad, grid), grid, S.n_layers, [256, 256, 256, 256])


def test_layer_skip_schedule():
    """A draft skipping layers: no item of a skipped layer, each kept layer's q|k|v waits for the
    previous kept layer's residual, the final norm for the last kept layer; counters consistent."""
    S = synth.QWEN3_0_6B
    skip = sum(1 << l for l in range(5, 24, 2))
    cfg = pbd.make_config(S, 16, 1, 1024, draft_skip=skip)
    items, off = pbd.pbd_plan_pass(cfg, 0, [512], 256, 152)
    _check_counters(items, off, 152)
    op, lin, layer, a, b, c = _decode(items)
    kept = [l for l in range(S.n_layers) if not (skip >> l) & 1]
    assert set(layer[op == OP_LINEAR]) == set(kept)
    assert set(layer[op == OP_FINAL]) == {kept[-1]}
    # the verify pass of the same context runs every layer
    items_v, off_v = pbd.pbd_plan_pass(cfg, 1, [512], 256, 152)
    _check(S, items_v, off_v, 152, S.n_layers, [256, 256, 512, 256])
    # a mask keeping no layer, or naming a layer beyond the model, is rejected
    for bad in ((1 << S.n_layers) - 1, 1 << S.n_layers):
        with pytest.raises(pbd.PbdError):
            pbd.pbd_plan_pass(pbd.make_config(S, 16, 1, 1024, draft_skip=bad), 0, [512], 256, 152)


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("grid", [152, 37])
def test_attention_items_cover_the_keys(case, grid):
    """Each (layer, sequence, KV group) has attention items 0..n-1 that together cover every
    128-key split a pass of the generation can reach.  A context whose full-length split items
    exceed one wave of CTAs keeps one partial result per split and lets an item cover two
    consecutive splits (n = ceil(splits / 2)); otherwise an item is one split."""
    _, S, D, lens, G = case
    max_len = max(lens) + G + 8
    cfg = pbd.make_config(S, D, len(lens), max_len)
    items, off = pbd.pbd_plan_pass(cfg, 1, lens, G, grid)
    op, lin, layer, a, b, c = _decode(items)
    max_tokens = max_len + 2 * (D + 1)
    n_splits = -(-max_tokens // 128)
    span = 2 if len(lens) * n_splits * S.n_kv_heads > grid else 1
    pages = -(-max_tokens // 16)
    att = {}
    for i in np.nonzero(op == OP_ATTN)[0]:
        att.setdefault((int(layer[i]), int(a[i]), int(b[i])), []).append(int(c[i]))
    assert len(att) == S.n_layers * len(lens) * S.n_kv_heads
    for (l, bl, g), cs in att.items():
        reach = min(lens[bl] + G + 2 * (D + 1), pages * 16)
        splits = min(n_splits, -(-reach // 128))
        assert sorted(cs) == list(range(-(-splits // span))), (l, bl, g, span, splits, sorted(cs))


@pytest.mark.parametrize("kind", [0, 1, 2])
def test_schedule_on_few_ctas(kind):
    """Four CTAs (the fewest the tiny model allows: its down projection has three K slices) and a
    1000-token prompt: many items per CTA, and more attention items per head group than CTAs (the
    last item merges them all, so they need not sit on distinct CTAs)."""
    S, grid, lens, G = synth.TINY, 4, [1000], 48
    cfg = pbd.make_config(S, 16, 1, lens[0] + G + 8, max_ctas=grid)
    items, off = pbd.pbd_plan_pass(cfg, kind, lens, G, grid)
    _check(S, items, off, grid, S.n_layers, [256, 256, 256, 256])
    _check_counters(items, off, grid)
