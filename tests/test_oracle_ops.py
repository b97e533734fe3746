"""Closed-form pins of the oracle's single steps (RMSNorm, RoPE, linear+LoRA, attention).

Each check compares with something other than the oracle's own formula: a closed
form, an invariant, a special case that reduces to a textbook result, or the merged
weight x (W + s B A)^T evaluated in float64.
"""
import ctypes as C
import math

import numpy as np
import pytest

import oracle
from oracle import model as om
from paper_2607_12422_gb300 import synth


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def _bf16_round(x):
    return synth.bf16_to_f32(synth.bf16_bits(_f32(x)))


def rmsnorm(x, g, eps=1e-6):
    x = _f32(x)
    n, dim = x.shape
    y = np.empty_like(x)
    om.lib().orc_op_rmsnorm(n, dim, om._fp(x), om._u16(np.ascontiguousarray(g)), eps, om._fp(y))
    return y


def rope(x, pos, theta=1e6):
    x = _f32(x).copy()
    om.lib().orc_op_rope(om._fp(x), x.shape[0], pos, theta)
    return x


# ---------------------------------------------------------------- RMSNorm

def test_rmsnorm_constant_vector_gives_gains():
    dim = 256
    g = synth.bf16_bits(np.linspace(0.5, 2.0, dim).astype(np.float32))
    for c in (0.25, 3.0, -7.5):
        y = rmsnorm(np.full((1, dim), c), g)
        # x / rms(x) = sign(c) * (1 - O(eps/c^2)); rounds to sign(c) in bf16
        assert np.array_equal(y[0], np.sign(c) * synth.bf16_to_f32(g))


def test_rmsnorm_scale_invariant_power_of_two():
    rng = np.random.default_rng(0)
    x = _bf16_round(rng.standard_normal((4, 1024)))
    g = np.full(1024, 0x3F80, dtype=np.uint16)
    y1 = rmsnorm(x, g)
    y2 = rmsnorm(x * 8.0, g)  # exact scaling; eps is negligible at this magnitude
    assert np.array_equal(y1, y2)
    # unit RMS after normalisation (bf16 output rounding only)
    rms = np.sqrt((y1.astype(np.float64) ** 2).mean(axis=1))
    assert np.allclose(rms, 1.0, atol=4e-3)


# ---------------------------------------------------------------- RoPE

def test_rope_position_zero_is_identity():
    rng = np.random.default_rng(1)
    x = _bf16_round(rng.standard_normal(128))
    assert np.array_equal(rope(x, 0), x)


def test_rope_basis_vector_closed_form():
    """e_i rotates into (cos a, sin a) on the pair (i, i+d/2), a = pos * theta^(-2i/d)."""
    d, theta = 128, 1e6
    for i in (0, 1, 17, 63):
        for pos in (1, 5, 300, 4000):
            x = np.zeros(d, dtype=np.float32)
            x[i] = 1.0
            y = rope(x, pos, theta)
            a = pos * theta ** (-2.0 * i / d)
            assert abs(y[i] - math.cos(a)) <= 2 ** -8 * max(1e-30, abs(math.cos(a))) + 1e-38
            assert abs(y[i + d // 2] - math.sin(a)) <= 2 ** -8 * abs(math.sin(a)) + 1e-38
            mask = np.ones(d, bool)
            mask[[i, i + d // 2]] = False
            assert not y[mask].any()
            # second half of the pair rotates the other way: e_{i+d/2} -> (-sin a, cos a)
            x2 = np.zeros(d, dtype=np.float32)
            x2[i + d // 2] = 1.0
            y2 = rope(x2, pos, theta)
            assert abs(y2[i] + math.sin(a)) <= 2 ** -8 * abs(math.sin(a)) + 1e-38


def test_rope_relative_position():
    """<R(m) q, R(n) k> depends only on m - n."""
    rng = np.random.default_rng(2)
    q = _bf16_round(rng.standard_normal(128))
    k = _bf16_round(rng.standard_normal(128))
    ref = float(np.dot(rope(q, 7).astype(np.float64), rope(k, 3).astype(np.float64)))
    for off in (10, 200, 1000):
        got = float(np.dot(rope(q, 7 + off).astype(np.float64), rope(k, 3 + off).astype(np.float64)))
        assert abs(got - ref) < 0.05 * (1 + abs(ref))
    # norm preserved up to bf16 rounding
    for pos in (1, 99, 3000):
        assert abs(np.linalg.norm(rope(q, pos)) - np.linalg.norm(q)) < 0.01 * np.linalg.norm(q)


# ---------------------------------------------------------------- linear + LoRA

def _linear(shape, x, W, A, B, on):
    cfg = om.make_config(shape)
    n, fin = x.shape
    fout = W.shape[0]
    y = np.empty((n, fout), dtype=np.float32)
    x = _f32(x)
    om.lib().orc_op_linear(C.byref(cfg), n, fin, fout, om._fp(x), om._u16(W), om._u16(A), om._u16(B), int(on),
                           om._fp(y))
    return y


def test_linear_lora_equals_merged_weight():
    S = synth.TINY
    rng = np.random.default_rng(3)
    fin, fout, r, s = 256, 192, S.lora_rank, S.lora_scale
    x = _bf16_round(rng.standard_normal((5, fin)))
    W = synth.bf16_bits(rng.standard_normal((fout, fin)).astype(np.float32) * 0.02)
    A = synth.bf16_bits(rng.standard_normal((r, fin)).astype(np.float32) * 0.02)
    B = synth.bf16_bits(rng.standard_normal((fout, r)).astype(np.float32) * 0.02)
    Wf, Af, Bf = (synth.bf16_to_f32(t).astype(np.float64) for t in (W, A, B))
    merged = x.astype(np.float64) @ (Wf + s * Bf @ Af).T
    plain = x.astype(np.float64) @ Wf.T
    y_on = _linear(S, x, W, A, B, True)
    y_off = _linear(S, x, W, A, B, False)
    # output rounding (2^-9 relative) plus the bf16 rounding of u = x A^T propagated through s*B
    u = x.astype(np.float64) @ Af.T
    tol_u = s * (np.abs(u) * 2 ** -8) @ np.abs(Bf).T
    assert np.all(np.abs(y_on - merged) <= np.abs(merged) * 2 ** -8 + tol_u + 1e-6)
    assert np.all(np.abs(y_off - plain) <= np.abs(plain) * 2 ** -8 + 1e-6)
    # the delta is far above rounding, so a dropped term or flipped sign cannot pass
    assert np.abs(merged - plain).mean() > 4 * (np.abs(merged) * 2 ** -8 + tol_u).mean()


# ---------------------------------------------------------------- attention

def _attention(shape, cache, L, n, mode, q):
    cfg = om.make_config(shape)
    out = np.empty((n, shape.n_q_heads * shape.head_dim), dtype=np.float32)
    q = _f32(q)
    om.lib().orc_op_attention(C.byref(cfg), 0, cache.ptr, L, n, mode, om._fp(q), om._fp(out))
    return out


@pytest.fixture(scope="module")
def attn_model(tiny):
    return tiny["model"]


def test_attention_zero_query_reveals_visible_set(attn_model):
    """q = 0 gives uniform weights, so with one-hot values the output is 1/|visible| on visible keys."""
    S = attn_model.shape
    d, Hkv, Hq = S.head_dim, S.n_kv_heads, S.n_q_heads
    L, D = 20, 8
    n = D + 1
    T = L + n
    assert T <= d
    cache = attn_model.new_cache(64)
    K = np.zeros((T, Hkv * d), np.float32)
    V = np.zeros((T, Hkv * d), np.float32)
    for t in range(T):
        for g in range(Hkv):
            V[t, g * d + t] = 1.0
    cache.write(0, 0, K, V)
    q = np.zeros((n, Hq * d), np.float32)
    for mode in (oracle.MASK_CAUSAL, oracle.MASK_BLOCK_DRAFT):
        out = _attention(S, cache, L, n, mode, q)
        for i in range(n):
            if mode == oracle.MASK_CAUSAL:
                vis = set(range(L + i + 1))
            elif i == 0:
                vis = set(range(L + 1))          # the pending row: cache and itself
            else:
                vis = set(range(L + n))          # a mask row: cache, pending row, whole mask block
            for h in range(Hq):
                row = out[i, h * d:(h + 1) * d]
                got = set(np.nonzero(row)[0].tolist())
                assert got == vis, (mode, i, h)
                assert np.allclose(row[list(vis)], 1.0 / len(vis), rtol=2 ** -8)


def test_attention_gqa_head_mapping(attn_model):
    """With V constant per KV head, query head h returns the constant of KV head h // (Hq/Hkv)."""
    S = attn_model.shape
    d, Hkv, Hq = S.head_dim, S.n_kv_heads, S.n_q_heads
    L, n = 33, 5
    rng = np.random.default_rng(4)
    cache = attn_model.new_cache(64)
    K = _bf16_round(rng.standard_normal((L + n, Hkv * d)))
    V = np.zeros((L + n, Hkv * d), np.float32)
    for g in range(Hkv):
        V[:, g * d:(g + 1) * d] = g + 1.0
    cache.write(0, 0, K, V)
    q = _bf16_round(rng.standard_normal((n, Hq * d)))
    out = _attention(S, cache, L, n, oracle.MASK_CAUSAL, q)
    for h in range(Hq):
        assert np.all(out[:, h * d:(h + 1) * d] == h // (Hq // Hkv) + 1.0)


def test_attention_single_visible_key_returns_its_value(attn_model):
    """Row 0 of a prompt at L = 0 sees one key: softmax is exactly 1 and the output is v_0."""
    S = attn_model.shape
    d, Hkv, Hq = S.head_dim, S.n_kv_heads, S.n_q_heads
    rng = np.random.default_rng(5)
    cache = attn_model.new_cache(16)
    K = _bf16_round(rng.standard_normal((4, Hkv * d)))
    V = _bf16_round(rng.standard_normal((4, Hkv * d)))
    cache.write(0, 0, K, V)
    q = _bf16_round(rng.standard_normal((4, Hq * d)) * 3)
    out = _attention(S, cache, 0, 4, oracle.MASK_CAUSAL, q)
    for h in range(Hq):
        g = h // (Hq // Hkv)
        assert np.array_equal(out[0, h * d:(h + 1) * d], V[0, g * d:(g + 1) * d])


class _AttnShape:
    """The fields the oracle's config and cache need, for attention-only pins at any (d, Hq, Hkv)."""

    def __init__(self, d, hq, hkv):
        self.n_layers, self.hidden, self.n_q_heads, self.n_kv_heads, self.head_dim = 1, hq * d, hq, hkv, d
        self.intermediate, self.vocab, self.rms_eps, self.rope_theta = 4 * d, 16, 1e-6, 1e6
        self.lora_rank, self.lora_alpha = 8, 16.0


class _AttnHolder:
    def __init__(self, shape):
        self.shape, self.cfg = shape, om.make_config(shape)


def _visible(mode, L, n, i):
    """Key positions row i of an n-row block at L may read, written out from the masks' definitions
    (Section 3 and Appendix A.4): causal rows see every earlier position and themselves; under the
    draft mask the pending row (i = 0) sees the cache and itself, a mask row the whole block."""
    if mode == oracle.MASK_CAUSAL or i == 0:
        return list(range(L + i + 1))
    return list(range(L + n))


@pytest.mark.parametrize("d,hq,hkv", [(64, 4, 2), (128, 16, 8), (32, 3, 1), (64, 6, 3)])
@pytest.mark.parametrize("offset", [0.0, 100.0])
def test_attention_weights_follow_exp_of_scaled_scores(d, hq, hkv, offset):
    """Scores built as s_k = offset + ln(w_k) with integer w_k make the softmax weights exactly
    w_k / sum(w) over the visible keys, so every output is a known mixture of the values.

    Query head h is c * e_{j(h)} and key k of KV group g is sum_j a_{k,j} e_j with
    a_{k,j} = sqrt(d) (offset + ln w[g][k][j]) / c: the score q.k / sqrt(d) is offset + ln w.
    A scale of 1/d or none, a wrong exponent base, a wrong query-head to KV-group map or a
    masked key taken in changes the mixture; at offset 100 the scores overflow exp in fp32
    unless the row maximum is subtracted first (exp(100) > 3.4e38), so a softmax without the
    max shift returns NaN.  Values are bf16 numbers; the output is rounded once to bf16."""
    S = _AttnShape(d, hq, hkv)
    holder = _AttnHolder(S)
    grp = hq // hkv
    L, D = 5, 3
    n = D + 1
    T = L + n
    rng = np.random.default_rng(100 + d + hq)
    # weights 1..9 per (group, key, query column j); query head h uses column j(h) = h % grp
    w = rng.integers(1, 10, size=(hkv, T, grp)).astype(np.float64)
    c = 4.0
    K = np.zeros((T, hkv * d), np.float64)
    for g in range(hkv):
        for k in range(T):
            for j in range(grp):
                K[k, g * d + j] = math.sqrt(d) * (offset + math.log(w[g, k, j])) / c
    V = _bf16_round(rng.standard_normal((T, hkv * d)))
    cache = om.OracleCache(holder, T)
    cache.write(0, 0, K.astype(np.float32), V)
    q = np.zeros((n, hq * d), np.float32)
    for h in range(hq):
        q[:, h * d + h % grp] = c
    for mode in (oracle.MASK_CAUSAL, oracle.MASK_BLOCK_DRAFT):
        out = _attention(S, cache, L, n, mode, q)
        assert np.all(np.isfinite(out)), (mode, offset)
        for i in range(n):
            vis = _visible(mode, L, n, i)
            for h in range(hq):
                g = h // grp
                wk = w[g, vis, h % grp]
                ref = (wk[:, None] * V[vis, g * d:(g + 1) * d].astype(np.float64)).sum(0) / wk.sum()
                got = out[i, h * d:(h + 1) * d].astype(np.float64)
                # bf16 rounding of the output (2^-9 relative) plus the fp32 scores' relative error
                # (~1e-7 of |s| <= 103) carried through exp
                assert np.allclose(got, ref, rtol=2 ** -8, atol=2 ** -8 * np.abs(ref).max() + 1e-6), (mode, i, h)


def test_attention_two_keys_three_to_one():
    """Two visible keys, scores 0 and ln 3: weights 1/4 and 3/4, output v0/4 + 3 v1/4 (the row at
    position 1 of a prompt, causal).  A 1/d scale would give weights 0.466 / 0.534 at d = 64."""
    S = _AttnShape(64, 2, 1)
    holder = _AttnHolder(S)
    cache = om.OracleCache(holder, 4)
    d = 64
    K = np.zeros((2, d), np.float32)
    K[1, 0] = math.sqrt(d) * math.log(3.0) / 2.0
    V = np.zeros((2, d), np.float32)
    V[0, :] = 1.0
    V[1, :] = 2.0
    cache.write(0, 0, K, V)
    q = np.zeros((2, 2 * d), np.float32)
    q[:, 0] = 2.0
    q[:, d] = 2.0
    out = _attention(S, cache, 0, 2, oracle.MASK_CAUSAL, q)
    # row 1 mixes 1.0 and 2.0 with weights 1/4, 3/4 = 1.75 exactly (a bf16 number)
    assert np.allclose(out[1], 1.75, rtol=0, atol=2 ** -7)
    assert np.all(out[0] == 1.0)


# ---------------------------------------------------------------- SwiGLU

def _swiglu(g, u):
    g, u = _f32(g), _f32(u)
    out = np.empty_like(g)
    om.lib().orc_op_swiglu(g.size, om._fp(g), om._fp(u), om._fp(out))
    return out


def test_swiglu_closed_forms():
    """silu(x) - silu(-x) = x;  silu(0) = 0;  silu(x) -> x and silu(-x) -> 0 for large x;  linear in u."""
    rng = np.random.default_rng(6)
    x = _bf16_round(rng.standard_normal(4096) * 3)
    one = np.ones_like(x)
    a, b = _swiglu(x, one), _swiglu(-x, one)
    assert np.allclose(a - b, x, rtol=0, atol=2 ** -7 * np.abs(x).max() + 1e-6)
    assert np.all(_swiglu(np.zeros(8), np.full(8, 5.0)) == 0)
    big = np.array([40.0, 80.0], np.float32)
    assert np.array_equal(_swiglu(big, np.ones(2)), big)
    assert np.all(np.abs(_swiglu(-big, np.ones(2))) < 1e-12)
    # the product with the up projection: scaling u by 4 scales the output by 4 exactly
    assert np.array_equal(_swiglu(x, one * 4.0), 4.0 * a)


# ---------------------------------------------------------------- whole model, special case

def test_zero_block_weights_reduce_to_embedding_readout(tiny):
    """With every block linear zero, each layer adds exactly 0 to the residual stream, so the
    logits are final_norm(e_t) . E^T for the input token t (tied head), computed here in fp64."""
    S = tiny["shape"]
    base = dict(tiny["base"])
    for n in synth.LINEARS:
        base["w" + n] = np.zeros_like(base["w" + n])
    m = oracle.OracleModel(S, base, tiny["adapter"])
    toks = [5, 77, 4000, 1234]
    cache = m.new_cache(16)
    am, lg, _ = m.forward(cache, 0, toks, False, oracle.MASK_CAUSAL, 0, 4, want_logits=True)
    E = synth.bf16_to_f32(base["embed"]).astype(np.float64)
    for i, t in enumerate(toks):
        e = E[t]
        xn = e / np.sqrt((e * e).mean() + 1e-6)
        ref = E @ xn
        assert np.allclose(lg[i], ref, atol=0.02 * np.abs(ref).max())
        assert am[i] == t  # the tied head reads the token back
