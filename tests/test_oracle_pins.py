"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these compares the oracle with itself: each check is a closed form,
an invariant, a special case that reduces to a textbook computation done
with library routines (numpy / scipy), brute force on tiny inputs, or a
number printed in the paper (tests/golden/).
"""
import json
import math
import os

import numpy as np
import pytest
import scipy.special

from oracle import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rnd(rng, *shape, scale=1.0):
    return (rng.standard_normal(shape) * scale).astype(np.float32)


def rms(x):
    x = np.asarray(x, dtype=np.float64)
    return np.linalg.norm(x) / math.sqrt(x.size)


def rope_complex(y, pos, theta):
    """RoPE written as a complex rotation: (y_i + i y_{i+d/2}) * exp(i pos w_i)."""
    y = np.asarray(y, dtype=np.float64)
    h = y.size // 2
    w = np.float64(theta) ** (-np.arange(h) * 2.0 / y.size)
    z = (y[:h] + 1j * y[h:]) * np.exp(1j * pos * w)
    return np.concatenate([z.real, z.imag])


def make_paged(rng, kch, seq_lens, Hkv, d, P, permute, dtype=np.float32):
    npg = [-(-s // P) for s in seq_lens]
    num_pages = sum(npg)
    phys = rng.permutation(num_pages) if permute else np.arange(num_pages)
    pt = np.full((len(seq_lens), max(npg)), -1, dtype=np.int32)
    o = 0
    for b, n in enumerate(npg):
        pt[b, :n] = phys[o:o + n]
        o += n
    kp = rnd(rng, kch, num_pages, Hkv, P, d)
    vp = rnd(rng, kch, num_pages, Hkv, P, d)
    return kp, vp, pt


def gather(pool, chan, pt, b, hkv, S, P):
    """Logical slots 0..S-1 of (sequence b, kv head) from the documented layout."""
    return np.stack([pool[chan, pt[b, t // P], hkv, t % P] for t in range(S)]).astype(np.float64)


# ----------------------------------------------------------------- attention

@pytest.mark.parametrize("Hq,Hkv,d,P,permute", [
    (4, 4, 8, 4, False), (4, 2, 16, 8, True), (6, 3, 12, 4, True), (2, 1, 8, 16, True)])
def test_attention_matches_brute_force_softmax(Hq, Hkv, d, P, permute):
    rng = np.random.default_rng(Hq * 100 + d)
    seq_lens = [1, 7, 23, 16]
    kp, vp, pt = make_paged(rng, 3, seq_lens, Hkv, d, P, permute)
    q = rnd(rng, len(seq_lens), Hq, d)
    chan = 1
    out = O.decode_attn(q, kp, vp, pt, seq_lens, chan=chan, Hq=Hq, Hkv=Hkv, d=d, P=P)
    for b, S in enumerate(seq_lens):
        for hq in range(Hq):
            hkv = hq // (Hq // Hkv)
            K = gather(kp, chan, pt, b, hkv, S, P)
            V = gather(vp, chan, pt, b, hkv, S, P)
            ref = scipy.special.softmax(K @ q[b, hq].astype(np.float64) / math.sqrt(d)) @ V
            np.testing.assert_allclose(out[b, hq], ref, rtol=0, atol=1e-12)


def test_attention_dummy_only_returns_dummy_value():
    rng = np.random.default_rng(1)
    kp, vp, pt = make_paged(rng, 2, [1, 1], 2, 8, 4, True)
    q = rnd(rng, 2, 2, 8, scale=5.0)
    out = O.decode_attn(q, kp, vp, pt, [1, 1], chan=1, Hq=2, Hkv=2, d=8, P=4)
    for b in range(2):
        for h in range(2):
            assert np.array_equal(out[b, h], vp[1, pt[b, 0], h, 0].astype(np.float64))


def test_attention_equal_keys_give_mean_value():
    rng = np.random.default_rng(2)
    S, P, d = 37, 8, 16
    kp, vp, pt = make_paged(rng, 1, [S], 1, d, P, True)
    kp[:] = rnd(rng, d)  # every slot holds the same key
    q = rnd(rng, 1, 1, d, scale=3.0)
    out = O.decode_attn(q, kp, vp, pt, [S], chan=0, Hq=1, Hkv=1, d=d, P=P)
    V = gather(vp, 0, pt, 0, 0, S, P)
    np.testing.assert_allclose(out[0, 0], V.mean(axis=0), rtol=0, atol=1e-13)


def test_attention_planted_key_dominates():
    rng = np.random.default_rng(3)
    S, P, d, t_star = 50, 16, 32, 29
    kp, vp, pt = make_paged(rng, 1, [S], 1, d, P, True)
    q = rnd(rng, 1, 1, d)
    qq = q[0, 0].astype(np.float64)
    kp[:] = 0.0
    kp[0, pt[0, t_star // P], 0, t_star % P] = (qq * 40.0 * math.sqrt(d) / qq.dot(qq)).astype(np.float32)
    out = O.decode_attn(q, kp, vp, pt, [S], chan=0, Hq=1, Hkv=1, d=d, P=P)
    want = vp[0, pt[0, t_star // P], 0, t_star % P].astype(np.float64)
    np.testing.assert_allclose(out[0, 0], want, rtol=0, atol=1e-12 * (1 + np.abs(want).max()))


def test_attention_ignores_slots_beyond_length_and_page_permutation():
    rng = np.random.default_rng(4)
    seq_lens, P, d = [13, 29], 8, 16
    kp, vp, pt = make_paged(rng, 2, seq_lens, 2, d, P, False)
    q = rnd(rng, 2, 2, d)
    base = O.decode_attn(q, kp, vp, pt, seq_lens, chan=1, Hq=2, Hkv=2, d=d, P=P)
    # poison every slot at or beyond the length in the last page of each sequence
    kp2, vp2 = kp.copy(), vp.copy()
    for b, S in enumerate(seq_lens):
        pg = pt[b, (S - 1) // P]
        kp2[:, pg, :, S % P or P:, :] = np.nan
        vp2[:, pg, :, S % P or P:, :] = np.nan
    poisoned = O.decode_attn(q, kp2, vp2, pt, seq_lens, chan=1, Hq=2, Hkv=2, d=d, P=P)
    assert np.array_equal(base, poisoned)
    # move the pages to a random physical permutation: identical result
    perm = rng.permutation(kp.shape[1])
    kp3 = np.empty_like(kp)
    vp3 = np.empty_like(vp)
    kp3[:, perm] = kp
    vp3[:, perm] = vp
    pt3 = np.where(pt >= 0, perm[np.maximum(pt, 0)], -1).astype(np.int32)
    moved = O.decode_attn(q, kp3, vp3, pt3, seq_lens, chan=1, Hq=2, Hkv=2, d=d, P=P)
    assert np.array_equal(base, moved)


def test_attention_reads_bf16_inputs_as_their_values():
    from wm_synth import gen
    rng = np.random.default_rng(5)
    kp, vp, pt = make_paged(rng, 1, [20], 2, 8, 4, True)
    q = rnd(rng, 1, 2, 8)
    kb, vb, qb = (gen.f32_to_bf16_bits(a) for a in (kp, vp, q))
    out_b = O.decode_attn(qb, kb, vb, pt, [20], chan=0, Hq=2, Hkv=2, d=8, P=4)
    widened = [gen.bf16_bits_to_f32(a) for a in (qb, kb, vb)]
    out_f = O.decode_attn(widened[0], widened[1], widened[2], pt, [20], chan=0, Hq=2, Hkv=2,
                          d=8, P=4)
    assert np.array_equal(out_b, out_f)


def test_attention_rejects_bad_page_ids():
    rng = np.random.default_rng(6)
    kp, vp, pt = make_paged(rng, 1, [9], 1, 8, 4, False)
    pt[0, 1] = kp.shape[1]  # one past the pool
    with pytest.raises(IndexError):
        O.decode_attn(rnd(rng, 1, 1, 8), kp, vp, pt, [9], chan=0, Hq=1, Hkv=1, d=8, P=4)


# ---------------------------------------------------------------- RMSNorm/RoPE

# ----------------------------------------------------- prefill attention (Sec. 3.2-3.3)

def _prefill_case(rng, T, B, Hq, Hkv, d, P, permute):
    """Channel caches holding the dummy and T tokens (slots 0..T) per sequence."""
    kp, vp, pt = make_paged(rng, 2, [T + 1] * B, Hkv, d, P, permute)
    return kp, vp, pt


@pytest.mark.parametrize("Hq,Hkv,d,P,permute", [(4, 2, 8, 4, True), (2, 2, 16, 8, False),
                                                (6, 3, 12, 16, True)])
def test_prefill_matches_dense_masked_softmax(Hq, Hkv, d, P, permute):
    """Sec. 3.2: causal SDPA over the dummy-offset cache, written as one dense
    score matrix per head with the mask slot > position set to -inf."""
    rng = np.random.default_rng(100 + d)
    T, B = 37, 2
    kp, vp, pt = _prefill_case(rng, T, B, Hq, Hkv, d, P, permute)
    # rows at arbitrary positions (unsorted, repeated): any set of positions is one call
    pos = np.stack([rng.permutation(T)[:20], rng.integers(0, T, 20)]).astype(np.int32)
    q = rnd(rng, B, 20, Hq, d)
    chan = 1
    out = O.prefill_attn(q, kp, vp, pt, pos, chan=chan, Hq=Hq, Hkv=Hkv, d=d, P=P)
    slots = np.arange(T + 1)
    for b in range(B):
        for hq in range(Hq):
            hkv = hq // (Hq // Hkv)
            K = gather(kp, chan, pt, b, hkv, T + 1, P)
            V = gather(vp, chan, pt, b, hkv, T + 1, P)
            S = q[b, :, hq].astype(np.float64) @ K.T / math.sqrt(d)      # [rows][slots]
            S = np.where(slots[None, :] <= pos[b][:, None], S, -np.inf)
            ref = scipy.special.softmax(S, axis=1) @ V
            np.testing.assert_allclose(out[b, :, hq], ref, rtol=0, atol=1e-12)


def test_prefill_position_zero_reads_only_the_dummy():
    rng = np.random.default_rng(101)
    kp, vp, pt = _prefill_case(rng, 9, 1, 2, 2, 8, 4, True)
    q = rnd(rng, 1, 3, 2, 8, scale=5.0)
    pos = np.zeros((1, 3), dtype=np.int32)
    out = O.prefill_attn(q, kp, vp, pt, pos, chan=0, Hq=2, Hkv=2, d=8, P=4)
    for r in range(3):
        for h in range(2):
            assert np.array_equal(out[0, r, h], vp[0, pt[0, 0], h, 0].astype(np.float64))


def test_prefill_never_reads_the_queries_own_slot():
    """Sec. 3.2: the token at position i must not read slot i + 1 (its own
    channels).  A key planted there with a huge logit changes nothing; the
    same key one slot earlier (slot i, the previous token) dominates."""
    rng = np.random.default_rng(102)
    T, P, d, i = 40, 8, 16, 23
    kp, vp, pt = _prefill_case(rng, T, 1, 1, 1, d, P, True)
    q = rnd(rng, 1, 1, 1, d)
    qq = q[0, 0, 0].astype(np.float64)
    big = (qq * 40.0 * math.sqrt(d) / qq.dot(qq)).astype(np.float32)
    pos = np.array([[i]], dtype=np.int32)
    base = O.prefill_attn(q, kp, vp, pt, pos, chan=0, Hq=1, Hkv=1, d=d, P=P)
    own = kp.copy()
    own[0, pt[0, (i + 1) // P], 0, (i + 1) % P] = big
    assert np.array_equal(O.prefill_attn(q, own, vp, pt, pos, chan=0, Hq=1, Hkv=1, d=d, P=P), base)
    prev = kp.copy()
    prev[0, pt[0, i // P], 0, i % P] = big
    got = O.prefill_attn(q, prev, vp, pt, pos, chan=0, Hq=1, Hkv=1, d=d, P=P)[0, 0, 0]
    want = vp[0, pt[0, i // P], 0, i % P].astype(np.float64)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12 * (1 + np.abs(want).max()))


def test_prefill_row_equals_decode_of_the_same_token():
    """The token at position i decodes with i + 1 cache slots (Sec. 3.2): one
    prefill row and one decode step of that token give the same output."""
    rng = np.random.default_rng(103)
    T, B, Hq, Hkv, d, P = 30, 3, 4, 2, 8, 4
    kp, vp, pt = _prefill_case(rng, T, B, Hq, Hkv, d, P, True)
    pos = np.array([[0, 5, 29], [17, 3, 11], [29, 28, 1]], dtype=np.int32)
    q = rnd(rng, B, 3, Hq, d)
    out = O.prefill_attn(q, kp, vp, pt, pos, chan=1, Hq=Hq, Hkv=Hkv, d=d, P=P)
    for r in range(3):
        dec = O.decode_attn(q[:, r], kp, vp, pt, pos[:, r] + 1, chan=1, Hq=Hq, Hkv=Hkv, d=d, P=P)
        np.testing.assert_allclose(out[:, r], dec, rtol=0, atol=1e-13)


def test_prefill_rejects_positions_beyond_the_table():
    rng = np.random.default_rng(104)
    kp, vp, pt = _prefill_case(rng, 7, 1, 1, 1, 8, 4, False)
    q = rnd(rng, 1, 1, 1, 8)
    with pytest.raises(IndexError):
        O.prefill_attn(q, kp, vp, pt, np.array([[8]], np.int32), chan=0, Hq=1, Hkv=1, d=8, P=4)
    with pytest.raises(IndexError):
        O.prefill_attn(q, kp, vp, pt, np.array([[-1]], np.int32), chan=0, Hq=1, Hkv=1, d=8, P=4)


def test_rmsnorm_unit_rms_scale_invariance_and_gain():
    rng = np.random.default_rng(7)
    x = rng.standard_normal(96) * 3.7
    y = O.rmsnorm(x, 0.0)
    assert abs(rms(y) - 1.0) < 1e-14
    np.testing.assert_allclose(O.rmsnorm(x * 123.0, 0.0), y, rtol=1e-14, atol=0)
    g = rng.uniform(0.5, 2.0, 96)
    np.testing.assert_allclose(O.rmsnorm(x, 0.0, g) / g, y, rtol=1e-14, atol=0)
    # eps enters as mean(x^2) + eps
    ye = O.rmsnorm(x, 0.5)
    assert abs(rms(ye) - rms(x) / math.sqrt(rms(x) ** 2 + 0.5)) < 1e-14


@pytest.mark.parametrize("d,pos", [(8, 0), (16, 1), (64, 777), (128, 131071)])
def test_rope_is_the_complex_rotation(d, pos):
    rng = np.random.default_rng(d + pos)
    y = rng.standard_normal(d)
    got = O.rope(y, pos, 1e6)
    # the fp64 angle pos * w carries a rounding error of about pos * 2**-53
    atol = 1e-13 + 4e-16 * pos * np.abs(y).max()
    np.testing.assert_allclose(got, rope_complex(y, pos, 1e6), rtol=0, atol=atol)
    h = d // 2
    np.testing.assert_allclose(got[:h] ** 2 + got[h:] ** 2, y[:h] ** 2 + y[h:] ** 2, rtol=1e-13)
    if pos == 0:
        assert np.array_equal(got, y)


def test_rope_logits_depend_only_on_relative_position():
    rng = np.random.default_rng(8)
    d = 64
    q, k = rng.standard_normal(d), rng.standard_normal(d)
    base = O.rope(q, 100, 1e6).dot(O.rope(k, 37, 1e6))
    for shift in (1, 1000, 60000):
        s = O.rope(q, 100 + shift, 1e6).dot(O.rope(k, 37 + shift, 1e6))
        assert abs(s - base) < 1e-9


# ------------------------------------------------------------------- router

def route_inputs(rng, L, k, D, p):
    Lp = -(-L // p)
    h = rnd(rng, L, D)
    pre_g = np.ones((2, D), np.float32)
    Wr = rnd(rng, 2, k * L, Lp * D, scale=1.0 / math.sqrt(Lp * D))
    br = rnd(rng, 2, k * L)
    return h, pre_g, Wr, br


@pytest.mark.parametrize("L,k,p", [(4, 2, 2), (5, 3, 2), (7, 7, 3), (6, 1, 1)])
def test_router_zero_weights_gives_bias_reshaped_row_major(L, k, p):
    rng = np.random.default_rng(L * 10 + k)
    D = 16
    h, pre_g, Wr, br = route_inputs(rng, L, k, D, p)
    Wr[:] = 0
    hhat, alpha, _ = O.pool_route(h, pre_g, Wr, br, L=L, k=k, D=D, p=p, eps=1e-6)
    for X in range(2):
        assert np.array_equal(alpha[X], br[X].astype(np.float64).reshape(k, L))
        for l in range(L):
            assert abs(rms(hhat[X, l]) - 1.0) < 1e-5


@pytest.mark.parametrize("L,k,p", [(4, 2, 2), (5, 3, 2), (7, 2, 3)])
def test_router_reads_every_pth_layer_counting_down(L, k, p):
    """One non-zero router weight at (output o, input c) moves alpha[o // L][o % L]
    by exactly the normed state of layer L-1-(c // D)*p at element c % D."""
    rng = np.random.default_rng(11 + L)
    D = 8
    Lp = -(-L // p)
    h, pre_g, Wr, br = route_inputs(rng, L, k, D, p)
    for X in range(2):
        for o, c in [(0, 0), (k * L - 1, Lp * D - 1), (L + 1, D + 3), (k * L // 2, (Lp - 1) * D)]:
            W = np.zeros_like(Wr)
            W[X, o, c] = 1.0
            hhat, alpha, _ = O.pool_route(h, pre_g, W, br, L=L, k=k, D=D, p=p, eps=0.0)
            want = br.astype(np.float64).reshape(2, k, L).copy()
            layer = L - 1 - (c // D) * p
            want[X, o // L, o % L] += hhat[X, layer, c % D]
            assert np.array_equal(alpha, want)
            # the normed state itself: unit RMS, direction of h_layer
            hh = h[layer].astype(np.float64)
            np.testing.assert_allclose(hhat[X, layer], hh / rms(hh), rtol=1e-13)


def test_router_scale_invariance_and_gain():
    rng = np.random.default_rng(12)
    L, k, D, p = 6, 3, 32, 2
    h, pre_g, Wr, br = route_inputs(rng, L, k, D, p)
    _, a0, _ = O.pool_route(h, pre_g, Wr, br, L=L, k=k, D=D, p=p, eps=0.0)
    hs = (h * (1.0 + 0.1 * np.arange(L))[:, None] * 4).astype(np.float32)
    _, a1, _ = O.pool_route(hs, pre_g, Wr, br, L=L, k=k, D=D, p=p, eps=0.0)
    np.testing.assert_allclose(a1, a0, rtol=1e-6, atol=1e-6)  # inputs rounded to fp32
    g = rng.uniform(0.5, 1.5, (2, D)).astype(np.float32)
    hhat_g, _, _ = O.pool_route(h, g, Wr, br, L=L, k=k, D=D, p=p, eps=0.0)
    hhat_1, _, _ = O.pool_route(h, pre_g, Wr, br, L=L, k=k, D=D, p=p, eps=0.0)
    np.testing.assert_allclose(hhat_g, hhat_1 * g[:, None, :], rtol=1e-14)


# ------------------------------------------------------------------ channel

def test_channel_mix_is_linear_and_matches_sum_of_states():
    rng = np.random.default_rng(13)
    L, D, Hkv, d = 5, 32, 2, 8
    hhat = rng.standard_normal((L, D))
    W = rnd(rng, Hkv * d, D, scale=0.2)
    g = np.ones(D, np.float32)
    qg = np.ones(d, np.float32)
    kw = dict(is_key=False, pos=0, Hkv=Hkv, d=d, eps=1e-6, eps_qk=1e-6, theta=1e6)
    a1, a2 = rng.standard_normal(L), rng.standard_normal(L)
    t1, _, _ = O.pool_channel(hhat, a1, g, W, qg, **kw)
    t2, _, _ = O.pool_channel(hhat, a2, g, W, qg, **kw)
    t12, _, _ = O.pool_channel(hhat, a1 + a2, g, W, qg, **kw)
    np.testing.assert_allclose(t12, t1 + t2, rtol=0, atol=1e-13)
    onehot = np.array([1.0, 0, 1.0, 0, 1.0])  # cyclic assignment l -> l mod 2, channel 0
    t, _, _ = O.pool_channel(hhat, onehot, g, W, qg, **kw)
    np.testing.assert_allclose(t, hhat[0] + hhat[2] + hhat[4], rtol=0, atol=1e-14)


def test_value_branch_is_projection_of_normed_channel():
    rng = np.random.default_rng(14)
    L, D, Hkv, d = 3, 24, 3, 8
    hhat = rng.standard_normal((L, D))
    alpha = rng.standard_normal(L)
    W = rnd(rng, Hkv * d, D, scale=0.2)
    g = rng.uniform(0.5, 1.5, D).astype(np.float32)
    ht, out, macs = O.pool_channel(hhat, alpha, g, W, np.ones(d, np.float32), is_key=False,
                                   pos=5, Hkv=Hkv, d=d, eps=0.0, eps_qk=0.0, theta=1e6)
    x = ht / rms(ht) * g.astype(np.float64)
    np.testing.assert_allclose(out, W.astype(np.float64) @ x, rtol=1e-12, atol=1e-13)
    assert macs == (L * D, Hkv * d * D)


def test_key_branch_heads_are_qknormed_then_rotated():
    rng = np.random.default_rng(15)
    L, D, Hkv, d, pos = 3, 24, 3, 8, 41
    hhat = rng.standard_normal((L, D))
    alpha = rng.standard_normal(L)
    W = rnd(rng, Hkv * d, D, scale=0.2)
    g = np.ones(D, np.float32)
    qg = rng.uniform(0.5, 1.5, d).astype(np.float32)
    _, vout, _ = O.pool_channel(hhat, alpha, g, W, qg, is_key=False, pos=pos, Hkv=Hkv, d=d,
                                eps=0.0, eps_qk=0.0, theta=1e6)
    _, kout, _ = O.pool_channel(hhat, alpha, g, W, qg, is_key=True, pos=pos, Hkv=Hkv, d=d,
                                eps=0.0, eps_qk=0.0, theta=1e6)
    for hh in range(Hkv):
        raw = vout[hh * d:(hh + 1) * d]
        want = rope_complex(raw / rms(raw) * qg.astype(np.float64), pos, 1e6)
        np.testing.assert_allclose(kout[hh * d:(hh + 1) * d], want, rtol=0, atol=1e-12)


# ---------------------------------------------------------- vanilla reduction

def vanilla_kv(h_l, WK, WV, pos, D, Hkv, d):
    """A standard per-layer Qwen3-style KV: RMSNorm, projection, per-head
    key norm, RoPE on keys (library routines, no oracle code)."""
    x = h_l / rms(h_l)
    K = (WK @ x).reshape(Hkv, d)
    V = (WV @ x).reshape(Hkv, d)
    K = np.stack([rope_complex(kh / rms(kh), pos, 1e6) for kh in K])
    return K, V


@pytest.mark.parametrize("eps,tol", [(0.0, 1e-11), (1e-6, 3e-6)])
def test_identity_routing_reduces_to_vanilla_per_layer_kv_and_attention(eps, tol):
    """k = L, c(l) = l, zero router weights and alpha = identity: channel j
    holds exactly the vanilla layer-j KV, and layer l's decode attention over
    it is vanilla SDPA."""
    rng = np.random.default_rng(16)
    B, L, D, Hkv, d, P, S = 2, 4, 32, 2, 8, 4, 9
    k = L
    Lp = -(-L // 2)
    h = rnd(rng, B, L, D)
    ones = lambda *s: np.ones(s, np.float32)
    Wr = np.zeros((2, k * L, Lp * D), np.float32)
    br = np.stack([np.eye(k, L, dtype=np.float32).reshape(-1)] * 2)
    Wkv = rnd(rng, 2, k, Hkv * d, D, scale=1 / math.sqrt(D))
    pos = np.array([S - 1, S - 1], dtype=np.float64)
    K, V, alpha, _ = O.kv_mix(h, pos, ones(2, D), Wr, br, ones(2, k, D), Wkv, ones(k, d),
                              L=L, k=k, D=D, Hkv=Hkv, d=d, p=2, eps=eps, eps_qk=eps, theta=1e6)
    assert np.array_equal(alpha[0, 0], np.eye(k, L))
    for b in range(B):
        for j in range(k):
            Kv, Vv = vanilla_kv(h[b, j].astype(np.float64), Wkv[0, j].astype(np.float64),
                                Wkv[1, j].astype(np.float64), S - 1, D, Hkv, d)
            np.testing.assert_allclose(K[b, j], Kv, rtol=0, atol=tol * np.abs(Kv).max())
            np.testing.assert_allclose(V[b, j], Vv, rtol=0, atol=tol * np.abs(Vv).max())
    # decode attention of layer l over channel l == vanilla SDPA of layer l
    kp, vp, pt = make_paged(rng, k, [S] * B, Hkv, d, P, True)
    q = rnd(rng, B, Hkv, d)
    for l in range(L):
        out = O.decode_attn(q, kp, vp, pt, [S] * B, chan=l, Hq=Hkv, Hkv=Hkv, d=d, P=P)
        for b in range(B):
            for hh in range(Hkv):
                Kl = gather(kp, l, pt, b, hh, S, P)
                Vl = gather(vp, l, pt, b, hh, S, P)
                s = Kl @ q[b, hh].astype(np.float64) / math.sqrt(d)
                ref = np.exp(s - s.max()) @ Vl / np.exp(s - s.max()).sum()
                np.testing.assert_allclose(out[b, hh], ref, rtol=0, atol=1e-12)


def test_pool_is_invariant_to_per_layer_scale_of_states():
    rng = np.random.default_rng(17)
    B, L, k, D, Hkv, d = 2, 6, 3, 32, 2, 8
    Lp = 3
    h = rnd(rng, B, L, D)
    args = (rnd(rng, 2, D, scale=0.1) + 1, rnd(rng, 2, k * L, Lp * D, scale=1 / math.sqrt(Lp * D)),
            rnd(rng, 2, k * L), rnd(rng, 2, k, D, scale=0.1) + 1,
            rnd(rng, 2, k, Hkv * d, D, scale=1 / math.sqrt(D)), rnd(rng, k, d, scale=0.1) + 1)
    kw = dict(L=L, k=k, D=D, Hkv=Hkv, d=d, p=2, eps=0.0, eps_qk=0.0, theta=1e6)
    pos = np.array([10.0, 2000.0])
    K0, V0, _, _ = O.kv_mix(h, pos, *args, **kw)
    scale = np.float32(2.0) ** np.arange(L, dtype=np.float32)  # exact in fp32
    K1, V1, _, _ = O.kv_mix((h * scale[None, :, None]).astype(np.float32), pos, *args, **kw)
    np.testing.assert_allclose(K1, K0, rtol=0, atol=1e-12)
    np.testing.assert_allclose(V1, V0, rtol=0, atol=1e-12)


# ----------------------------------------------------------- Table 2 (paper)

def test_table2_decode_flops_from_oracle_counters():
    """Decode FLOPs per token printed in Table 2, rebuilt from the oracle's own
    multiply-accumulate counters for the pool and the attention, plus the
    parts of a Qwen3 layer outside the path (q/o projections and the MLP)."""
    g = json.load(open(os.path.join(GOLDEN, "table2_decode_flops.json")))
    m = g["model"]
    D, Hq, Hkv, d, I, p, ctx = m["D"], m["Hq"], m["Hkv"], m["d"], m["intermediate"], m["p"], m["context"]
    want = g["decode_gflop_per_token"]
    rng = np.random.default_rng(18)
    # one query token of one layer over a ctx-slot cache: counted attention MACs
    kp, vp, pt = make_paged(rng, 1, [ctx], Hkv, d, 64, False)
    _, attn_macs = O.decode_attn(rnd(rng, 1, Hq, d), kp, vp, pt, [ctx], chan=0, Hq=Hq, Hkv=Hkv,
                                 d=d, P=64, return_macs=True)
    other = D * Hq * d + Hq * d * D + 3 * D * I   # q-proj, o-proj, SwiGLU MLP
    vanilla_kv = 2 * D * Hkv * d
    for L in (16, 24, 32):
        gflop = 2 * L * (other + vanilla_kv + attn_macs) / 1e9
        assert round(gflop, 3) == want[f"vanilla_{L}L"]
    L = 16
    for k in (8, 16):
        Lp = -(-L // p)
        h = rnd(rng, 1, L, D)
        _, _, _, macs = O.kv_mix(
            h, np.array([5.0]), np.ones((2, D), np.float32),
            rnd(rng, 2, k * L, Lp * D, scale=0.01), rnd(rng, 2, k * L), np.ones((2, k, D), np.float32),
            rnd(rng, 2, k, Hkv * d, D, scale=0.05), np.ones((k, d), np.float32),
            L=L, k=k, D=D, Hkv=Hkv, d=d, p=p, eps=1e-6, eps_qk=1e-6, theta=1e6)
        router, mix, proj = macs
        assert router == 2 * k * L * Lp * D and proj == 2 * k * Hkv * d * D
        gflop = 2 * (L * (other + attn_macs) + router + mix + proj) / 1e9
        assert round(gflop, 3) == want[f"whitematter_L16_k{k}"]
