"""Pins of the oracle transformer against things other than itself.

Closed forms (RoPE as a complex rotation, RMS of RMSNorm, one-key attention), invariants
(relative-position property of RoPE, causality, verify == sequential decode, batching and
forking invariance) and a scalar loop-by-loop restatement of the model on tiny shapes."""
import cmath
import math

import numpy as np
import pytest

import synth
from oracle import Transformer, log_softmax, rms_norm, rope, silu, softmax


def tiny_shape(layers=2, d=16, heads=4, kv=2, ffn=24, vocab=11):
    return synth.ModelShape(n_layers=layers, d_model=d, n_heads=heads, n_kv_heads=kv,
                            d_ffn=ffn, vocab=vocab)


def rand_weights(shape, seed, scale=0.3, random_gains=True):
    rng = np.random.default_rng(seed)
    w = {}
    for name, shp in shape.weight_specs():
        if len(shp) == 1:
            w[name] = (1.0 + 0.2 * rng.standard_normal(shp)).astype(np.float32) if random_gains \
                else np.ones(shp, np.float32)
        else:
            w[name] = (scale * rng.standard_normal(shp)).astype(np.float32)
    return w


# ---------------------------------------------------------------- closed forms

def test_rope_is_complex_rotation():
    rng = np.random.default_rng(1)
    n, H, hd, theta = 5, 3, 8, 10000.0
    x = rng.standard_normal((n, H, hd))
    pos = np.array([0, 1, 7, 100, 4095])
    y = rope(x, pos, theta)
    half = hd // 2
    for i in range(n):
        for h in range(H):
            for m in range(half):
                z = complex(x[i, h, m], x[i, h, m + half])
                zr = z * cmath.exp(1j * pos[i] * theta ** (-2.0 * m / hd))
                assert abs(y[i, h, m] - zr.real) < 1e-12
                assert abs(y[i, h, m + half] - zr.imag) < 1e-12


def test_rope_relative_position():
    rng = np.random.default_rng(2)
    q = rng.standard_normal((1, 1, 16))
    k = rng.standard_normal((1, 1, 16))
    for m, n, s in [(3, 1, 10), (50, 49, 700), (0, 9, 33)]:
        a = np.sum(rope(q, np.array([m]), 1e4) * rope(k, np.array([n]), 1e4))
        b = np.sum(rope(q, np.array([m + s]), 1e4) * rope(k, np.array([n + s]), 1e4))
        assert abs(a - b) < 1e-10
    # position 0 is the identity
    assert np.allclose(rope(q, np.array([0]), 1e4), q)


def test_rmsnorm_unit_rms():
    rng = np.random.default_rng(3)
    x = 5.0 * rng.standard_normal((4, 64))
    eps = 1e-5
    y = rms_norm(x, np.ones(64), eps)
    ms = np.mean(x * x, axis=-1)
    assert np.allclose(np.sqrt(np.mean(y * y, axis=-1)), np.sqrt(ms / (ms + eps)), atol=1e-12)
    g = rng.standard_normal(64)
    assert np.allclose(rms_norm(x, g, eps), y * g)


def test_softmax_and_log_softmax():
    rng = np.random.default_rng(4)
    v = 10 * rng.standard_normal((7, 300))
    p = softmax(v)
    assert np.all(np.abs(p.sum(-1) - 1) < 1e-12)
    lp = log_softmax(v)
    assert np.all(lp <= 0)
    assert np.allclose(np.exp(lp), p)
    lse = v - lp
    assert np.all(lse >= v.max(-1, keepdims=True) - 1e-12)
    assert np.allclose(silu(np.array([0.0, 1.0, -2.0])),
                       [0.0, 1.0 / (1 + math.exp(-1)), -2.0 / (1 + math.exp(2))])


def test_one_key_attention_ignores_q_and_k():
    """With a single position, softmax over one key is 1: the output is v, whatever Wq, Wk."""
    shape = tiny_shape(layers=1)
    w = rand_weights(shape, 5)
    a = Transformer(shape, w).forward_full([3])[0]
    w2 = dict(w)
    rng = np.random.default_rng(6)
    w2["l0.wq"] = rng.standard_normal(w["l0.wq"].shape).astype(np.float32)
    w2["l0.wk"] = rng.standard_normal(w["l0.wk"].shape).astype(np.float32)
    b = Transformer(shape, w2).forward_full([3])[0]
    assert np.allclose(a, b, atol=1e-12)
    # ... while a second position does depend on them
    a2 = Transformer(shape, w).forward_full([3, 4])[0]
    b2 = Transformer(shape, w2).forward_full([3, 4])[0]
    assert np.allclose(a2[0], b2[0], atol=1e-12) and not np.allclose(a2[1], b2[1], atol=1e-6)


# ---------------------------------------------------------------- scalar restatement

def loop_forward(shape, w, tokens):
    """The decoder written out with scalar loops, complex-number RoPE and explicit GQA."""
    D, H, KV, hd, F = shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.d_ffn
    G = H // KV
    W = {k: np.asarray(v, dtype=np.float64).tolist() for k, v in w.items()}

    def matvec(M, x):
        return [sum(M[o][i] * x[i] for i in range(len(x))) for o in range(len(M))]

    def norm(x, g):
        r = math.sqrt(sum(t * t for t in x) / len(x) + shape.norm_eps)
        return [x[i] / r * g[i] for i in range(len(x))]

    def rot(vec, p):
        out = list(vec)
        for m in range(hd // 2):
            z = complex(vec[m], vec[m + hd // 2]) * cmath.exp(
                1j * p * shape.rope_theta ** (-2.0 * m / hd))
            out[m], out[m + hd // 2] = z.real, z.imag
        return out

    hs = [list(W["embed"][t]) for t in tokens]
    for l in range(shape.n_layers):
        Ks, Vs, Qs = [], [], []
        for p, h in enumerate(hs):
            a = norm(h, W[f"l{l}.attn_norm"])
            q, k, v = matvec(W[f"l{l}.wq"], a), matvec(W[f"l{l}.wk"], a), matvec(W[f"l{l}.wv"], a)
            Qs.append([rot(q[hh * hd:(hh + 1) * hd], p) for hh in range(H)])
            Ks.append([rot(k[g * hd:(g + 1) * hd], p) for g in range(KV)])
            Vs.append([v[g * hd:(g + 1) * hd] for g in range(KV)])
        new = []
        for p, h in enumerate(hs):
            att = []
            for hh in range(H):
                g = hh // G
                s = [sum(Qs[p][hh][e] * Ks[t][g][e] for e in range(hd)) / math.sqrt(hd)
                     for t in range(p + 1)]
                mx = max(s)
                e_ = [math.exp(x - mx) for x in s]
                z = sum(e_)
                att += [sum(e_[t] / z * Vs[t][g][e] for t in range(p + 1)) for e in range(hd)]
            o = matvec(W[f"l{l}.wo"], att)
            h2 = [h[i] + o[i] for i in range(D)]
            a = norm(h2, W[f"l{l}.ffn_norm"])
            gt, up = matvec(W[f"l{l}.w_gate"], a), matvec(W[f"l{l}.w_up"], a)
            act = [gt[i] / (1 + math.exp(-gt[i])) * up[i] for i in range(F)]
            dn = matvec(W[f"l{l}.w_down"], act)
            new.append([h2[i] + dn[i] for i in range(D)])
        hs = new
    return np.array([matvec(W["lm_head"], norm(h, W["final_norm"])) for h in hs])


@pytest.mark.parametrize("heads,kv", [(4, 2), (4, 4), (4, 1)])
def test_matches_scalar_loops(heads, kv):
    shape = tiny_shape(heads=heads, kv=kv)
    w = rand_weights(shape, 7 + heads + kv)
    toks = [1, 5, 2, 9, 0, 10]
    ref = loop_forward(shape, w, toks)
    got = Transformer(shape, w).forward_full(toks)[0]
    assert np.max(np.abs(ref - got)) < 1e-10


def test_bf16_weights_are_widened_bit_exactly():
    shape = tiny_shape(layers=1)
    w32 = rand_weights(shape, 8)
    wb = {k: synth.f32_to_bf16_bits(v) for k, v in w32.items()}
    # reference widening: place the 16 bits on top of a float32
    back = {k: np.frombuffer((v.astype(np.uint32) << 16).tobytes(), dtype=np.float32).reshape(v.shape)
            for k, v in wb.items()}
    a = Transformer(shape, wb).forward_full([1, 2, 3])[0]
    b = Transformer(shape, back).forward_full([1, 2, 3])[0]
    assert np.array_equal(a, b)


# ---------------------------------------------------------------- cache invariants

def test_verify_equals_sequential_decode():
    """One pass over pfx + x_1..x_d equals d+1 incremental decode calls (Alg. 1 verification)."""
    shape = tiny_shape(layers=2, d=32, heads=4, kv=2, ffn=40, vocab=50)
    m = Transformer(shape, rand_weights(shape, 9))
    pfx, xs = [3, 14, 15, 9, 2, 6], [5, 35, 8, 9]
    full = m.forward_full(pfx + xs)[0]
    cache = m.new_cache()
    m.forward([(cache, pfx)])
    one_pass = m.forward([(cache.fork(), xs)])[0][0]
    seq = []
    c = cache.fork()
    for t in xs:
        seq.append(m.forward([(c, [t])])[0][0][0])
    seq = np.stack(seq)
    assert np.max(np.abs(one_pass - seq)) < 1e-10
    assert np.max(np.abs(full[len(pfx):] - one_pass)) < 1e-10


def test_causality_and_batching():
    shape = tiny_shape(layers=2, d=32, heads=4, kv=2, ffn=40, vocab=50)
    m = Transformer(shape, rand_weights(shape, 10))
    a = m.forward_full([1, 2, 3, 4, 5])[0]
    b = m.forward_full([1, 2, 3, 40, 41])[0]
    assert np.allclose(a[:3], b[:3], atol=1e-12) and not np.allclose(a[3], b[3])
    # several sequences through one call == each alone
    c1, c2, c3 = m.new_cache(), m.new_cache(), m.new_cache()
    m.forward([(c1, [7, 8])])
    lg, _ = m.forward([(c1, [9, 10, 11]), (c2, [1]), (c3, [4, 5, 6, 7])])
    assert np.allclose(lg[0], m.forward_full([7, 8, 9, 10, 11])[0][2:], atol=1e-12)
    assert np.allclose(lg[1], m.forward_full([1])[0], atol=1e-12)
    assert np.allclose(lg[2], m.forward_full([4, 5, 6, 7])[0], atol=1e-12)


def test_fork_shares_prefix_only():
    shape = tiny_shape(layers=1, d=16, heads=2, kv=1, ffn=8, vocab=20)
    m = Transformer(shape, rand_weights(shape, 11))
    base = m.new_cache()
    m.forward([(base, [1, 2, 3])])
    f1, f2 = base.fork(), base.fork()
    l1 = m.forward([(f1, [4])])[0][0]
    m.forward([(f2, [9, 9, 9])])
    l1b = m.forward([(base.fork(), [4])])[0][0]
    assert np.allclose(l1, l1b) and len(f1) == 4 and len(f2) == 6 and len(base) == 3
    t = f2.truncated(4)
    assert len(t) == 4
    assert np.allclose(m.forward([(t, [5])])[0][0], m.forward_full([1, 2, 3, 9, 5])[0][-1:])
