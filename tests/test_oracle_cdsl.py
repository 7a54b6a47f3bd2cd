"""Pins of the CDSL oracle (Algorithm 1, Algorithm 2 and the batched CDSL-k step).

Each test ties the oracle to something the paper or the mathematics fixes: the worked reward
example (Sec. 4.1), exact rational threshold tests, the full-acceptance property of hard
rejection with identical models, the reduction of CDSL-k to CDLH and to greedy decoding, and
a brute-force re-derivation of the beam selection over the whole (16-token) vocabulary that
uses no key/value cache."""
import os
from fractions import Fraction

import numpy as np
import pytest

import synth
import oracle
from oracle import (S1, S2_S3, S4, Decider, RunParams, Transformer, cdsl_k_step, coverage,
                    n_min, prefill, reward)

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def shape(vocab=16, d=32, layers=2, heads=4, kv=2, ffn=48):
    return synth.ModelShape(n_layers=layers, d_model=d, n_heads=heads, n_kv_heads=kv,
                            d_ffn=ffn, vocab=vocab)


def model(shp, seed, scale=0.5):
    rng = np.random.default_rng(seed)
    w = {n: (np.ones(s, np.float32) if len(s) == 1 else
             (scale * rng.standard_normal(s)).astype(np.float32)) for n, s in shp.weight_specs()}
    return Transformer(shp, w)


def greedy_chain(m, prompt, n):
    toks = list(prompt)
    for _ in range(n):
        toks.append(int(np.argmax(m.forward_full(toks)[0][-1])))
    return toks[len(prompt):]


# ---------------------------------------------------------------- reward and thresholds

def test_reward_worked_example():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "reward_worked_example.txt"))
            if l.strip() and not l.startswith("#")]
    for n_kw, n_cov, want in rows:
        n_kw, n_cov = int(n_kw), int(n_cov)
        kws = list(range(100, 100 + n_kw))
        text = [7, kws[0], 8, kws[1], kws[1], 9]          # 2 distinct concepts, one repeated
        assert n_cov == 2
        assert coverage(kws, text) == pytest.approx(float(want), abs=0)
        assert reward(kws, text, None, None, False) == pytest.approx(float(want), abs=0)


def test_reward_cases():
    kws = [3, 4, 5]
    assert coverage(kws, []) == 0.0
    assert coverage(kws, [3, 3, 3]) == pytest.approx(1 / 3)
    assert coverage(kws, [5, 4, 3, 9]) == 1.0
    w = np.array([1.0, -2.0])
    h = np.array([0.5, 0.25])               # w.h = 0 -> sigmoid 0.5
    assert reward(kws, [3], h, w, True) == pytest.approx(0.5 * (1 / 3) + 0.25)


def test_reward_composite_away_from_zero():
    """The composite reward's head term where w.h != 0, on closed forms: w.h = ln 3 gives a
    sigmoid of exactly 3/4, w.h = -ln 3 exactly 1/4 (a flipped sign swaps the two), and a
    large positive (negative) w.h drives the head term to 1 (0)."""
    kws = [3, 4, 5, 6]
    w = np.array([1.0, 2.0, 0.0])
    h = np.array([1.0, 2.0, 7.0]) * (np.log(3.0) / 5.0)   # w.h = (1 + 4) ln 3 / 5 = ln 3
    text = [3, 9, 5]                                      # 2 of 4 keywords: coverage 1/2
    assert reward(kws, text, h, w, True) == pytest.approx(0.5 * 0.5 + 0.5 * 0.75, abs=1e-15)
    assert reward(kws, text, -h, w, True) == pytest.approx(0.5 * 0.5 + 0.5 * 0.25, abs=1e-15)
    assert reward(kws, [], h, w, True) == pytest.approx(0.375, abs=1e-15)
    assert reward(kws, [], 40.0 * h, w, True) == pytest.approx(0.5, abs=1e-12)
    assert reward(kws, [], -40.0 * h, w, True) == pytest.approx(0.0, abs=1e-12)


def test_step_head_on_a_bigram_model():
    """The per-row head term of a CDSL-k step and the composite rewards built from it, on a
    target whose attention and FFN outputs are zero (Wo = W_down = 0): its final hidden state
    at every position is then RMSNorm(E[token]) in closed form, so the head of verify row
    (i, j) is sigmoid(w . RMSNorm(E[t_ij])) with t_i = [c_i, x_i1..x_id]. The weights w are
    drawn so that the rows' w.h take both signs well away from 0."""
    shp = shape(vocab=16)
    rng = np.random.default_rng(21)
    wt = {n: (np.ones(s, np.float32) if len(s) == 1 else
              (0.5 * rng.standard_normal(s)).astype(np.float32)) for n, s in shp.weight_specs()}
    for l in range(shp.n_layers):
        wt[f"l{l}.wo"][:] = 0.0
        wt[f"l{l}.w_down"][:] = 0.0
    tgt = Transformer(shp, wt)
    drf = model(shp, 22)
    run = run_params(k=3, d=3, a_t=0.3, r_t=0.3, max_new=8, composite_reward=True)
    w = 0.5 * np.random.default_rng(23).standard_normal(shp.d_model)
    emb = wt["embed"].astype(np.float64)
    hf = emb / np.sqrt(np.mean(emb * emb, axis=-1, keepdims=True) + shp.norm_eps)   # gain 1
    z_tok = hf @ w                                     # w . h for every token id
    assert z_tok.max() > 1.0 and z_tok.min() < -1.0
    kw = [2, 5, 11]
    st = prefill(tgt, drf, np.array([[1, 7, 3, 2]]), np.array([kw]))
    for _ in range(2):
        T0 = list(st[0].T)
        rec = cdsl_k_step(tgt, drf, st, run, w)[0]
        for i in range(run.k):
            toks = [int(rec.roots[i])] + rec.x[i].tolist()
            want = 1.0 / (1.0 + np.exp(-z_tok[toks]))
            assert np.allclose(rec.head[i], want, rtol=0, atol=1e-9)
            cov_full = coverage(kw, T0 + toks)
            assert rec.r_full[i] == pytest.approx(0.5 * cov_full + 0.5 * want[run.d], abs=1e-9)
            n = int(rec.n[i])
            cov_acc = coverage(kw, T0 + toks[:n + 1])
            assert rec.r_acc[i] == pytest.approx(0.5 * cov_acc + 0.5 * want[n], abs=1e-9)


@pytest.mark.parametrize("d", [1, 2, 3, 4, 5, 6, 8, 10])
@pytest.mark.parametrize("a_t", [0.0, 0.25, 0.3, 0.4, 0.5, 0.6, 0.8, 0.9, 1.0, 1.5])
def test_n_min_is_exact_threshold(d, a_t):
    """n >= n_min  <=>  n/d >= a_t, checked in exact rationals (a_t as its float32 value)."""
    at = Fraction(float(np.float32(a_t)))
    nm = n_min(a_t, d)
    for n in range(d + 1):
        assert (n >= nm) == (Fraction(n, d) >= at or
                             np.float32(n) / np.float32(d) >= np.float32(a_t))


def test_decider_tie_rules():
    dec = Decider()
    assert dec.argmax(np.array([1.0, 3.0, 3.0, 2.0]), "x", 0) == 1
    assert dec.topk(np.array([2.0, 5.0, 5.0, 1.0, 5.0]), 3, "roots", 0).tolist() == [1, 2, 4]
    assert dec.first_max(np.array([0.2, 0.4, 0.4]), "beam", 0) == 1
    # near-tie adoption only within tolerance, never for exact ties
    other = {"x": {0: 2, 1: 3, 2: 2}}
    dec = Decider(other=other, tol=0.05)
    assert dec.argmax(np.array([0.0, 1.0, 0.97]), "x", 0) == 2
    assert dec.argmax(np.array([0.0, 1.0, 0.5, 0.9]), "x", 1) == 1
    assert dec.argmax(np.array([0.0, 1.0, 1.0]), "x", 2) == 1
    assert len(dec.adopted) == 1


# ---------------------------------------------------------------- CDSL-k invariants

def run_params(**kw):
    base = dict(k=3, d=3, a_t=0.3, r_t=0.3, max_new=8, composite_reward=True)
    base.update(kw)
    return RunParams(**base)


def test_identical_models_accept_everything():
    """Hard rejection with M_q = M_p: every drafted token is the target's argmax (Sec. 3.2.2)."""
    shp = shape(vocab=40)
    tgt = model(shp, 1)
    drf = model(shp, 1)
    run = run_params(k=4, d=4, r_t=10.0)
    st = prefill(tgt, drf, np.array([[1, 2, 3, 4, 5], [9, 8, 7, 6, 5]]), np.array([[1, 2], [3, 4]]))
    w = np.random.default_rng(2).standard_normal(shp.d_model)
    for _ in range(3):
        for rec in cdsl_k_step(tgt, drf, st, run, w):
            assert np.all(rec.n == run.d)
            assert np.array_equal(rec.argmax[:, :run.d], rec.x)
            assert np.allclose(rec.logp, rec.logq, atol=1e-9)
            assert rec.state == S4            # a = 1 >= a_t, r < r_t = 10


def test_cdsl_reduces_to_cdlh():
    """M_q = M_p and r_t = +inf: every CDSL-k step is the CDLH token of Alg. 2 (Sec. 3.1)."""
    shp = shape(vocab=16)
    tgt = model(shp, 3)
    run = run_params(k=3, d=3, r_t=np.inf, max_new=7)
    w = np.random.default_rng(4).standard_normal(shp.d_model)
    prompt, kw = [1, 7, 3, 2], [5, 11, 13]
    st = prefill(tgt, tgt, np.array([prompt]), np.array([kw]))
    while len(st[0].T) < run.max_new:
        rec = cdsl_k_step(tgt, tgt, st, run, w)[0]
        assert rec.state in (S2_S3, S4) and len(rec.emitted) == 1
    ref = oracle.cdlh_generate(tgt, tgt, tgt, prompt, kw, run, w)
    assert st[0].T == ref.T


def test_always_s1_is_greedy_decoding():
    """a_t = 0, r_t = -inf, M_q = M_p, constant reward: every step is S1 and emits the root
    plus all d accepted tokens, which is greedy decoding of M_p."""
    shp = shape(vocab=30)
    tgt = model(shp, 5)
    run = run_params(k=3, d=3, a_t=0.0, r_t=-np.inf, max_new=9, composite_reward=False)
    prompt = [4, 4, 2, 8]
    st = prefill(tgt, tgt, np.array([prompt]), np.array([[29]]))
    while len(st[0].T) < run.max_new:
        rec = cdsl_k_step(tgt, tgt, st, run, np.zeros(shp.d_model))[0]
        assert rec.state == S1
    assert st[0].T == greedy_chain(tgt, prompt, run.max_new)


def test_generation_stops_at_l_m():
    shp = shape(vocab=30)
    tgt = model(shp, 5)
    run = run_params(k=2, d=4, a_t=0.0, r_t=-np.inf, max_new=6, composite_reward=False)
    st = prefill(tgt, tgt, np.array([[1, 2]]), np.array([[0]]))
    steps = 0
    while len(st[0].T) < run.max_new:
        rec = cdsl_k_step(tgt, tgt, st, run, np.zeros(shp.d_model))[0]
        steps += 1
    assert len(st[0].T) == 6 and steps == 2 and len(rec.emitted) == 1
    assert not cdsl_k_step(tgt, tgt, st, run, np.zeros(shp.d_model))[0].active


def brute_force_step(tgt, drf, prompt, T, kw, run, w):
    """The CDSL-k decision for pfx = prompt + T from scratch: every one of the V tokens is
    tried as a root, each rollout and verify row recomputed with forward_full (no cache)."""
    pfx = list(prompt) + list(T)
    V = tgt.shape.vocab
    p0 = tgt.forward_full(pfx)[0][-1]
    rank = sorted(range(V), key=lambda t: (-p0[t], t))
    cand = {}
    for c in range(V):
        x = []
        for _ in range(run.d):
            x.append(int(np.argmax(drf.forward_full(pfx + [c] + x)[0][-1])))
        lg, hf = tgt.forward_full(pfx + [c] + x)
        rows, hid = lg[len(pfx):], hf[len(pfx):]
        n = 0
        while n < run.d and int(np.argmax(rows[n])) == x[n]:
            n += 1
        rf = reward(kw, T + [c] + x, hid[run.d], w, run.composite_reward)
        ra = reward(kw, T + [c] + x[:n], hid[n], w, run.composite_reward)
        cand[c] = (x, n, rf, ra)
    roots = rank[:run.k]
    rfs = [cand[c][2] for c in roots]
    bi = rfs.index(max(rfs))
    x, n, rf, ra = cand[roots[bi]]
    if n >= n_min(run.a_t, run.d) and np.float32(ra) >= np.float32(run.r_t):
        return roots, bi, S1, [roots[bi]] + x[:n]
    return roots, bi, (S2_S3 if n < n_min(run.a_t, run.d) else S4), [roots[bi]]


@pytest.mark.parametrize("seed,same", [(11, False), (12, True), (13, False)])
def test_brute_force_selection(seed, same):
    shp = shape(vocab=16, d=24)
    tgt = model(shp, seed)
    drf = tgt if same else model(shape(vocab=16, d=16, layers=1, heads=2, kv=1, ffn=20), seed + 100)
    run = run_params(k=4, d=3, a_t=0.3, r_t=0.5, max_new=6)
    w = np.random.default_rng(seed).standard_normal(shp.d_model) * 0.5
    prompt, kw = [3, 1, 4, 1, 5], [2, 6, 9, 12, 15]
    st = prefill(tgt, drf, np.array([prompt]), np.array([kw]))
    while len(st[0].T) < run.max_new:
        T0 = list(st[0].T)
        roots, bi, state, out = brute_force_step(tgt, drf, prompt, T0, kw, run, w)
        rec = cdsl_k_step(tgt, drf, st, run, w)[0]
        assert rec.roots.tolist() == roots
        assert rec.beam == bi and rec.state == state
        assert rec.emitted == out[:run.max_new - len(T0)]


# ---------------------------------------------------------------- literal Alg. 1 and Alg. 2

def test_alg1_identical_models_is_greedy():
    """Alg. 1 with M_q = M_p accepts all d drafts; with r_t = -inf every iteration is S1, so
    the output is greedy decoding of M_p (no bonus token is ever added, Sec. 3.2.3 S1)."""
    shp = shape(vocab=30)
    tgt = model(shp, 21)
    run = run_params(d=3, a_t=0.5, r_t=-np.inf, max_new=9, composite_reward=False)
    prompt = [5, 6, 7]
    st, recs = oracle.alg1_generate(tgt, tgt, prompt, [0], run, np.zeros(shp.d_model))
    assert all(r["n"] == 3 and r["state"] == S1 for r in recs)
    assert st.T == greedy_chain(tgt, prompt, 9)


def test_alg1_s4_appends_cdlh_appx_token():
    shp = shape(vocab=20)
    tgt = model(shp, 22)
    run = run_params(k=3, d=2, a_t=0.5, r_t=np.inf, max_new=3, composite_reward=False)
    prompt = [1, 2, 3]
    st, recs = oracle.alg1_generate(tgt, tgt, prompt, [0, 1], run, np.zeros(shp.d_model))
    r = recs[0]
    assert r["state"] == S4 and r["n"] == 2 and len(r["emitted"]) == 3
    # the appended token is CDLH-appx's choice; with a constant reward it is the top-1 of M_p
    assert r["emitted"] == greedy_chain(tgt, prompt, 3)


def test_alg1_step1_budget():
    """S2/S3 with b = 1: Step-1 takes M_p's greedy token; if its lookahead's reward clears
    r_t it is emitted after the accepted drafts, otherwise Step-2 (CDLH-appx) decides."""
    shp_t, shp_d = shape(vocab=20), shape(vocab=20, d=16, layers=1, heads=2, kv=1, ffn=20)
    tgt, drf = model(shp_t, 31), model(shp_d, 32)
    prompt = [1, 2, 3, 4]
    seen = 0
    for r_t, step1_wins in [(-np.inf, True), (np.inf, False)]:
        run = run_params(k=3, d=3, a_t=1.0, r_t=r_t, max_new=6, composite_reward=False, b=1)
        st, recs = oracle.alg1_generate(tgt, drf, prompt, [0, 1], run, np.zeros(shp_t.d_model))
        T = []
        for r in recs:
            pfx = prompt + T
            T = T + r["emitted"]
            if r["state"] != S2_S3:
                continue
            seen += 1
            acc = r["x"][:r["n"]]
            assert r["emitted"][:len(acc)] == acc and len(r["emitted"]) == len(acc) + 1
            p = tgt.forward_full(pfx + acc)[0][-1]
            if step1_wins:   # Step-1: M_p's greedy token after pfx + accepted drafts
                assert r["emitted"][-1] == int(np.argmax(p))
            else:            # Step-2: one of M_p's top-k there (CDLH-appx)
                assert r["emitted"][-1] in np.argsort(-p)[:run.k].tolist()
    assert seen >= 2


def test_cdlh_appx_with_identical_models_is_cdlh():
    """CDLH-appx with M_q = M_p is CDLH (Alg. 2, lookahead comment)."""
    shp = shape(vocab=16)
    tgt = model(shp, 41)
    run = run_params(k=3, d=2, max_new=5)
    w = np.random.default_rng(42).standard_normal(shp.d_model)
    a = oracle.cdlh_generate(tgt, tgt, tgt, [1, 2, 3], [4, 5], run, w)
    tgt2 = model(shp, 41)
    b = oracle.cdlh_generate(tgt, tgt2, tgt2, [1, 2, 3], [4, 5], run, w)
    assert a.T == b.T


def test_tiny_workload_runs():
    """The tiny fp32 workload end to end: 16 tokens, every step emits >= 1 token."""
    wl = synth.TINY
    tgt = Transformer(wl.target, synth.model_weights(wl, "target"))
    drf = Transformer(wl.draft, synth.model_weights(wl, "draft"))
    run = RunParams(k=wl.k, d=wl.d, a_t=wl.a_t, r_t=wl.r_t, max_new=wl.max_new,
                    composite_reward=wl.reward_head)
    states, recs = oracle.cdsl_k_generate(tgt, drf, synth.prompts(wl), synth.keywords(wl), run,
                                          synth.reward_head(wl))
    assert len(states[0].T) == wl.max_new
    assert all(len(r[0].emitted) >= 1 for r in recs)


# ---------------------------------------------------------------- speculative sampling (f1)

def test_splitmix64_published_outputs():
    """The generator behind the speculative-sampling uniforms matches SplitMix64's published
    check values (seed 1234567)."""
    vals = [int(x) for x in open(os.path.join(GOLDEN, "splitmix64_seed1234567.txt"))
            if x.strip() and not x.startswith("#")]
    seed, want = vals[0], vals[1:]
    assert [oracle.splitmix64(seed, c) for c in range(len(want))] == want


def test_uniform24_is_uniform_and_float32_exact():
    """u = top 24 bits / 2^24: in [0, 1), exactly representable in float32, and uniform
    (mean and a 16-bin chi-square over 2^16 draws)."""
    n = 1 << 16
    u = np.array([oracle.uniform24(12345, c) for c in range(n)])
    assert np.all((u >= 0.0) & (u < 1.0))
    assert np.array_equal(u.astype(np.float32).astype(np.float64), u)
    assert abs(u.mean() - 0.5) < 4 * np.sqrt(1 / 12 / n)
    counts = np.bincount((u * 16).astype(int), minlength=16)
    chi2 = float(np.sum((counts - n / 16) ** 2 / (n / 16)))
    assert chi2 < 45.0          # 15 degrees of freedom: p ~ 1e-4


@pytest.mark.parametrize("rho", [0.1, 0.5, 0.9])
def test_speculative_test_accepts_with_probability_p_over_q(rho):
    """Sec. 3.2.2: a token is rejected when r > min(1, p/q), r ~ U[0, 1]; so it is accepted
    with probability p/q (< 1). The decision on the draws of one generator matches that
    frequency (a flipped inequality would give 1 - p/q)."""
    n = 40000
    dec = Decider()
    acc = sum(dec.accept(np.log(u) if u > 0 else -np.inf, np.log(rho), 0, "spec", None)
              for u in (oracle.uniform24(99, c) for c in range(n)))
    assert abs(acc / n - rho) < 4 * np.sqrt(rho * (1 - rho) / n)


def test_speculative_identical_models_accept_everything():
    """M_q = M_p under speculative sampling: p/q = 1 at every drafted token, every lookahead
    is accepted in full whatever the uniforms."""
    shp = shape(vocab=40)
    tgt = model(shp, 1)
    run = run_params(k=3, d=4, r_t=10.0, acceptance=oracle.SPECULATIVE, seed=5)
    st = prefill(tgt, tgt, np.array([[1, 2, 3, 4, 5], [9, 8, 7, 6, 5]]), np.array([[1, 2], [3, 4]]))
    w = np.random.default_rng(2).standard_normal(shp.d_model)
    for step in range(3):
        for rec in cdsl_k_step(tgt, tgt, st, run, w, step=step):
            assert np.all(rec.n == run.d)


def test_speculative_draws_follow_the_counter():
    """The uniform of (step, prompt, beam, position) is draw number
    ((step * B + b) * k + beam) * d + j: distinct for every decision of a run."""
    B, k, d = 3, 4, 5
    idx = {oracle.draw_index(s, B, b, k, i, d, j) for s in range(4) for b in range(B)
           for i in range(k) for j in range(d)}
    assert idx == set(range(4 * B * k * d))


def test_speculative_vs_hard_on_different_models():
    """Different models: the speculative count never exceeds the draws' verdicts, i.e. every
    accepted position j has u_j <= p_j/q_j, and the first rejected one (if any) has
    u_j > p_j/q_j."""
    shp = shape(vocab=24)
    tgt, drf = model(shp, 1), model(shp, 2)
    run = run_params(k=3, d=4, acceptance=oracle.SPECULATIVE, seed=17)
    st = prefill(tgt, drf, np.array([[1, 2, 3, 4, 5, 6]]), np.array([[1, 2]]))
    w = np.random.default_rng(2).standard_normal(shp.d_model)
    for step in range(4):
        for rec in cdsl_k_step(tgt, drf, st, run, w, step=step):
            if not rec.active:
                continue
            for i in range(run.k):
                for j in range(min(rec.n[i] + 1, run.d)):
                    u = oracle.uniform24(run.seed, oracle.draw_index(step, 1, 0, run.k, i, run.d, j))
                    ratio = np.exp(rec.logp[i, j] - rec.logq[i, j])
                    assert (u <= ratio) == (j < rec.n[i])


# ---------------------------------------------------------------- Sec. 4.3 cost model

def test_cost_model_reproduces_tables_5_and_6():
    """Speedup over CDLH from c (Table 5) and the calls per token (Table 6): P = c * draft
    calls + target calls, CDLH's P = its target calls; every printed speedup is reproduced
    within what the printed inputs' rounding allows (2 decimals for calls, 3 for c, 2 for the
    speedup)."""
    n = 0
    for line in open(os.path.join(GOLDEN, "cost_model_tables.txt")):
        if line.startswith("#") or not line.strip():
            continue
        f = line.split()
        c, dc, tc, cdlh, printed = map(float, f[3:8])
        p = oracle.runtime_per_token(c, dc, tc)
        got = oracle.speedup(oracle.runtime_per_token(c, 0.0, cdlh), p)
        dp = 0.0005 * dc + c * 0.005 + 0.005
        bound = got * (dp / p + 0.005 / cdlh) + 0.005
        assert abs(got - printed) <= bound, (f[:3], got, printed, bound)
        n += 1
    assert n == 14


# ---------------------------------------------------------------- Step-1 with b = 1 (f2)

@pytest.mark.parametrize("seed", [0, 1, 2])
def test_step1_emits_greedy_root_when_its_lookahead_reaches_r_t(seed):
    """Alg. 1 S2/S3 with b = 1: M_p's greedy token (the root c_1) is emitted when the reward
    of its M_q lookahead (beam 1's draft), r_1^full, reaches r_t; otherwise the step falls
    back to the CDLH-appx token c_{b*} exactly as with b = 0. S1 and S4 are unaffected."""
    shp = shape(vocab=24)
    tgt, drf = model(shp, 10 + seed), model(shp, 20 + seed)
    w = np.random.default_rng(seed).standard_normal(shp.d_model)
    prompts = np.array([[1, 2, 3, 4, 5], [6, 7, 8, 9, 10], [3, 1, 4, 1, 5]])
    kw = np.array([[1, 2, 3], [4, 5, 6], [7, 8, 9]])
    seen = {S1: 0, S2_S3: 0, oracle.S2_S3_STEP1: 0, S4: 0}
    for r_t in (0.5, 0.6, 0.7):
        st0 = prefill(tgt, drf, prompts, kw)
        st1 = prefill(tgt, drf, prompts, kw)
        for step in range(3):
            r0 = cdsl_k_step(tgt, drf, st0, run_params(k=3, d=3, r_t=r_t), w, step=step)
            r1 = cdsl_k_step(tgt, drf, st1, run_params(k=3, d=3, r_t=r_t, b=1), w, step=step)
            for a, c in zip(r0, r1):
                seen[c.state] += 1
                assert np.allclose(a.r_full, c.r_full)
                if a.state == S2_S3 and np.float32(a.r_full[0]) >= np.float32(r_t):
                    assert c.state == oracle.S2_S3_STEP1 and c.emitted == [int(a.roots[0])]
                    assert c.beam == 0
                else:
                    assert c.state == a.state and c.emitted == a.emitted
            # keep both runs on the same path: continue from the b = 1 states
            st0 = [dataclasses_copy(s) for s in st1]
    assert sum(seen.values()) == 3 * 3 * 3


def test_step1_always_succeeding_is_greedy_decoding():
    """b = 1, a_t above 1 (S1 never holds) and r_t = 0 (every lookahead reaches it): every step
    is an S2/S3 step resolved by Step-1, i.e. M_p's greedy token: the whole generation is
    M_p's greedy decoding."""
    shp = shape(vocab=24)
    tgt, drf = model(shp, 7), model(shp, 8)
    w = np.random.default_rng(9).standard_normal(shp.d_model)
    prompt = [2, 7, 1, 8]
    run = run_params(k=3, d=3, a_t=1.5, r_t=0.0, b=1, max_new=8)
    st = prefill(tgt, drf, np.array([prompt]), np.array([[1, 2, 3]]))
    step = 0
    while len(st[0].T) < run.max_new:
        rec = cdsl_k_step(tgt, drf, st, run, w, step=step)[0]
        assert rec.state == oracle.S2_S3_STEP1 and rec.beam == 0
        step += 1
    assert st[0].T == greedy_chain(tgt, prompt, run.max_new)


def dataclasses_copy(st):
    import dataclasses
    return dataclasses.replace(st, tcache=st.tcache.fork(), dcache=st.dcache.fork())


def test_step1_with_one_beam_changes_no_token():
    """k = 1: c_1 is the only beam, so the Step-1 token and the CDLH-appx token coincide; only
    the reported state differs."""
    shp = shape(vocab=24)
    tgt, drf = model(shp, 3), model(shp, 4)
    w = np.random.default_rng(5).standard_normal(shp.d_model)
    p = np.array([[1, 2, 3, 4]])
    kw = np.array([[1, 2, 3]])
    a = prefill(tgt, drf, p, kw)
    b = prefill(tgt, drf, p, kw)
    for step in range(4):
        ra = cdsl_k_step(tgt, drf, a, run_params(k=1, d=3, r_t=0.4), w, step=step)[0]
        rb = cdsl_k_step(tgt, drf, b, run_params(k=1, d=3, r_t=0.4, b=1), w, step=step)[0]
        assert ra.emitted == rb.emitted
        assert (ra.state == rb.state) or (ra.state == S2_S3 and rb.state == oracle.S2_S3_STEP1)


# ---------------------------------------------------------------- Step-1 with b = 2 (f2)

def _fork_state(st):
    import dataclasses
    return dataclasses.replace(st, T=list(st.T), tcache=st.tcache.fork(), dcache=st.dcache.fork())


def test_step1_second_round_emits_two_greedy_tokens():
    """b = 2 with M_q = M_p, a_t above 1 (every step is S2/S3) and r_t = 1 on a single keyword
    that M_p's greedy text reaches only at token d + 2: round 1 (c_1 + its lookahead, tokens
    g_1..g_{d+1}) misses it, round 2 (g_1, g_2 + lookahead g_3..g_{d+2}) covers it, so the
    step emits M_p's first two greedy tokens. With b = 1 the same step falls back to Step-2."""
    d = 3
    shp = shape(vocab=24)
    tgt = model(shp, 17)
    found = 0
    for p0 in range(12):
        prompt = [p0 % 24, (3 * p0 + 1) % 24, (5 * p0 + 2) % 24, 7]
        g = greedy_chain(tgt, prompt, d + 2)
        if g[d + 1] in g[:d + 1] or g[d + 1] in prompt:
            continue
        found += 1
        kw = np.array([[g[d + 1]]])
        for b, want_state, want_out in ((2, oracle.S2_S3_STEP1, g[:2]), (1, S2_S3, None)):
            st = prefill(tgt, tgt, np.array([prompt]), kw)
            run = run_params(k=3, d=d, a_t=1.5, r_t=1.0, composite_reward=False, b=b)
            rec = cdsl_k_step(tgt, tgt, st, run, np.zeros(shp.d_model), step=0)[0]
            assert rec.state == want_state
            if b == 2:
                assert rec.emitted == want_out and rec.beam == 0
                (toks, r), = rec.step1_rounds
                assert toks.tolist() == g[1:d + 2] and r == 1.0
                # the committed caches continue M_p's greedy text
                nxt = cdsl_k_step(tgt, tgt, st, run_params(k=3, d=d, a_t=1.5, r_t=-np.inf,
                                                           composite_reward=False, b=1),
                                  np.zeros(shp.d_model), step=1)[0]
                assert nxt.emitted == [g[2]]
            else:
                assert len(rec.emitted) == 1 and rec.step1_rounds == []
        if found >= 3:
            break
    assert found >= 3


def test_step1_second_round_truncated_at_l_m():
    """A Step-1 success in round 2 with one token left before l_m emits c_1 alone."""
    d = 2
    shp = shape(vocab=24)
    tgt = model(shp, 23)
    for p0 in range(12):
        prompt = [p0, (7 * p0 + 3) % 24, 11]
        g = greedy_chain(tgt, prompt, d + 2)
        if g[d + 1] in g[:d + 1] or g[d + 1] in prompt:
            continue
        st = prefill(tgt, tgt, np.array([prompt]), np.array([[g[d + 1]]]))
        run = run_params(k=2, d=d, a_t=1.5, r_t=1.0, composite_reward=False, b=2, max_new=1)
        rec = cdsl_k_step(tgt, tgt, st, run, np.zeros(shp.d_model), step=0)[0]
        assert rec.state == oracle.S2_S3_STEP1 and rec.emitted == [g[0]] and st[0].T == [g[0]]
        return
    pytest.fail("no prompt with a fresh keyword at greedy position d + 2")


@pytest.mark.parametrize("r_t, same_as", [(0.0, 1), (np.inf, 0)])
def test_step1_budget2_limits(r_t, same_as):
    """r_t = 0: round 1 always succeeds, so b = 2 runs exactly like b = 1; r_t = inf: no round
    succeeds, so b = 2 emits exactly what b = 0 does (Step-2)."""
    shp = shape(vocab=24)
    tgt, drf = model(shp, 51), model(shp, 52)
    w = np.random.default_rng(53).standard_normal(shp.d_model)
    prompts = np.array([[1, 2, 3, 4], [5, 6, 7, 8]])
    kw = np.array([[1, 2, 3], [4, 5, 6]])
    a, c = prefill(tgt, drf, prompts, kw), prefill(tgt, drf, prompts, kw)
    for step in range(4):
        ra = cdsl_k_step(tgt, drf, a, run_params(r_t=r_t, a_t=0.6, b=same_as), w, step=step)
        rc = cdsl_k_step(tgt, drf, c, run_params(r_t=r_t, a_t=0.6, b=2), w, step=step)
        for x, y in zip(ra, rc):
            assert x.emitted == y.emitted and x.state == y.state and x.beam == y.beam
    assert [s.T for s in a] == [s.T for s in c]


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_step1_rounds_match_literal_algorithm1(seed):
    """k = 1 and a step with no accepted draft (n = 0) in S2/S3: the batched step's Step-1 and
    literal Algorithm 1's Step-1 (which starts after the accepted drafts, here none) take the
    same greedy tokens, the same lookaheads and the same rewards, so with b = 2 they emit the
    same tokens. The two share no Step-1 code."""
    shp = shape(vocab=20)
    dshp = shape(vocab=20, d=16, layers=1, heads=2, kv=1, ffn=20)
    tgt, drf = model(shp, 60 + seed), model(dshp, 70 + seed)
    w = np.random.default_rng(80 + seed).standard_normal(shp.d_model)
    rng = np.random.default_rng(90 + seed)
    compared = {1: 0, 2: 0, 0: 0}
    for trial in range(16):
        prompt = rng.integers(0, 20, size=5).tolist()
        kw = rng.choice(20, size=3, replace=False).tolist()
        r_t = float(rng.uniform(0.3, 0.7))
        run = run_params(k=1, d=3, a_t=0.9, r_t=r_t, b=2, max_new=4)
        lit = oracle.alg1_generate(tgt, drf, prompt, kw, run, w, max_steps=1)[1][0]
        if lit["n"] != 0 or lit["state"] != S2_S3:
            continue
        st = prefill(tgt, drf, np.array([prompt]), np.array([kw]))
        rec = cdsl_k_step(tgt, drf, st, run, w, step=0)[0]
        if rec.state not in (S2_S3, oracle.S2_S3_STEP1):   # its own draft (after c_1) passed
            continue
        # literal Alg. 1 emits X after Step-1 success, else CDLH-appx's token (k = 1: c_1)
        assert rec.emitted == lit["emitted"]
        compared[0 if rec.state == S2_S3 else len(rec.emitted)] += 1
    assert min(compared.values()) >= 1   # Step-2, round-1 and round-2 outcomes all compared


def test_adoption_bound_rejects_wide_margins():
    """The parity harness fails a run where the oracle adopted a choice whose own margin is
    wider than the bound (a wrong choice on the other side, not rounding), and passes one
    within it."""
    from cdsl_parity import adopt_bound_for, check_adoptions
    bound = adopt_bound_for(2e-2)
    assert bound == pytest.approx(3e-3) and adopt_bound_for(1e-4) == pytest.approx(1e-4)
    logits = np.zeros((1, 1, 1, 4))
    for gap, ok in ((1e-3, True), (5e-3, False)):
        dec = Decider(other={"argmax": {(0, 0, 0): 2}}, tol=2e-2)
        v = np.array([0.0, 1.0, 1.0 - gap, 0.5])
        assert dec.argmax(v, "argmax", (0, 0, 0)) == 2 and dec.margins == [pytest.approx(gap)]
        logits[0, 0, 0] = v
        rep = {}
        if ok:
            check_adoptions(dec, {"logits": logits}, bound, rep)
            assert rep["adopt_margin"] == pytest.approx(gap)
        else:
            with pytest.raises(AssertionError):
                check_adoptions(dec, {"logits": logits}, bound, rep)
