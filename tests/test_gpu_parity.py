"""CUDA path vs the oracle, element by element, through the C ABI.

Tolerances (stated by the target of this work for the two precisions): logits / log-probs
|diff| <= 1e-4 for the float32 workload, <= 2e-2 for bf16 weights with fp32 accumulation.
Token ids, n_b, b*, the state and the emitted tokens must be identical; at a near tie (the
oracle's own margin below the tolerance) the oracle adopts the CUDA path's choice and the run
continues along it."""
import numpy as np
import pytest

import synth
import oracle
from cdsl_parity import (compare_step, decider_from, gpu_step_outputs, make_engine, make_setup,
                         oracle_models, oracle_prefill, run_params, run_parity)

pytestmark = pytest.mark.gpu

TOL32 = 1e-4
TOL16 = 2e-2


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2412_10418_gb300 import build
    build.build()


def tokens_match(eng, states):
    t, n = eng.tokens()
    t, n = t.cpu().numpy(), n.cpu().numpy()
    for b, st in enumerate(states):
        want = st.prompt + st.T
        assert n[b] == len(want)
        assert t[b, :n[b]].tolist() == want


def test_tiny_fp32_full_run():
    s = make_setup(synth.TINY)
    eng, states, rep, adopted, n = run_parity(s, steps=40, tol=TOL32, tol_r=TOL32)
    assert all(len(st.T) == synth.TINY.max_new for st in states)
    tokens_match(eng, states)
    c = eng.counters()
    assert c[0] == n and c[3] == synth.TINY.max_new


def greedy_chain(tgt, prompt, n):
    toks = list(prompt)
    for _ in range(n):
        toks.append(int(np.argmax(tgt.forward_full(toks)[0][-1])))
    return toks[len(prompt):]


def test_tiny_forced_acceptance_s1_and_pending_rows():
    """Draft := target: every lookahead is accepted (n = d). Keywords taken from the target's
    greedy continuation make the reward clear r_t, so steps are S1 and emit d+1 tokens; the
    next step's first draft call must then fill the draft KV of the last drafted token."""
    wl = synth.scaled(synth.TINY, draft=synth.TINY.target, max_new=24)
    s = make_setup(wl, draft_equals_target=True)
    tgt = oracle.Transformer(wl.target, s.t_host)
    chain = greedy_chain(tgt, s.prompts[0].tolist(), 12)
    s.keywords = np.array([[chain[2], chain[7], chain[11]]], dtype=np.int32)
    eng, states, rep, adopted, n = run_parity(s, steps=30, tol=TOL32, tol_r=TOL32)
    tokens_match(eng, states)
    c = eng.counters()
    assert c[4] >= 2, f"expected S1 steps, counters {c}"
    assert c[3] == wl.max_new


def test_ragged_batch_small_pages():
    wl = synth.scaled(synth.TINY, batch=3, prompt_len=40, max_new=12)
    s = make_setup(wl, lens=[40, 17, 33])
    eng, states, rep, adopted, n = run_parity(s, steps=20, tol=TOL32, tol_r=TOL32, page_size=16,
                                              max_chunk=24)
    tokens_match(eng, states)


@pytest.mark.parametrize("k,d", [(1, 1), (2, 3), (16, 2), (8, 12)])
def test_beam_and_lookahead_extremes(k, d):
    """(8, 12) with one query head per KV head: the draft rows' beam tails (up to 8 x 12 keys
    per query block) span two tail-key chunks of the attention."""
    wl = synth.scaled(synth.TINY, k=k, d=d, max_new=7)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=10, tol=TOL32, tol_r=TOL32)
    tokens_match(eng, states)


def test_tiny_maximum_context():
    """The longest context the attention takes (8128 positions): an 8100-token prompt, so the
    passes see 127 prefix chunks of 64 keys plus the beam tails, 8 chunks per block of a
    16-block cluster; the prefill runs 127 passes of 64 rows."""
    wl = synth.scaled(synth.TINY, prompt_len=8100, max_new=8, k=2, d=2)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=4, tol=TOL32, tol_r=TOL32)
    tokens_match(eng, states)


def test_graph_step_equals_separate_calls():
    import torch
    wl = synth.scaled(synth.TINY, batch=2, max_new=12)
    s = make_setup(wl)
    a = make_engine(s)
    b = make_engine(s)
    for _ in range(12):
        a.step()
        b.lookahead(); b.verify(); b.select()
    ta, na = a.tokens()
    tb, nb = b.tokens()
    assert torch.equal(na, nb) and torch.equal(ta, tb)
    assert a.counters()[:6] == b.counters()[:6] and a.counters()[6] > 0
    assert int(na[0]) == wl.prompt_len + wl.max_new


def test_small_bf16_parity():
    s = make_setup(synth.SMALL)
    eng, states, rep, adopted, n = run_parity(s, steps=4, tol=TOL16, tol_r=TOL16)
    assert n == 4
    print("max |diff|:", rep, "near ties adopted:", len(adopted))


@pytest.mark.parametrize("batch,k", [(1, 4), (2, 2), (1, 8)])
def test_small_bf16_few_rows(batch, k):
    """Draft calls with B*k (+B) <= 8 rows: the tensor-core GEMM's cluster split-K schedules
    at the smallest activation tile (16 rows, of which at most 8 are live)."""
    wl = synth.scaled(synth.SMALL, batch=batch, k=k, max_new=10)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=4, tol=TOL16, tol_r=TOL16)
    tokens_match(eng, states)
    print("few rows", batch, k, "max |diff|:", rep)


def test_small_bf16_forced_acceptance():
    """bf16, draft := target, B = 1: full acceptance and S1 emissions (multi-token commits),
    including the pending draft row of the next step's first draft call."""
    wl = synth.scaled(synth.SMALL, batch=1, draft=synth.SMALL.target, max_new=16, n_keywords=3)
    s = make_setup(wl, draft_equals_target=True)
    tgt = oracle.Transformer(wl.target, s.t_host)
    chain = greedy_chain(tgt, s.prompts[0].tolist(), 8)
    s.keywords = np.array([[chain[1], chain[5], chain[7]]], dtype=np.int32)
    eng, states, rep, adopted, n = run_parity(s, steps=8, tol=TOL16, tol_r=TOL16)
    tokens_match(eng, states)
    assert eng.counters()[4] >= 1


def test_nonfinite_logits_are_flagged():
    """A NaN planted in the input (an embedding row the prompt uses) is reported through the
    device status word as CDSL_ENONFINITE; nothing faults."""
    import torch
    wl = synth.scaled(synth.TINY, max_new=2)
    s = make_setup(wl)
    tw = synth.to_torch(s.t_host, wl.dtype)
    dw = synth.to_torch(s.d_host, wl.dtype)
    tw["embed"][int(s.prompts[0, 5])] = float("nan")
    eng = make_engine(s, torch_weights=(tw, dw))
    eng.lookahead(); eng.verify(); eng.select()
    assert eng.status() == 5


@pytest.mark.parametrize("seed", [1, 7])
def test_tiny_speculative_sampling(seed):
    """Speculative-sampling validation (Sec. 3.2.2): n_b from u <= min(1, p/q) with the
    SplitMix64 uniforms both sides draw from the same counters."""
    wl = synth.scaled(synth.TINY, batch=2, max_new=24)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=24, tol=TOL32, tol_r=TOL32,
                                              acceptance=oracle.SPECULATIVE, seed=seed)
    tokens_match(eng, states)
    assert rep["accepted"] > 0      # some drafted tokens passed u <= p/q
    print("speculative sampling", seed, "max |diff|:", rep, "adopted:", len(adopted))


def test_tiny_speculative_sampling_draft_equals_target():
    """M_q = M_p: p/q = 1 at every drafted token, so every lookahead is accepted in full."""
    wl = synth.scaled(synth.TINY, draft=synth.TINY.target, max_new=20)
    s = make_setup(wl, draft_equals_target=True)
    eng, states, rep, adopted, n = run_parity(s, steps=20, tol=TOL32, tol_r=TOL32,
                                              acceptance=oracle.SPECULATIVE, seed=3)
    tokens_match(eng, states)
    g = gpu_step_outputs(eng)
    if g["n_emitted"].sum() > 0:
        assert np.all(g["n_accept"][g["n_emitted"] > 0] == wl.d)


def test_small_bf16_speculative_sampling():
    wl = synth.scaled(synth.SMALL, batch=2, max_new=16)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=4, tol=TOL16, tol_r=TOL16,
                                              acceptance=oracle.SPECULATIVE, seed=11)
    tokens_match(eng, states)
    assert rep["accepted"] > 0
    print("bf16 speculative sampling max |diff|:", rep, "adopted:", len(adopted))


def test_tiny_cdlh_on_the_same_kernels():
    """Alg. 2 CDLH on the GPU path: M_p drafts its own lookaheads and no reward reaches r_t,
    so every step emits one token: the CDLH token of the oracle's Alg. 2 (Sec. 3.1), step by
    step and over the whole generation."""
    wl = synth.scaled(synth.TINY, draft=synth.TINY.target, r_t=2.0, max_new=10)
    s = make_setup(wl, draft_equals_target=True)
    eng, states, rep, adopted, n = run_parity(s, steps=10, tol=TOL32, tol_r=TOL32)
    assert n == wl.max_new                # one token per step
    tokens_match(eng, states)
    tgt = oracle.Transformer(wl.target, s.t_host)
    run = run_params(wl)
    for b in range(wl.batch):
        ref = oracle.cdlh_generate(tgt, tgt, tgt, s.prompts[b].tolist(), s.keywords[b].tolist(),
                                   run, s.w_head)
        assert states[b].T == ref.T


def test_tiny_gqa_wide_query_blocks():
    """Grouped-query attention (2 query heads per KV head): the 4 x 5 verify rows make 40 query
    vectors per KV head, taken by one block of 40 (5 per warp); the draft rows by blocks of 16
    and 32. Ragged batch."""
    tgt = synth.ModelShape(n_layers=2, d_model=256, n_heads=4, n_kv_heads=2, d_ffn=688, vocab=512)
    drf = synth.ModelShape(n_layers=1, d_model=128, n_heads=2, n_kv_heads=1, d_ffn=344, vocab=512)
    wl = synth.scaled(synth.TINY, target=tgt, draft=drf, batch=2, prompt_len=40, max_new=16)
    s = make_setup(wl, lens=[40, 23])
    eng, states, rep, adopted, n = run_parity(s, steps=16, tol=TOL32, tol_r=TOL32)
    tokens_match(eng, states)


def test_tiny_step1_always_succeeding_is_greedy():
    """Step-1 budget b = 1 with a_t above 1 and r_t = 0: every step is an S2/S3 step resolved
    by Step-1 (state 3), emitting M_p's greedy token."""
    wl = synth.scaled(synth.TINY, a_t=1.5, r_t=0.0, max_new=12)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=12, tol=TOL32, tol_r=TOL32,
                                              step1_budget=1)
    tokens_match(eng, states)
    tgt = oracle.Transformer(wl.target, s.t_host)
    assert states[0].T == greedy_chain(tgt, s.prompts[0].tolist(), wl.max_new)


def test_tiny_step1_mixed_states():
    """b = 1 with keywords from M_p's greedy continuation: Step-1 resolves some S2/S3 steps,
    the others fall back to the CDLH-appx token; GPU and oracle agree step by step."""
    wl = synth.scaled(synth.TINY, batch=2, max_new=20)
    t_host = synth.model_weights(wl, "target", device="host")
    tgt = oracle.Transformer(wl.target, t_host)
    p = synth.prompts(wl)
    kw = np.stack([np.array(greedy_chain(tgt, p[b].tolist(), 12)[3:12:4], np.int32)
                   for b in range(wl.batch)])
    s = make_setup(wl, keywords=kw)
    eng, states, rep, adopted, n = run_parity(s, steps=20, tol=TOL32, tol_r=TOL32,
                                              step1_budget=1)
    tokens_match(eng, states)
    assert rep.get(f"state{oracle.S2_S3_STEP1}", 0) > 0, rep
    print("step-1 states:", {k: v for k, v in rep.items() if k.startswith("state")})


def test_tiny_step1_second_round_follows_greedy_text():
    """Step-1 budget b = 2, one beam (k = 1: Step-2 emits c_1, M_p's greedy token), M_q = M_p,
    a_t above 1 (every step S2/S3), r_t = 1 over keywords g_1, g_2 and g_p (M_p's greedy
    tokens, p = d + 5): round 2, taking g_t+1, g_t+2 with lookahead g_t+3..g_t+d+2, first
    covers g_p at t = 3: that step emits two tokens, after three single-token steps; then
    round 1 succeeds every step. The whole generation is M_p's greedy text, GPU and oracle
    step by step (with k = 1 the round's d+2 target rows outnumber the verify rows)."""
    wl = synth.scaled(synth.TINY, k=1, a_t=1.5, r_t=1.0, max_new=12)
    t_host = synth.model_weights(wl, "target", device="host")
    tgt = oracle.Transformer(wl.target, t_host)
    p = synth.prompts(wl)[0].tolist()
    g = greedy_chain(tgt, p, wl.max_new)
    pk = wl.d + 5
    assert len({g[0], g[1], g[pk - 1]}) == 3 and g[pk - 1] not in g[:pk - 1]
    s = make_setup(wl, keywords=np.array([[g[0], g[1], g[pk - 1]]], np.int32),
                   draft_equals_target=True)
    eng, states, rep, adopted, n = run_parity(s, steps=12, tol=TOL32, tol_r=TOL32,
                                              step1_budget=2)
    tokens_match(eng, states)
    assert states[0].T == g
    assert rep.get("round2_ok", 0) == 1 and rep.get("round2", 0) == 4, rep


def test_tiny_step1_budget2_mixed_states():
    """b = 2 with independent models and keywords from M_p's greedy continuation: round 1,
    round 2 and Step-2 each decide some S2/S3 steps; GPU and oracle agree step by step
    (tokens and reward of every round 2 included)."""
    wl = synth.scaled(synth.TINY, batch=2, max_new=24, r_t=0.6)
    t_host = synth.model_weights(wl, "target", device="host")
    tgt = oracle.Transformer(wl.target, t_host)
    p = synth.prompts(wl)
    kw = np.stack([np.array(greedy_chain(tgt, p[b].tolist(), 12)[2:12:4], np.int32)
                   for b in range(wl.batch)])
    s = make_setup(wl, keywords=kw)
    eng, states, rep, adopted, n = run_parity(s, steps=24, tol=TOL32, tol_r=TOL32,
                                              step1_budget=2)
    tokens_match(eng, states)
    print("budget-2 report:", rep)
    assert rep.get("round2", 0) > 0, rep


def test_tiny_step1_budget2_reward_head():
    """b = 2 with the composite reward (coverage and the sigmoid head on M_p's hidden state):
    round 2's reward takes the head at lh_d from the round's own target pass; r_t sits where
    one covered keyword plus the head decides, so all outcomes occur."""
    wl = synth.scaled(synth.TINY, batch=2, max_new=20, r_t=0.42, reward_head=True)
    t_host = synth.model_weights(wl, "target", device="host")
    tgt = oracle.Transformer(wl.target, t_host)
    p = synth.prompts(wl)
    kw = np.stack([np.array(greedy_chain(tgt, p[b].tolist(), 12)[1:12:4], np.int32)
                   for b in range(wl.batch)])
    s = make_setup(wl, keywords=kw)
    eng, states, rep, adopted, n = run_parity(s, steps=20, tol=TOL32, tol_r=TOL32,
                                              step1_budget=2)
    tokens_match(eng, states)
    print("budget-2 head report:", rep)
    assert rep.get("round2", 0) > 0, rep


def test_tiny_speculative_sampling_with_step1_budget2():
    """Speculative-sampling validation (f1) together with the Step-1 budget b = 2 (f2): the
    acceptance counts come from the draws, round 2 from the verify row of beam 1."""
    wl = synth.scaled(synth.TINY, batch=2, max_new=16, r_t=0.6)
    t_host = synth.model_weights(wl, "target", device="host")
    tgt = oracle.Transformer(wl.target, t_host)
    p = synth.prompts(wl)
    kw = np.stack([np.array(greedy_chain(tgt, p[b].tolist(), 12)[2:12:4], np.int32)
                   for b in range(wl.batch)])
    s = make_setup(wl, keywords=kw)
    eng, states, rep, adopted, n = run_parity(s, steps=16, tol=TOL32, tol_r=TOL32,
                                              acceptance=1, seed=11, step1_budget=2)
    tokens_match(eng, states)
    print("speculative + budget-2 report:", rep)


def test_small_bf16_step1_budget2():
    """b = 2 on the bf16 path (12-layer target, 4-layer draft, 8 prompts)."""
    wl = synth.scaled(synth.SMALL, max_new=10)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=10, tol=TOL16, tol_r=TOL16,
                                              step1_budget=2)
    tokens_match(eng, states)
    print("small budget-2 report:", rep, "adopted:", len(adopted))


def test_tiny_cdlh_appx_on_the_same_kernels():
    """Alg. 2 CDLH-appx on the GPU path: M_q's lookaheads are never accepted (a_t, r_t above
    any score), so every step emits c_{b*}: the CDLH-appx token of the oracle's Alg. 2 with
    M_q as the lookahead model, step by step and over the whole generation."""
    wl = synth.scaled(synth.TINY, a_t=2.0, r_t=2.0, max_new=10)
    s = make_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=10, tol=TOL32, tol_r=TOL32)
    assert n == wl.max_new
    tokens_match(eng, states)
    tgt = oracle.Transformer(wl.target, s.t_host)
    drf = oracle.Transformer(wl.draft, s.d_host)
    run = run_params(wl)
    for b in range(wl.batch):
        ref = oracle.cdlh_generate(tgt, drf, drf, s.prompts[b].tolist(), s.keywords[b].tolist(),
                                   run, s.w_head)
        assert states[b].T == ref.T
