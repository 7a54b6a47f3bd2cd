"""CUDA path vs the oracle at the full sizes of the 7B and 13B workloads and of the verify
sweep, in the launch configurations bench.py times (same projection and attention shapes,
batch, prompt lengths, k, d and verify rows), with each model cut to two layers so that the
fp64 oracle finishes: every output of each step is compared element by element (tolerance
2e-2 for bf16 weights, exact token ids and decisions), as in test_gpu_parity.py."""
import numpy as np
import pytest

import synth
from cdsl_parity import Setup, make_engine, run_parity

pytestmark = pytest.mark.gpu

TOL16 = 2e-2


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2412_10418_gb300 import build
    build.build()


def full_size_setup(wl):
    """Device-drawn weights (the bench's), their host copies for the oracle."""
    tw = synth.model_weights(wl, "target", device="cuda")
    dw = synth.model_weights(wl, "draft", device="cuda")
    s = Setup(wl, synth.to_host(tw), synth.to_host(dw), synth.prompts(wl),
              [wl.prompt_len] * wl.batch, synth.keywords(wl), synth.reward_head(wl))
    return s, (tw, dw)


def check(wl, steps, page_size=64):
    s, tdw = full_size_setup(wl)
    eng, states, rep, adopted, n = run_parity(s, steps=steps, tol=TOL16, tol_r=TOL16,
                                              torch_weights=tdw, page_size=page_size,
                                              keep_widened=False)
    t, nt = eng.tokens()
    t, nt = t.cpu().numpy(), nt.cpu().numpy()
    for b, st in enumerate(states):
        want = st.prompt + st.T
        assert nt[b] == len(want) and t[b, :nt[b]].tolist() == want
    print(wl.name, f"k={wl.k} d={wl.d} prompt={wl.prompt_len} B={wl.batch}:", rep,
          "near ties adopted:", len(adopted))
    eng.close()


def test_7b_shapes_bench_configuration():
    """7B-shaped target and 1B-shaped draft (GQA 32/8 and 16/4, FFN 11008 / 5504, V 32000),
    one 512-token prompt, k = 4, d = 4: 20 verify rows, composite reward."""
    check(synth.SEVEN_B_SLICE, steps=3)


def test_7b_full_depth_bench_configuration():
    """The whole 7B workload as bench.py times it (32-layer target, 16-layer draft, the
    512-token prompt, k = 4, d = 4), two steps (the second over the first one's committed
    K/V): prefill roots, draft tokens and log q, every verify logit (bf16 error accumulated
    over all 32 layers, still within 2e-2: measured 2.6e-4), n_b, the rewards, b*, the state
    and the emission against the oracle at full depth."""
    check(synth.SEVEN_B, steps=2)


def test_13b_shapes_bench_configuration():
    """13B-shaped target (GQA 40/8, FFN 13824) with the 1B-shaped draft, 4 prompts of 1024
    tokens, k = 8, d = 6: 224 verify rows (two MMAs per K step: hi and lo no longer fit one)."""
    check(synth.THIRTEEN_B_SLICE, steps=2)


@pytest.mark.parametrize("k,d,prefix", [(16, 10, 1024), (2, 2, 4096), (8, 6, 2048)])
def test_verify_sweep_points(k, d, prefix):
    """Points of the verify sweep on the 7B shapes: up to 176 verify rows, up to a 4096-token
    prefix (65 key chunks per pass)."""
    wl = synth.scaled(synth.SEVEN_B_SLICE, k=k, d=d, prompt_len=prefix, max_new=64)
    check(wl, steps=2)
