"""In-graph kernel timing (cdsl_profile mode 2) on the GPU: the per-launch charges of a
graph-replayed step are disjoint, so per step they add up to no more than the span from the
first stamped entry to the last stamped exit, which itself lies inside the step's wall time;
every projection and attention launch of the step carries a record; the attention kernel's
own byte count matches the keys the step's passes read."""
import pytest

import synth
from cdsl_parity import make_engine, make_setup

pytestmark = pytest.mark.gpu


def test_in_graph_charges_fit_the_step():
    import torch
    import paper_2412_10418_gb300 as cdsl

    wl = synth.scaled(synth.SMALL, batch=2, max_new=40)
    s = make_setup(wl)
    eng = make_engine(s)
    eng.step()
    eng.stream.synchronize()
    n = 4
    cdsl.cdsl_profile(eng.ctx, cdsl.PROFILE_IN_GRAPH)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    wall = 0.0
    for _ in range(n):
        e0.record(eng.stream)
        eng.step()                     # synchronizes (mode 2 folds the stamps after the step)
        e1.record(eng.stream)
        e1.synchronize()
        wall += e0.elapsed_time(e1)
    prof = {name: cdsl.cdsl_get_profile(eng.ctx, impl) for impl, name in cdsl.KERNEL_CLASSES.items()}
    steps = cdsl.cdsl_get_profile(eng.ctx, cdsl.STAMPED_STEPS)
    launches = cdsl.cdsl_get_profile_launches(eng.ctx)
    cdsl.cdsl_profile(eng.ctx, cdsl.PROFILE_OFF)
    assert steps["launches"] == n
    charged = sum(v["ms"] for v in prof.values())
    assert 0 < charged <= steps["ms"] * (1 + 1e-9) <= wall
    # projections: 5 GEMMs per layer per pass (QKV, O, gate/up, down) + the LM head
    t_l, d_l = wl.target.n_layers, wl.draft.n_layers
    gemms = wl.d * (4 * d_l + 1) + (4 * t_l + 1)
    tc = prof["gemm_tc"]
    assert tc["launches"] == n * gemms and tc["ms"] > 0 and tc["bytes"] > 0
    att = prof["attention"]
    assert att["launches"] == n * (wl.d * d_l + t_l) and att["ms"] > 0
    # every attention launch counted at least the K and V of its prompts' prefixes once
    hd = wl.target.head_dim
    min_keys = wl.batch * wl.prompt_len
    for cls, ms, by, fl in launches:
        if cls == 3:
            assert by >= min_keys * min(wl.target.n_kv_heads, wl.draft.n_kv_heads) * hd * 8
    assert eng.status() == 0
