"""Error reporting of the C ABI on a live context (GPU): calls out of order return
CDSL_ESTATE before anything is launched and leave the context usable; the device status word
stays CDSL_OK through correct use."""
import pytest

import synth
from cdsl_parity import make_setup

pytestmark = pytest.mark.gpu


def engine(s, prefilled=True):
    import torch
    import paper_2412_10418_gb300 as cdsl
    wl = s.wl
    tw = synth.to_torch(s.t_host, wl.dtype)
    dw = synth.to_torch(s.d_host, wl.dtype)
    eng = cdsl.Engine(wl.target, wl.draft, wl.dtype,
                      [tw[n] for n, _ in wl.target.weight_specs()],
                      [dw[n] for n, _ in wl.draft.weight_specs()],
                      batch=wl.batch, k=wl.k, d=wl.d, max_prompt=wl.prompt_len,
                      max_new=wl.max_new, n_keywords=s.keywords.shape[1], a_t=wl.a_t, r_t=wl.r_t)
    if prefilled:
        eng.prefill(torch.from_numpy(s.prompts), s.lens, torch.from_numpy(s.keywords))
    return eng


def test_calls_out_of_order_are_refused():
    import paper_2412_10418_gb300 as cdsl
    s = make_setup(synth.scaled(synth.SMALL, batch=1, max_new=8))

    def refused(fn, what):
        with pytest.raises(cdsl.CdslError) as e:
            fn()
        assert e.value.code == cdsl.CDSL_ESTATE, (what, str(e.value))

    eng = engine(s, prefilled=False)
    refused(eng.lookahead, "lookahead before prefill")
    refused(eng.step, "step before prefill")
    refused(eng.verify, "verify before prefill")
    eng.close()

    eng = engine(s)
    refused(eng.verify, "verify before lookahead")
    refused(eng.select, "select before verify")
    eng.lookahead()
    refused(eng.lookahead, "lookahead twice")
    refused(eng.step, "step between lookahead and verify")
    refused(eng.select, "select before verify")
    eng.verify()
    refused(eng.verify, "verify twice")
    refused(eng.step, "step between verify and select")
    eng.select()
    refused(eng.select, "select twice")
    # the refusals launched nothing: the context goes on stepping normally
    for _ in range(3):
        eng.step()
    assert eng.status() == cdsl.CDSL_OK
    assert eng.counters()[0] >= 4
    eng.close()


def test_expired_waits_latch_etimeout_and_the_device_stays_usable():
    """With a wait limit of 0 every bounded wait of the tensor-core GEMM and attention that is
    not already satisfied gives up: the step latches CDSL_ETIMEOUT, every block winds down
    (its own copies and MMAs drained, its cluster barriers met) and the launches end, so the
    CUDA context stays usable; a new context on the same device then matches the oracle."""
    import torch
    import paper_2412_10418_gb300 as cdsl
    from cdsl_parity import run_parity

    s = make_setup(synth.scaled(synth.SMALL, batch=1, max_new=8))
    eng = engine(s)
    eng.step()
    assert eng.status() == cdsl.CDSL_OK
    cdsl.cdsl_set_wait_limit(eng.ctx, 0)
    eng.step()                                  # the call itself succeeds: the error is on the device
    assert eng.status() == cdsl.CDSL_ETIMEOUT
    torch.cuda.synchronize()                    # no sticky CUDA error: the launches ended
    eng.close()

    eng2, states, rep, adopted, n = run_parity(s, steps=3, tol=2e-2, tol_r=2e-2)
    assert n == 3 and eng2.status() == cdsl.CDSL_OK
    eng2.close()


def test_expired_waits_in_the_large_row_gemm_and_tensor_core_attention():
    """The same with k = 8, d = 8: 72 verify rows, so the projections run the large-row GEMM
    (more than 64 rows: stream-K with the contributors' shared fixup, whose counter waits are
    bounded too) and the verify attention runs on the tensor cores (72 query vectors per KV
    head). Every block gives up or finishes, the launches end, and a new context on the same
    device matches the oracle at this shape."""
    import torch
    import paper_2412_10418_gb300 as cdsl
    from cdsl_parity import run_parity

    s = make_setup(synth.scaled(synth.SMALL, batch=1, k=8, d=8, max_new=8))
    eng = engine(s)
    eng.step()
    assert eng.status() == cdsl.CDSL_OK
    cdsl.cdsl_set_wait_limit(eng.ctx, 0)
    eng.step()
    assert eng.status() == cdsl.CDSL_ETIMEOUT
    torch.cuda.synchronize()
    eng.close()

    eng2, states, rep, adopted, n = run_parity(s, steps=2, tol=2e-2, tol_r=2e-2)
    assert n == 2 and eng2.status() == cdsl.CDSL_OK
    eng2.close()
