"""cdsl_gemv_noalloc (the GEMM entry point that allocates no device memory) against the step
library's own verify pass.

Some callers of this library cannot allocate device memory: code that runs while a stream is
captured in global mode, host frameworks whose allocator already holds the GPU's memory, and
latency-critical loops that must not block on cudaMalloc. cdsl_gemv_noalloc serves them: its
scratch is a fixed array inside the library. This test builds a bf16 model whose layers leave
the residual stream unchanged (the attention-output and FFN-down projections are zero), so
cdsl_verify's logits are lm_head(RMSNorm(E[token])) for every verify row. It recomputes those
normalized rows in plain fp32 torch, runs them through cdsl_gemv_noalloc in chunks of at most
8 rows, and compares with the verify logits, for two rounds of calls in a row. This file is
named so that pytest collects it last."""
import numpy as np
import pytest

import synth
from cdsl_parity import make_engine, make_setup

pytestmark = pytest.mark.gpu

TOL16 = 2e-2   # the bf16 logits tolerance of the parity tests


def test_noalloc_gemv_matches_verify_logits():
    import torch
    from paper_2412_10418_gb300 import build
    build.build()
    import paper_2412_10418_gb300 as cdsl

    tshape = synth.ModelShape(n_layers=2, d_model=768, n_heads=12, n_kv_heads=12, d_ffn=3072,
                              vocab=32000)
    wl = synth.scaled(synth.SMALL, batch=1, k=4, d=4, max_new=4, target=tshape)
    s = make_setup(wl)
    for l in range(tshape.n_layers):
        s.t_host[f"l{l}.wo"][:] = 0
        s.t_host[f"l{l}.w_down"][:] = 0
    eng = make_engine(s)
    eng.lookahead()
    V, R = tshape.vocab, wl.k * (wl.d + 1)
    logits = torch.empty((1, wl.k, wl.d + 1, V), dtype=torch.float32, device="cuda")
    eng.verify(logits)
    eng.stream.synchronize()
    want = logits.reshape(R, V)

    roots = eng.roots.cpu().numpy()[0]
    drafts = eng.draft_tok.cpu().numpy()[0]
    rows = [t for i in range(wl.k) for t in [int(roots[i])] + drafts[i].tolist()]
    tw = synth.to_torch(s.t_host, wl.dtype)
    h = tw["embed"].float()[torch.tensor(rows, device="cuda")]
    x = h * torch.rsqrt(h.pow(2).mean(-1, keepdim=True) + tshape.norm_eps) * tw["final_norm"].float()
    w = tw["lm_head"].contiguous()

    stream = torch.cuda.current_stream()
    results = []
    for _ in range(2):                      # two rounds of calls in a row
        ys = []
        for r0 in range(0, R, 8):
            xc = x[r0:r0 + 8].contiguous()
            y = torch.full((xc.shape[0], V), float("nan"), dtype=torch.float32, device="cuda")
            cdsl.cdsl_gemv_noalloc(w, xc, y, stream.cuda_stream)
            ys.append(y)
        stream.synchronize()
        y = torch.cat(ys)
        err = float((y - want).abs().max())
        assert err <= TOL16, f"max |diff| {err}"
        results.append(y)
    assert torch.equal(results[0], results[1])   # fixed-order split-K sum: same bits again

    # sizes beyond the fixed scratch are refused before anything is launched
    big = torch.zeros((9, 768), dtype=torch.float32, device="cuda")
    with pytest.raises(cdsl.CdslError) as e:
        cdsl.cdsl_gemv_noalloc(w, big, torch.empty((9, V), device="cuda"), stream.cuda_stream)
    assert e.value.code == 1 and "R <= 8" in str(e.value)
