"""cdsl_gemv_noalloc (the GEMM entry point that allocates no device memory) against an fp64
product computed by torch, and against the step library's own verify pass.

Some callers of this library cannot allocate device memory: host frameworks whose caching
allocator already holds the GPU's memory, real-time loops that must not block on cudaMalloc,
runtimes that forbid device allocation after start-up. cdsl_gemv_noalloc serves them: its
scratch is a fixed array inside the library. The first test checks it against x @ w^T in fp64
over every row count it takes (1..8), outputs that are not a multiple of the 128-row tile,
inputs that are not a multiple of the 256-wide K step and the 8192 K limit, at 2e-5 of the
sum of |x||w| (the hi/lo split of x keeps about 17 bits; the products and sums are fp32).
The second builds a bf16 model whose layers leave the residual stream unchanged (the
attention-output and FFN-down projections are zero), so cdsl_verify's logits are
lm_head(RMSNorm(E[token])) for every verify row; it recomputes those normalized rows in fp32
torch, runs them through cdsl_gemv_noalloc in chunks of at most 8 rows, and compares with the
verify logits, for two rounds of calls in a row. This file is named so that pytest collects
it last."""
import numpy as np
import pytest

import synth
from cdsl_parity import make_engine, make_setup

pytestmark = pytest.mark.gpu

TOL16 = 2e-2   # the bf16 logits tolerance of the parity tests
REL = 2e-5     # of sum_k |x_k| |w_k|: the hi/lo split and fp32 accumulation


@pytest.mark.parametrize("R,K,N", [(1, 768, 1000), (2, 1000, 129), (3, 2048, 3072),
                                   (4, 8192, 4096), (5, 5504, 2048), (6, 1000, 32000),
                                   (7, 8192, 1000), (8, 4096, 32000)])
def test_noalloc_gemv_matches_fp64_product(R, K, N):
    import torch
    from paper_2412_10418_gb300 import build
    build.build()
    import paper_2412_10418_gb300 as cdsl

    g = torch.Generator(device="cpu").manual_seed(1000 * R + K % 997)
    w = (0.02 * torch.randn((N, K), generator=g)).to(torch.bfloat16).cuda()
    x = torch.randn((R, K), generator=g).cuda()
    ref = x.double() @ w.double().t()
    bound = REL * (x.double().abs() @ w.double().abs().t()) + 1e-30
    stream = torch.cuda.current_stream()
    outs = []
    for _ in range(2):                      # two calls in a row share the scratch
        y = torch.full((R, N), float("nan"), dtype=torch.float32, device="cuda")
        cdsl.cdsl_gemv_noalloc(w, x, y, stream.cuda_stream)
        stream.synchronize()
        excess = float(((y.double() - ref).abs() - bound).max())
        assert excess <= 0.0, f"R={R} K={K} N={N}: error exceeds the bound by {excess:.3g}"
        outs.append(y)
    assert torch.equal(outs[0], outs[1])


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
