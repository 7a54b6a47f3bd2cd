"""The C-ABI library loads, exports every symbol include/cdsl.h declares, and validates its
host-side arguments (no GPU needed: these calls launch nothing)."""
import ctypes
import os
import re

import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def cdsl():
    from paper_2412_10418_gb300 import build as b
    b.build()
    import paper_2412_10418_gb300 as pkg
    return pkg


def declared_symbols():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            src = open(os.path.join(ROOT, "include", h)).read()
            names |= set(re.findall(r"CDSL_API[^;(]*?\b(cdsl_\w+)\s*\(", src))
    return names


def test_exports_every_declared_symbol(cdsl):
    names = declared_symbols()
    assert {"cdsl_init", "cdsl_lookahead", "cdsl_verify", "cdsl_select", "cdsl_step"} <= names
    lib = ctypes.CDLL(cdsl.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    # the binding declares exactly the exported entry points
    assert set(cdsl.EXPORTS) <= names


def cfgs(cdsl, wl=synth.TINY, **run_kw):
    t = cdsl.model_cfg(wl.target, wl.dtype)
    d = cdsl.model_cfg(wl.draft, wl.dtype)
    kw = dict(batch=wl.batch, k=wl.k, d=wl.d, max_prompt=wl.prompt_len, max_new=wl.max_new,
              n_keywords=wl.n_keywords, a_t=wl.a_t, r_t=wl.r_t, reward_head=wl.reward_head)
    kw.update(run_kw)
    return t, d, cdsl.run_cfg(**kw)


def test_num_weights(cdsl):
    t, d, _ = cfgs(cdsl)
    assert cdsl.cdsl_num_weights(t) == len(synth.TINY.target.weight_specs())
    assert cdsl.cdsl_num_weights(d) == len(synth.TINY.draft.weight_specs())


def test_workspace_size_grows_with_work(cdsl):
    t, d, r = cfgs(cdsl)
    n1 = cdsl.cdsl_workspace_size(t, d, r)
    t2, d2, r2 = cfgs(cdsl, batch=4, k=8, d=6, max_new=64)
    n2 = cdsl.cdsl_workspace_size(t2, d2, r2)
    assert 0 < n1 < n2 and n1 % 256 == 0
    # 7B-shaped target: the KV pool alone is 32 layers * 2 * 8 * 128 * 2 B per position
    wl = synth.SEVEN_B
    t7, d7, r7 = cfgs(cdsl, wl)
    n7 = cdsl.cdsl_workspace_size(t7, d7, r7)
    assert n7 > (wl.prompt_len + wl.max_new) * 32 * 2 * 8 * 128 * 2


@pytest.mark.parametrize("field,value,msg", [
    ("head_dim", 96, "head_dim"),
    ("n_kv_heads", 3, "n_kv_heads"),
    ("dtype", 7, "dtype"),
    ("d_model", 100, "d_model"),
])
def test_bad_model_config(cdsl, field, value, msg):
    t, d, r = cfgs(cdsl)
    setattr(t, field, value)
    with pytest.raises(cdsl.CdslError) as e:
        cdsl.cdsl_workspace_size(t, d, r)
    assert e.value.code == 1 and msg in str(e.value)


@pytest.mark.parametrize("field,value", [("k", 0), ("k", 17), ("d", 0), ("n_keywords", 33),
                                         ("page_size", 48), ("batch", 0), ("acceptance", 2),
                                         ("step1_budget", 3), ("step1_budget", -1)])
def test_bad_run_config(cdsl, field, value):
    t, d, r = cfgs(cdsl)
    setattr(r, field, value)
    with pytest.raises(cdsl.CdslError) as e:
        cdsl.cdsl_workspace_size(t, d, r)
    assert e.value.code == 1


def test_vocab_and_dtype_must_match(cdsl):
    t, d, r = cfgs(cdsl)
    d.vocab = 256
    with pytest.raises(cdsl.CdslError, match="vocab"):
        cdsl.cdsl_workspace_size(t, d, r)
    t, d, r = cfgs(cdsl)
    d.dtype = 1
    with pytest.raises(cdsl.CdslError, match="dtype"):
        cdsl.cdsl_workspace_size(t, d, r)


def test_init_rejects_before_touching_the_device(cdsl):
    """cdsl_init validates everything on the host first: NULL weights, NULL workspace,
    a missing reward head."""
    t, d, r = cfgs(cdsl)
    lib = cdsl.lib()
    ctx = ctypes.c_void_p(0)
    nt = cdsl.cdsl_num_weights(t)
    nd = cdsl.cdsl_num_weights(d)
    tw = (ctypes.c_void_p * nt)(*([None] * nt))
    dw = (ctypes.c_void_p * nd)(*([None] * nd))
    code = lib.cdsl_init(ctypes.byref(t), tw, ctypes.byref(d), dw, ctypes.byref(r), None,
                         None, 0, None, ctypes.byref(ctx))
    assert code == 1 and "workspace" in cdsl.cdsl_last_error(None)
    fake = (ctypes.c_void_p * nt)(*([4096] * nt))
    fake_d = (ctypes.c_void_p * nd)(*([4096] * nd))
    code = lib.cdsl_init(ctypes.byref(t), tw, ctypes.byref(d), fake_d, ctypes.byref(r), None,
                         1 << 20, 1 << 30, None, ctypes.byref(ctx))
    assert code == 1 and "weight" in cdsl.cdsl_last_error(None)
    r.reward_head = 1
    code = lib.cdsl_init(ctypes.byref(t), fake, ctypes.byref(d), fake_d, ctypes.byref(r), None,
                         1 << 20, 1 << 30, None, ctypes.byref(ctx))
    assert code == 1 and "reward" in cdsl.cdsl_last_error(None)
    assert ctx.value is None


def test_step1_budget_2_adds_the_round_buffers(cdsl):
    """Budget 2 carves the Step-1 round's KV tail regions (d+2 target and d+1 draft slots per
    prompt, every layer) and its d+2-row target pass on top of budget 1."""
    wl = synth.scaled(synth.TINY, k=1)   # one beam: the round's d+2 rows exceed the d+1 verify rows
    t, d, r1 = cfgs(cdsl, wl, step1_budget=1)
    _, _, r2 = cfgs(cdsl, wl, step1_budget=2)
    n1, n2 = cdsl.cdsl_workspace_size(t, d, r1), cdsl.cdsl_workspace_size(t, d, r2)
    tails = 4 * 2 * (wl.target.n_layers * (wl.d + 2) * wl.target.n_kv_heads * wl.target.head_dim
                     + wl.draft.n_layers * (wl.d + 1) * wl.draft.n_kv_heads * wl.draft.head_dim)
    assert n2 - n1 >= tails * wl.batch


def test_get_step1_needs_a_context(cdsl):
    assert cdsl.lib().cdsl_get_step1(None, None, None, None) == 1   # CDSL_EINVAL


@pytest.mark.parametrize("R,K,N,offset", [
    (0, 768, 32000, 0),       # no rows
    (9, 768, 32000, 0),       # more rows than the fixed scratch holds
    (4, 8200, 1000, 0),       # K beyond 8192
    (4, 4, 1000, 0),          # K below 8
    (4, 772, 1000, 0),        # K not a multiple of 8
    (4, 768, 0, 0),           # no outputs
    (4, 768, 32769, 0),       # N beyond 32768
    (4, 768, 1000, 8),        # misaligned pointers
])
def test_gemv_noalloc_rejects_before_any_cuda_call(cdsl, R, K, N, offset):
    """Sizes beyond the fixed scratch and misaligned pointers return CDSL_EINVAL from the
    host-side checks, before the library touches CUDA (the pointers are never dereferenced)."""
    lib = cdsl.lib()
    base = 1 << 20
    rc = lib.cdsl_gemv_noalloc(base + offset, N, K, base + 4096 + offset, R,
                               base + 8192 + offset, None)
    assert rc == cdsl.CDSL_EINVAL
    assert "cdsl_gemv_noalloc" in cdsl.cdsl_last_error(None)
    assert lib.cdsl_gemv_noalloc(None, 1000, 768, base, 4, base, None) == cdsl.CDSL_EINVAL


def test_gemv_noalloc_binding_checks_tensors(cdsl):
    """The binding refuses dtypes, shapes, layouts and devices the C ABI cannot check."""
    import torch
    w = torch.zeros((64, 32), dtype=torch.bfloat16)
    x = torch.zeros((2, 32), dtype=torch.float32)
    y = torch.zeros((2, 64), dtype=torch.float32)
    cases = [(w.float(), x, y, "bfloat16"), (w, x.double(), y, "float32"),
             (w, torch.zeros((2, 16)), y, "shapes"), (w, x, torch.zeros((2, 63)), "shapes"),
             (w, torch.zeros((32, 2)).t(), y, "contiguous"), (w, x, y, "CUDA device")]
    for ww, xx, yy, msg in cases:
        with pytest.raises(cdsl.CdslError) as e:
            cdsl.cdsl_gemv_noalloc(ww, xx, yy)
        assert e.value.code == cdsl.CDSL_EINVAL and msg in str(e.value), (msg, str(e.value))
