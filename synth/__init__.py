"""Seeded synthetic inputs for the CDSL lookahead step.

This module is the only code shared by the CUDA path's callers (tests, bench, smoke) and the
oracle. It produces inputs only -- model shapes, random-init weights, prompt token ids, keyword
ids and the reward-head vector -- and holds none of the method's arithmetic.

Recipe (stands in for the paper's CommonGen / HH-RLHF prompts and its OPT/Bloomz/Qwen weights,
none of which exist here; Sec. 4.1-4.2 and App. C describe the real workloads):

* Weights: every matrix N(0, 0.02), every RMSNorm gain 1.0, no biases, untied LM head.
  Small models are drawn with numpy ``default_rng([seed, stream])`` (platform independent, so
  stored fixtures can be regenerated anywhere). 7B/13B-shaped models are drawn on the GPU with
  torch's Philox generator because the host draw would take minutes; a CPU copy is handed to
  the oracle where a test needs one.
* bf16 models: the fp32 draw is rounded once to bf16 (round to nearest even); both sides read
  the same bf16 bits.
* Prompts: ``uniform`` ids in [0, V) or ``zipf`` ids: rank ~ Zipf(1.1) truncated to [1, V] by
  rejection, id = rank - 1 (frequent ids are small, as in BPE vocabularies).
* Keywords: per prompt, ``n_keywords`` distinct ids drawn uniformly from [0, V).
* Reward head: w ~ N(0, 0.02) of length d_model (the semantic-reward stand-in for the
  trained reward model of Sec. 4.1).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Tuple

import numpy as np

# Stream ids for numpy's SeedSequence: one independent stream per kind of input.
_STREAM_TARGET, _STREAM_DRAFT, _STREAM_PROMPTS, _STREAM_KEYWORDS, _STREAM_HEAD = range(5)

DTYPE_F32 = "f32"
DTYPE_BF16 = "bf16"


@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Shape of a pre-norm (Llama-style) decoder-only transformer."""

    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    d_ffn: int
    vocab: int
    rope_theta: float = 10000.0
    norm_eps: float = 1e-5

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_heads

    def weight_specs(self) -> List[Tuple[str, Tuple[int, ...]]]:
        """Names and shapes of every weight, in the order the C ABI takes them.

        Matrices are [out_features, in_features] row-major (y = x W^T)."""
        D, F, V, hd = self.d_model, self.d_ffn, self.vocab, self.head_dim
        specs: List[Tuple[str, Tuple[int, ...]]] = [("embed", (V, D))]
        for l in range(self.n_layers):
            specs += [
                (f"l{l}.attn_norm", (D,)),
                (f"l{l}.wq", (self.n_heads * hd, D)),
                (f"l{l}.wk", (self.n_kv_heads * hd, D)),
                (f"l{l}.wv", (self.n_kv_heads * hd, D)),
                (f"l{l}.wo", (D, self.n_heads * hd)),
                (f"l{l}.ffn_norm", (D,)),
                (f"l{l}.w_gate", (F, D)),
                (f"l{l}.w_up", (F, D)),
                (f"l{l}.w_down", (D, F)),
            ]
        specs += [("final_norm", (D,)), ("lm_head", (V, D))]
        return specs

    def n_params(self) -> int:
        return int(sum(int(np.prod(s)) for _, s in self.weight_specs()))


@dataclasses.dataclass(frozen=True)
class Workload:
    """One CDSL-k decoding workload: models, batch, beams, lookahead, reward."""

    name: str
    target: ModelShape
    draft: ModelShape
    dtype: str
    batch: int
    prompt_len: int
    prompt_dist: str
    k: int
    d: int
    max_new: int
    n_keywords: int
    reward_head: bool  # composite reward: 0.5 * coverage + 0.5 * sigmoid(w . h_last)
    a_t: float = 0.3
    r_t: float = 0.3
    seed: int = 0


TINY = Workload(
    name="tiny-fp32", dtype=DTYPE_F32,
    target=ModelShape(n_layers=2, d_model=256, n_heads=4, n_kv_heads=4, d_ffn=688, vocab=512),
    draft=ModelShape(n_layers=1, d_model=128, n_heads=2, n_kv_heads=2, d_ffn=344, vocab=512),
    batch=1, prompt_len=32, prompt_dist="uniform", k=4, d=4, max_new=16, n_keywords=3,
    reward_head=False)

SMALL = Workload(
    name="small-bf16", dtype=DTYPE_BF16,
    target=ModelShape(n_layers=12, d_model=768, n_heads=12, n_kv_heads=12, d_ffn=3072, vocab=32000),
    draft=ModelShape(n_layers=4, d_model=512, n_heads=8, n_kv_heads=8, d_ffn=2048, vocab=32000),
    batch=8, prompt_len=128, prompt_dist="zipf", k=4, d=4, max_new=64, n_keywords=5,
    reward_head=False)

DRAFT_1B = ModelShape(n_layers=16, d_model=2048, n_heads=16, n_kv_heads=4, d_ffn=5504, vocab=32000)

SEVEN_B = Workload(
    name="7b-bf16", dtype=DTYPE_BF16,
    target=ModelShape(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=8, d_ffn=11008, vocab=32000),
    draft=DRAFT_1B,
    batch=1, prompt_len=512, prompt_dist="zipf", k=4, d=4, max_new=128, n_keywords=5,
    reward_head=True)

THIRTEEN_B = Workload(
    name="13b-bf16", dtype=DTYPE_BF16,
    target=ModelShape(n_layers=40, d_model=5120, n_heads=40, n_kv_heads=8, d_ffn=13824, vocab=32000),
    draft=DRAFT_1B,
    batch=4, prompt_len=1024, prompt_dist="zipf", k=8, d=6, max_new=256, n_keywords=5,
    reward_head=True)

# Two layers of each 7B-shaped model: the same projection shapes (the gate/up weights alone,
# 180 MB, exceed the 129 MB L2) in about 1 GB of device memory, for kernel profiling captures.
SEVEN_B_SLICE = Workload(
    name="7b-2layer-bf16", dtype=DTYPE_BF16,
    target=dataclasses.replace(SEVEN_B.target, n_layers=2),
    draft=dataclasses.replace(DRAFT_1B, n_layers=2),
    batch=1, prompt_len=512, prompt_dist="zipf", k=4, d=4, max_new=128, n_keywords=5,
    reward_head=True)

# Two layers of each 13B-shaped model, in the 13B launch configuration (4 prompts of 1024
# tokens, k = 8, d = 6: 224 verify rows): full-size parity checks.
THIRTEEN_B_SLICE = Workload(
    name="13b-2layer-bf16", dtype=DTYPE_BF16,
    target=dataclasses.replace(THIRTEEN_B.target, n_layers=2),
    draft=dataclasses.replace(DRAFT_1B, n_layers=2),
    batch=4, prompt_len=1024, prompt_dist="zipf", k=8, d=6, max_new=256, n_keywords=5,
    reward_head=True)

WORKLOADS: Dict[str, Workload] = {w.name: w for w in (TINY, SMALL, SEVEN_B, THIRTEEN_B,
                                                      SEVEN_B_SLICE, THIRTEEN_B_SLICE)}


def scaled(w: Workload, **changes) -> Workload:
    """A copy of a workload with some fields replaced (smaller shapes for fast tests)."""
    return dataclasses.replace(w, **changes)


# ----------------------------------------------------------------------------------------
# bf16 storage helpers (data conversion of inputs; not part of the method)
# ----------------------------------------------------------------------------------------

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (round to nearest, ties to even); returns uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = ((u >> 16) & 1) + np.uint32(0x7FFF)
    return ((u + rounding) >> 16).astype(np.uint16)


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.default_rng([int(seed), int(stream)])


# ----------------------------------------------------------------------------------------
# Weights
# ----------------------------------------------------------------------------------------

def host_weights(shape: ModelShape, dtype: str, seed: int, stream: int) -> Dict[str, np.ndarray]:
    """Draw a model's weights on the host with numpy.

    Returns name -> array: float32 for ``f32`` models, uint16 bf16 bit patterns for ``bf16``."""
    rng = _rng(seed, stream)
    out: Dict[str, np.ndarray] = {}
    for name, shp in shape.weight_specs():
        if len(shp) == 1:
            w = np.ones(shp, dtype=np.float32)
        else:
            w = rng.standard_normal(shp, dtype=np.float32)
            w *= np.float32(0.02)
        out[name] = w if dtype == DTYPE_F32 else f32_to_bf16_bits(w)
    return out


def device_weights(shape: ModelShape, dtype: str, seed: int, stream: int, device="cuda"):
    """Draw a model's weights directly on a torch device with torch's Philox generator.

    Returns name -> torch tensor (float32 or bfloat16). Used for 7B/13B-sized models."""
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(int(seed) * 1000003 + int(stream))
    tdt = torch.float32 if dtype == DTYPE_F32 else torch.bfloat16
    out = {}
    for name, shp in shape.weight_specs():
        if len(shp) == 1:
            out[name] = torch.ones(shp, dtype=tdt, device=device)
        else:
            w = torch.randn(shp, generator=g, device=device, dtype=torch.float32)
            w.mul_(0.02)
            out[name] = w.to(tdt)
            del w
    return out


def to_torch(weights: Dict[str, np.ndarray], dtype: str, device="cuda"):
    """Move host weights (from host_weights) to torch tensors on a device, bit-exactly."""
    import torch

    out = {}
    for name, w in weights.items():
        if dtype == DTYPE_F32:
            t = torch.from_numpy(np.ascontiguousarray(w))
        else:
            t = torch.from_numpy(np.ascontiguousarray(w).view(np.int16)).view(torch.bfloat16)
        out[name] = t.to(device)
    return out


def to_host(weights) -> Dict[str, np.ndarray]:
    """torch tensors -> host numpy arrays in the oracle's storage format (f32 or bf16 bits)."""
    import torch

    out = {}
    for name, t in weights.items():
        t = t.detach().to("cpu")
        if t.dtype == torch.bfloat16:
            out[name] = t.view(torch.int16).numpy().view(np.uint16)
        else:
            out[name] = t.numpy()
    return out


def model_weights(w: Workload, which: str, device: str = "host"):
    """Weights of the workload's target or draft model.

    device="host": numpy dict (always numpy draw for small models).
    device="cuda": torch dict; small models are the numpy draw copied over, 7B/13B-sized models
    are drawn on the GPU."""
    shape = w.target if which == "target" else w.draft
    stream = _STREAM_TARGET if which == "target" else _STREAM_DRAFT
    big = shape.n_params() > 400_000_000 or shape.d_model >= 2048
    if device == "host":
        if big:
            raise ValueError("7B/13B-sized weights are drawn on the GPU; use device='cuda' then to_host()")
        return host_weights(shape, w.dtype, w.seed, stream)
    if big:
        return device_weights(shape, w.dtype, w.seed, stream, device=device)
    return to_torch(host_weights(shape, w.dtype, w.seed, stream), w.dtype, device=device)


# ----------------------------------------------------------------------------------------
# Prompts, keywords, reward head
# ----------------------------------------------------------------------------------------

def prompts(w: Workload) -> np.ndarray:
    """[batch, prompt_len] int32 prompt token ids."""
    rng = _rng(w.seed, _STREAM_PROMPTS)
    V = w.target.vocab
    n = w.batch * w.prompt_len
    if w.prompt_dist == "uniform":
        ids = rng.integers(0, V, size=n)
    elif w.prompt_dist == "zipf":
        ids = np.empty(n, dtype=np.int64)
        filled = 0
        while filled < n:
            r = rng.zipf(1.1, size=2 * (n - filled))
            r = r[r <= V]
            take = min(len(r), n - filled)
            ids[filled:filled + take] = r[:take] - 1
            filled += take
    else:
        raise ValueError(w.prompt_dist)
    return ids.reshape(w.batch, w.prompt_len).astype(np.int32)


def keywords(w: Workload) -> np.ndarray:
    """[batch, n_keywords] int32 distinct keyword ids per prompt."""
    rng = _rng(w.seed, _STREAM_KEYWORDS)
    return np.stack([rng.choice(w.target.vocab, size=w.n_keywords, replace=False)
                     for _ in range(w.batch)]).astype(np.int32)


def reward_head(w: Workload) -> np.ndarray:
    """[d_model] float32 linear reward-head vector (zeros when the workload has no head)."""
    if not w.reward_head:
        return np.zeros(w.target.d_model, dtype=np.float32)
    rng = _rng(w.seed, _STREAM_HEAD)
    return (rng.standard_normal(w.target.d_model, dtype=np.float32) * np.float32(0.02)).astype(np.float32)
