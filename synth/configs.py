"""Model shapes and seeded workload recipes (pure data, no arithmetic of the method).

Shapes are Llama-3 style decoders: L layers, width d, H_q query / H_kv KV heads of
dimension d_h, SwiGLU width d_f, vocabulary V (0 = no LM head). A mask unit is a
whole GQA group (one KV head with its g = H_q/H_kv query heads) or a block of
``chan_unit`` SwiGLU channels (Table 1 of the paper: 1,024-channel groups; the
single-layer case uses single channels because 1,408 is not a multiple of 1,024).
"""
from __future__ import annotations

from dataclasses import dataclass, field


@dataclass(frozen=True)
class ModelShape:
    L: int
    d: int
    Hq: int
    Hkv: int
    dh: int
    df: int
    vocab: int
    chan_unit: int
    eps: float = 1e-5
    rope_theta: float = 500000.0
    seed: int = 0
    quant_group: int = 0  # INT8 scale granularity: 0 = one scale per output row, else columns per scale

    @property
    def g(self) -> int:
        return self.Hq // self.Hkv

    @property
    def n_chan_units(self) -> int:
        return self.df // self.chan_unit

    @property
    def n_units(self) -> int:
        return self.Hkv + self.n_chan_units


@dataclass(frozen=True)
class MaskRecipe:
    mask_seed: int
    budget: float = 0.57
    r_lo: float = 0.35
    r_hi: float = 0.85


@dataclass(frozen=True)
class Workload:
    name: str
    shape: ModelShape
    masks: tuple = field(default_factory=tuple)
    t_prior: int = 0
    steps: int = 0
    kv_seed: int = 7
    x_seed: int = 11
    prompt_lens: tuple = ()
    n_turns: int = 1
    p_dense: float = 0.0


LAYER1 = ModelShape(L=1, d=512, Hq=8, Hkv=2, dh=64, df=1408, vocab=0, chan_unit=1)
LLAMA3_8B = ModelShape(L=32, d=4096, Hq=32, Hkv=8, dh=128, df=14336, vocab=128256, chan_unit=1024)
LLAMA3_70B = ModelShape(L=80, d=8192, Hq=64, Hkv=8, dh=128, df=28672, vocab=128256, chan_unit=1024)

MASK_SEEDS = tuple(1000 + k for k in range(5))

# The five workloads of the build's scope.
CFG1 = Workload("layer1_decode", LAYER1, masks=(MaskRecipe(MASK_SEEDS[0]),), t_prior=128, steps=16)
CFG2 = Workload("llama3_8b_decode", LLAMA3_8B, masks=tuple(MaskRecipe(s) for s in MASK_SEEDS),
                t_prior=2048, steps=128)
CFG3 = Workload("llama3_70b_decode", LLAMA3_70B, masks=(MaskRecipe(MASK_SEEDS[0]),),
                t_prior=4096, steps=128)
CFG4 = Workload("llama3_8b_prefill", LLAMA3_8B, masks=tuple(MaskRecipe(s) for s in MASK_SEEDS),
                steps=32, prompt_lens=(512, 2048, 8192))
CFG5 = Workload("llama3_70b_mixed_turns", LLAMA3_70B, masks=tuple(MaskRecipe(s) for s in MASK_SEEDS),
                steps=64, n_turns=16, p_dense=0.1, prompt_lens=(256, 2048))

CONFIGS = {1: CFG1, 2: CFG2, 3: CFG3, 4: CFG4, 5: CFG5}


def tiny_shape(L=2, d=128, Hq=4, Hkv=2, dh=32, df=192, vocab=64, chan_unit=16, seed=3, quant_group=0) -> ModelShape:
    """A small shape for fast oracle pins."""
    return ModelShape(L=L, d=d, Hq=Hq, Hkv=Hkv, dh=dh, df=df, vocab=vocab, chan_unit=chan_unit, seed=seed,
                      quant_group=quant_group)
