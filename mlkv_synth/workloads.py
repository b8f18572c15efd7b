"""Synthetic MLKV decode workloads (shapes, layer->owner maps, lengths, value scales).

The paper measures Pythia-160M / 410M variants on a dummy cache (Sec. 4.5) and lists the
(l, h, m, g) mappings in Table 2; there is no dataset in play, only shapes.  These workloads stand
in for those measurements with seeded random bf16 Q/K/V.  Owner maps are written out literally.

``seq_lens`` counts the new token: a sequence of context L attends positions [0, L).
"""
from dataclasses import dataclass, field

import numpy as np

from . import gen


@dataclass
class Workload:
    name: str
    l: int                 # layers
    h: int                 # query heads per layer
    d: int                 # head dimension
    owner: list            # layer -> owner layer
    g: int                 # KV heads per owner layer
    b: int                 # batch
    L: int                 # context (fixed) or the maximum of a uniform draw
    seed: int
    uniform_len: bool = False
    sigma_q: float = 1.0
    sigma_k: float = 1.0
    sigma_v: float = 1.0
    notes: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def max_seq(self):
        return self.L

    def seq_lens(self):
        if self.uniform_len:
            return gen.gen_seq_lens(self.seed, self.b, self.L)
        return np.full(self.b, self.L, dtype=np.int32)

    def owners(self):
        return sorted(set(int(o) for o in self.owner))


PYTHIA = dict(l=12, h=12, d=64)

_MHA12 = list(range(12))
_PAIRS = [0, 0, 2, 2, 4, 4, 6, 6, 8, 8, 10, 10]
_TRIPLES = [0, 0, 0, 3, 3, 3, 6, 6, 6, 9, 9, 9]
_SIXES = [0, 0, 0, 0, 0, 0, 6, 6, 6, 6, 6, 6]
_ONE = [0] * 12
_LLAMA_FOURS = [0, 0, 0, 0, 4, 4, 4, 4, 8, 8, 8, 8, 12, 12, 12, 12,
                16, 16, 16, 16, 20, 20, 20, 20, 24, 24, 24, 24, 28, 28, 28, 28]


def config(index):
    """The five workloads (1-based index); 5 returns the b=256 sweep, see sweep()."""
    if index == 1:
        return Workload("pythia160m-mlkv6-b1-L128", owner=_PAIRS, g=1, b=1, L=128, seed=1001,
                        **PYTHIA)
    if index == 2:
        return Workload("pythia160m-mlkv2-b64-L2048", owner=_SIXES, g=1, b=64, L=2048,
                        seed=1002, **PYTHIA)
    if index == 3:
        return Workload("pythia160m-gqa4-mlkv4-b128-Lu4096", owner=_TRIPLES, g=4, b=128,
                        L=4096, seed=1003, uniform_len=True, **PYTHIA)
    if index == 4:
        return Workload("llama2-7b-mlkv8-gqa4-b32-L16384", l=32, h=32, d=128,
                        owner=_LLAMA_FOURS, g=8, b=32, L=16384, seed=1004, sigma_k=0.5)
    raise ValueError(index)


SWEEP_MAPS = [
    ("mha", _MHA12, 12),
    ("gqa4", _MHA12, 4),
    ("mqa", _MHA12, 1),
    ("mlkv6", _PAIRS, 1),
    ("mlkv4", _TRIPLES, 1),
    ("mlkv2", _SIXES, 1),
    ("mlkv1", _ONE, 1),
]


def sweep(long_context=False):
    """The mapping sweep on the Pythia-160M shape: b=256, L=8192, or b=1, L=131072."""
    b, L = (1, 131072) if long_context else (256, 8192)
    tag = "b1-L131072" if long_context else "b256-L8192"
    return [Workload(f"pythia160m-{name}-{tag}", owner=list(own), g=g, b=b, L=L, seed=1005,
                     **PYTHIA) for name, own, g in SWEEP_MAPS]


def profiling_cases():
    """Smaller stand-ins for ncu captures that replay a kernel ~40 times: the Llama-2-7B shape at
    context 2048 (a 2 GiB cache instead of 16 GiB)."""
    return [Workload("llama2-7b-mlkv8-gqa4-b32-L2048", l=32, h=32, d=128, owner=_LLAMA_FOURS, g=8,
                     b=32, L=2048, seed=1004, sigma_k=0.5)]


def by_name(name):
    for i in range(1, 5):
        w = config(i)
        if w.name == name:
            return w
    for w in profiling_cases():
        if w.name == name:
            return w
    for w in sweep(False) + sweep(True):
        if w.name == name:
            return w
    raise KeyError(name)


def all_names():
    return [config(i).name for i in range(1, 5)] + [w.name for w in sweep(False) + sweep(True)]
