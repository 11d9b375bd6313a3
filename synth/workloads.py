"""The synthetic workloads (shapes, dtypes, seeds and value recipes).

They stand in for the paper's evaluation settings (Long Range Arena encoders,
BERT-base, ViT-B/16 and a long-context causal stream) by shape only: the
datasets and checkpoints are not used.  The feature dimension D = M * L uses
the paper's default of L = 8 channels (Sec. 5.3, Table 4), so D = 64 means
M = 8 projections and D = 128 means M = 16.
"""
from __future__ import annotations

import math
from dataclasses import dataclass


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    n: int
    d: int
    M: int
    L: int
    io: str            # "f32" or "bf16"
    causal: bool
    backward: bool     # fwd+bwd (True) or fwd only (False)
    seed: int
    qkv_scale: float
    len_range: tuple | None = None
    hidden: int = 64
    chunk: int = 64
    eps: float = 1e-6
    decode: bool = False  # one streaming-form step per (batch, head) after a causal prefill of n tokens

    @property
    def dv(self) -> int:
        return self.d

    @property
    def D(self) -> int:
        return self.M * self.L

    @property
    def tokens(self) -> int:
        return self.B * self.n


WORKLOADS = {
    "tiny_f32": Workload("tiny_f32", B=1, H=1, n=256, d=64, M=8, L=8, io="f32",
                         causal=False, backward=False, seed=0, qkv_scale=1.0),
    "lra": Workload("lra", B=32, H=4, n=4096, d=32, M=8, L=8, io="bf16",
                    causal=False, backward=True, seed=1, qkv_scale=1.0 / math.sqrt(32),
                    len_range=(2048, 4096)),
    "bert": Workload("bert", B=32, H=12, n=512, d=64, M=8, L=8, io="bf16",
                     causal=False, backward=True, seed=2, qkv_scale=1.0),
    "vit": Workload("vit", B=64, H=12, n=197, d=64, M=8, L=8, io="bf16",
                    causal=False, backward=False, seed=3, qkv_scale=1.0),
    "causal_long": Workload("causal_long", B=2, H=32, n=65536, d=128, M=16, L=8, io="bf16",
                            causal=True, backward=True, seed=4, qkv_scale=1.0 / math.sqrt(128)),
    # streaming inference: 64 sequences x 32 heads advance by one token per step from the state of a
    # 1024-token causal prefill (the long-context head shape)
    "decode": Workload("decode", B=64, H=32, n=1024, d=128, M=16, L=8, io="bf16",
                       causal=True, backward=False, seed=5, qkv_scale=1.0 / math.sqrt(128), decode=True),
}
