"""Seeded synthetic inputs shaped like the paper's LLaVA workloads.

This module draws random numbers and nothing else: no quantization, scoring or
selection arithmetic lives here. Both the CUDA path and the CPU oracle consume
the arrays it returns, so they see identical inputs.

Shapes follow the paper's settings: 576 visual tokens per image for
LLaVA-1.5 and 2880 = 5 x 576 for LLaVA-NeXT AnyRes (Sec. 4.1, Table 1), token
budgets 64 / 192 / 320 (Tables 1 and 2), and the decoder linears of 7B / 13B
LLaMA-style language models (4096 / 11008 and 5120 / 13824). No benchmark data
is used: the features are Gaussian with a few large outlier channels, the
concept embeddings are noisy copies of random visual tokens, and the CLS
saliency is a softmax per 576-token crop.
"""
from __future__ import annotations

import dataclasses

import numpy as np

N_OUTLIER_CHANNELS = 8
OUTLIER_GAIN = 20.0
CROP = 576  # tokens per vision-tower crop


@dataclasses.dataclass(frozen=True)
class Linear:
    name: str
    k_in: int
    n_out: int


def decoder_linears(d: int, ffn: int):
    """The seven linears of one LLaMA-style decoder layer (hidden d, FFN width ffn)."""
    return (Linear("q", d, d), Linear("k", d, d), Linear("v", d, d), Linear("o", d, d),
            Linear("gate", d, ffn), Linear("up", d, ffn), Linear("down", ffn, d))


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int          # images
    N: int          # visual tokens per image
    d: int          # projector / LLM hidden size
    K: int          # visual-token budget per image
    T: int          # text tokens per image
    J: int          # concept embeddings per image
    seed: int
    heavy_tail: bool
    linears: tuple  # Linear specs run on the pruned sequence
    layers: int = 1

    @property
    def M(self) -> int:
        """Rows entering the linears: B * (K + T)."""
        return self.B * (self.K + self.T)


LLAVA15_7B_ONE = Workload("llava15-7b-1img-576to64", B=1, N=576, d=4096, K=64, T=32, J=3, seed=0,
                          heavy_tail=False, linears=(Linear("q", 4096, 4096),))
LLAVA15_7B = Workload("llava15-7b-b8-576to192", B=8, N=576, d=4096, K=192, T=64, J=3, seed=1,
                      heavy_tail=False, linears=decoder_linears(4096, 11008))
LLAVANEXT_7B = Workload("llavanext-7b-b16-2880to320-32L", B=16, N=2880, d=4096, K=320, T=64, J=3,
                        seed=2, heavy_tail=False, linears=decoder_linears(4096, 11008), layers=32)
LLAVANEXT_13B = Workload("llavanext-13b-b32-2880to640", B=32, N=2880, d=5120, K=640, T=64, J=3,
                         seed=3, heavy_tail=True, linears=decoder_linears(5120, 13824))

WORKLOADS = {w.name: w for w in (LLAVA15_7B_ONE, LLAVA15_7B, LLAVANEXT_7B, LLAVANEXT_13B)}

# GEMM + quantizer sweep: M x (K_in, N_out)
SWEEP_M = (16, 64, 256, 1024, 4096, 16384, 65536)
SWEEP_KN = ((4096, 4096), (4096, 11008), (11008, 4096), (5120, 13824))
SWEEP_SEED = 4
# selector-only sweep: tokens per image x images x budget (percent of N), d = 4096
SWEEP_SEL_N = (576, 1152, 1728, 2304, 2880)
SWEEP_SEL_B = (1, 4, 16, 64)
SWEEP_SEL_PCT = (5.0, 10.0, 11.1, 25.0, 50.0)


def sweep_budget(N: int, pct: float) -> int:
    """Token budget of the selector sweep: pct percent of N, rounded, at least 1."""
    return max(1, int(round(N * pct / 100.0)))


def sweep_selector_workload(N: int, B: int, pct: float, d: int = 4096) -> Workload:
    return Workload(f"select-sweep-b{B}-n{N}-{pct:g}pct", B=B, N=N, d=d, K=sweep_budget(N, pct), T=0, J=3,
                    seed=SWEEP_SEED, heavy_tail=False, linears=())


def outlier_channels(d: int) -> np.ndarray:
    """The fixed outlier channels for hidden size d (drawn once with seed 0)."""
    return np.sort(np.random.default_rng(0).choice(d, N_OUTLIER_CHANNELS, replace=False))


def channel_gain(d: int, heavy_tail: bool) -> np.ndarray:
    """Per-channel gain: x20 on the outlier channels, or Student-t (nu = 3) tails."""
    if heavy_tail:
        t = np.random.default_rng(12345).standard_t(3, size=d)
        return np.minimum(1.0 + np.abs(t), 200.0).astype(np.float32)
    g = np.ones(d, np.float32)
    g[outlier_channels(d)] = OUTLIER_GAIN
    return g


def features(rng: np.random.Generator, shape, d: int, heavy_tail: bool) -> np.ndarray:
    """fp16 features ~ N(0, 1) times the per-channel gain, rounded to fp16 (RNE)."""
    z = rng.standard_normal(size=tuple(shape) + (d,), dtype=np.float32)
    z *= channel_gain(d, heavy_tail)
    return z.astype(np.float16)


def concepts(rng: np.random.Generator, V: np.ndarray, J: int) -> np.ndarray:
    """Stand-in concept embeddings: J noisy copies of random visual tokens per image."""
    B, N, d = V.shape
    rows = rng.integers(0, N, size=(B, J))
    base = np.take_along_axis(V.astype(np.float32), rows[:, :, None], axis=1)
    noise = rng.standard_normal(size=(B, J, d), dtype=np.float32) * np.float32(0.5)
    return (base + noise).astype(np.float16)


def cls_saliency(rng: np.random.Generator, B: int, N: int) -> np.ndarray:
    """Stand-in CLS-to-patch attention: softmax(2 z) within each 576-token crop, fp32."""
    z = rng.standard_normal(size=(B, N), dtype=np.float32) * np.float32(2.0)
    out = np.empty_like(z)
    for c0 in range(0, N, CROP):
        c1 = min(N, c0 + CROP)
        e = np.exp(z[:, c0:c1] - z[:, c0:c1].max(axis=1, keepdims=True))
        out[:, c0:c1] = e / e.sum(axis=1, keepdims=True)
    return out.astype(np.float32)


VIT_HEADS, VIT_HEAD_DIM = 16, 64  # CLIP ViT-L/14 vision tower: 1024 wide = 16 heads x 64


@dataclasses.dataclass
class VisionAttention:
    q_cls: np.ndarray  # [B, C, H, dh] fp16, the final layer's CLS query of each crop
    k_cls: np.ndarray  # [B, C, H, dh] fp16, its CLS key
    k: np.ndarray      # [B, N, H, dh] fp16, the patch keys (crop c = tokens c*CROP ..)


def vision_attention(B: int, N: int, seed: int, H: int = VIT_HEADS, dh: int = VIT_HEAD_DIM,
                     crop: int = CROP) -> VisionAttention:
    """Synthetic final-layer attention inputs of the vision tower, one CLS per
    crop of `crop` tokens (N a multiple of it): N(0, 1) keys, the CLS query
    N(0, 1) x 2 so that each head's attention row is peaked (logit spread
    about 2) like a trained ViT's."""
    assert N % crop == 0
    rng = np.random.default_rng(seed)
    C = N // crop
    q = (rng.standard_normal(size=(B, C, H, dh), dtype=np.float32) * np.float32(2.0)).astype(np.float16)
    kc = rng.standard_normal(size=(B, C, H, dh), dtype=np.float32).astype(np.float16)
    k = rng.standard_normal(size=(B, N, H, dh), dtype=np.float32).astype(np.float16)
    return VisionAttention(q, kc, k)


@dataclasses.dataclass
class SelectorInputs:
    V: np.ndarray      # [B, N, d] fp16
    Q: np.ndarray      # [B, J, d] fp16
    A: np.ndarray      # [B, N] fp32
    text: np.ndarray   # [B, T, d] fp16


def selector_inputs(w: Workload, B: int | None = None, N: int | None = None, d: int | None = None,
                    seed: int | None = None) -> SelectorInputs:
    """Selector inputs of workload w (optionally resized for small tests)."""
    B = w.B if B is None else B
    N = w.N if N is None else N
    d = w.d if d is None else d
    rng = np.random.default_rng(w.seed if seed is None else seed)
    V = features(rng, (B, N), d, w.heavy_tail)
    Q = concepts(rng, V, w.J)
    A = cls_saliency(rng, B, N)
    text = rng.standard_normal(size=(B, w.T, d), dtype=np.float32).astype(np.float16)
    return SelectorInputs(V, Q, A, text)


def weight(k_in: int, n_out: int, seed: int) -> np.ndarray:
    """fp16 weight [n_out, k_in] ~ N(0, 0.02)."""
    rng = np.random.default_rng(seed)
    w = rng.standard_normal(size=(n_out, k_in), dtype=np.float32) * np.float32(0.02)
    return w.astype(np.float16)


def weight_seed(layer: int, linear_id: int) -> int:
    return 1000 * layer + linear_id + 7


def activations(M: int, k_in: int, seed: int, heavy_tail: bool = False) -> np.ndarray:
    """fp16 activations [M, k_in] ~ N(0, 1) with the outlier channels."""
    return features(np.random.default_rng(seed), (M,), k_in, heavy_tail)
