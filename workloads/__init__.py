"""Seeded synthetic inputs for the packed ternary linear layer.

This module only draws random inputs (trit codes, fp16 scales/offsets, the
salience map and fp16 activations) and lays them out in the library's input
formats.  It contains none of the method's arithmetic; both the CPU oracle
(tests) and the CUDA path consume what it returns.

Distributions (the paper's workload is real Qwen3 weights, which are not
available; these stand in for them with the shapes of the paper's Qwen3-4B /
Qwen3-8B projections, "Model and Representation"):
  * T1, T2 i.i.d. in {-1, 0, +1} with p = 0.3 / 0.4 / 0.3;
  * s1, s2 ~ lognormal(mu=-4, sigma=0.5), rounded to fp16 (nearest even);
  * off ~ Normal(0, std=1e-3), rounded to fp16 (some values are subnormal);
  * salience: exactly round(f2 * N * G) groups, chosen by a seeded
    permutation of the N*G group ids (f2 = 0.1; 0 for the single-layer
    smoke shape); T2 is zero outside salient groups;
  * x ~ Normal(0, 1), rounded to fp16.
Seeds: numpy SeedSequence([seed, config, layer, proj, tensor_id]).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

GROUP = 128

# Qwen3-4B: hidden 2560, intermediate 9728, 32 q heads / 8 kv heads of 128.
QWEN3_4B = [
    ("q", 4096, 2560), ("k", 1024, 2560), ("v", 1024, 2560), ("o", 2560, 4096),
    ("gate", 9728, 2560), ("up", 9728, 2560), ("down", 2560, 9728),
]
# Qwen3-8B: 36 layers, hidden 4096, intermediate 12288, 32 q heads / 8 kv heads.
QWEN3_8B = [
    ("q", 4096, 4096), ("k", 1024, 4096), ("v", 1024, 4096), ("o", 4096, 4096),
    ("gate", 12288, 4096), ("up", 12288, 4096), ("down", 4096, 12288),
]
QWEN3_8B_LAYERS = 36

TENSOR_T1, TENSOR_S1, TENSOR_OFF, TENSOR_SAL, TENSOR_T2, TENSOR_S2, TENSOR_X, TENSOR_DENSE = range(8)


@dataclass(frozen=True)
class Projection:
    name: str
    N: int
    K: int
    layer: int
    proj: int


def config_projections(config: int):
    """The projection list of a workload configuration (0..4)."""
    if config == 0:
        return [Projection("single", 512, 1024, 0, 0)]
    if config == 1:
        return [Projection(n, N, K, 0, i) for i, (n, N, K) in enumerate(QWEN3_4B)]
    if config in (2, 3):
        return [Projection(n, N, K, l, i) for l in range(QWEN3_8B_LAYERS)
                for i, (n, N, K) in enumerate(QWEN3_8B)]
    if config == 4:
        return [Projection(n, N, K, 0, i) for i, (n, N, K) in enumerate(QWEN3_8B)]
    raise ValueError(config)


def config_salient_fraction(config: int) -> float:
    return 0.0 if config == 0 else 0.1


def config_M(config: int):
    return {0: [1], 1: [1], 2: [1], 3: [2, 4, 8, 16], 4: [2048]}[config]


def _rng(seed, config, layer, proj, tensor):
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, config, layer, proj, tensor])))


def _trits(rng, shape):
    u = rng.random(shape)
    return ((u >= 0.3).astype(np.int8) + (u >= 0.7).astype(np.int8) - 1).astype(np.int8)


def _fp16_bits(values: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(values.astype(np.float16)).view(np.uint16)


def bits_from_dense(sal_dense: np.ndarray) -> np.ndarray:
    """[N][G] bool -> [N][ceil(G/32)] uint32, bit g%32 of word g/32."""
    N, G = sal_dense.shape
    W = (G + 31) // 32
    padded = np.zeros((N, W * 32), np.uint64)
    padded[:, :G] = sal_dense.astype(np.uint64)
    weights = (np.uint64(1) << np.arange(32, dtype=np.uint64))
    return (padded.reshape(N, W, 32) * weights).sum(axis=2).astype(np.uint32)


@dataclass
class Weights:
    """Inputs of one projection in the library's formats (host numpy)."""
    N: int
    K: int
    T1: np.ndarray        # int8 [N][K]
    T2: np.ndarray        # int8 [N][K], 0 outside salient groups
    sal_dense: np.ndarray  # bool [N][G]
    sal: np.ndarray       # uint32 [N][ceil(G/32)]
    s1: np.ndarray        # uint16 fp16 bits [N][G]
    off: np.ndarray       # uint16 fp16 bits [N][G]
    s2: np.ndarray        # uint16 fp16 bits [nnz], salient groups in (n, g) order

    @property
    def G(self):
        return self.K // GROUP

    @property
    def nnz(self):
        return int(self.sal_dense.sum())


def gen_weights(N: int, K: int, salient_fraction: float, config: int = 0, layer: int = 0,
                proj: int = 0, seed: int = 0) -> Weights:
    assert K % GROUP == 0 and N >= 1
    G = K // GROUP
    T1 = _trits(_rng(seed, config, layer, proj, TENSOR_T1), (N, K))
    s1 = _fp16_bits(_rng(seed, config, layer, proj, TENSOR_S1).lognormal(-4.0, 0.5, (N, G)))
    off = _fp16_bits(_rng(seed, config, layer, proj, TENSOR_OFF).normal(0.0, 1e-3, (N, G)))
    nnz = int(round(salient_fraction * N * G))
    sal_dense = np.zeros(N * G, bool)
    if nnz:
        sal_dense[_rng(seed, config, layer, proj, TENSOR_SAL).permutation(N * G)[:nnz]] = True
    sal_dense = sal_dense.reshape(N, G)
    T2 = _trits(_rng(seed, config, layer, proj, TENSOR_T2), (N, K))
    T2 *= np.repeat(sal_dense, GROUP, axis=1).astype(np.int8)
    s2 = _fp16_bits(_rng(seed, config, layer, proj, TENSOR_S2).lognormal(-4.0, 0.5, nnz))
    return Weights(N, K, T1, T2, sal_dense, bits_from_dense(sal_dense), s1, off, s2)


def gen_x(M: int, K: int, config: int = 0, layer: int = 0, proj: int = 0, seed: int = 0) -> np.ndarray:
    """fp16 bits [M][K]."""
    return _fp16_bits(_rng(seed, config, layer, proj, TENSOR_X).normal(0.0, 1.0, (M, K)))


def gen_dense_weights(N: int, K: int, config: int = 0, layer: int = 0, proj: int = 0, seed: int = 0) -> np.ndarray:
    """fp16 bits [N][K] of a dense projection, the ternarizer's input.

    Stand-in for a rotated Qwen3 projection (the paper ternarizes real
    weights after an orthogonal rotation, which are not available): row n is
    Normal(m_n, sd_n) with sd_n ~ lognormal(log 0.02, 0.25) and a small row
    mean m_n ~ Normal(0, 1e-3); one weight in a thousand is an outlier, its
    value multiplied by 8."""
    rng = _rng(seed, config, layer, proj, TENSOR_DENSE)
    sd = np.exp(rng.normal(np.log(0.02), 0.25, (N, 1)))
    m = rng.normal(0.0, 1e-3, (N, 1))
    w = m + sd * rng.standard_normal((N, K))
    w[rng.random((N, K)) < 1e-3] *= 8.0
    return _fp16_bits(w)


def gen_dense_weights_torch(N: int, K: int, device, seed: int):
    """Device-side draw of the gen_dense_weights distribution (torch's
    generator, so values differ from gen_dense_weights): fp16 [N][K]."""
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(seed)
    sd = torch.exp(torch.randn((N, 1), generator=g, device=device) * 0.25 + float(np.log(0.02)))
    m = torch.randn((N, 1), generator=g, device=device) * 1e-3
    w = torch.randn((N, K), generator=g, device=device) * sd + m
    w = torch.where(torch.rand((N, K), generator=g, device=device) < 1e-3, w * 8.0, w)
    return w.half()


def half_bits_to_float(bits: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(bits, dtype=np.uint16).view(np.float16).astype(np.float64)


# ------------------------------------------------------------------ torch side
def gen_weights_torch(N: int, K: int, salient_fraction: float, device, seed: int):
    """Device-side draw of the same distributions (for full-size workloads
    whose int8 codes are too large to draw on the host).  Uses torch's
    generator, so values differ from gen_weights for the same seed.
    Returns a dict of torch tensors: T1, T2 (int8 [N][K]), sal_dense (bool
    [N][G]), sal (int32 view of uint32 words), s1, off (fp16 [N][G]), s2
    (fp16 [nnz])."""
    import torch

    G = K // GROUP
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    u = torch.rand((N, K), generator=g, device=device)
    T1 = ((u >= 0.3).to(torch.int8) + (u >= 0.7).to(torch.int8) - 1)
    s1 = torch.empty((N, G), device=device, dtype=torch.float32).log_normal_(-4.0, 0.5, generator=g).half()
    off = (torch.randn((N, G), generator=g, device=device) * 1e-3).half()
    nnz = int(round(salient_fraction * N * G))
    sal_dense = torch.zeros(N * G, dtype=torch.bool, device=device)
    if nnz:
        sal_dense[torch.randperm(N * G, generator=g, device=device)[:nnz]] = True
    sal_dense = sal_dense.view(N, G)
    u2 = torch.rand((N, K), generator=g, device=device)
    T2 = ((u2 >= 0.3).to(torch.int8) + (u2 >= 0.7).to(torch.int8) - 1)
    T2 *= sal_dense.repeat_interleave(GROUP, dim=1).to(torch.int8)
    s2 = torch.empty(nnz, device=device, dtype=torch.float32).log_normal_(-4.0, 0.5, generator=g).half()
    W = (G + 31) // 32
    padded = torch.zeros((N, W * 32), dtype=torch.int64, device=device)
    padded[:, :G] = sal_dense.to(torch.int64)
    words = (padded.view(N, W, 32) << torch.arange(32, device=device, dtype=torch.int64)).sum(dim=2)
    sal = words.to(torch.int64).bitwise_and(0xFFFFFFFF)
    sal = torch.where(sal >= 2 ** 31, sal - 2 ** 32, sal).to(torch.int32)
    return dict(T1=T1, T2=T2, sal_dense=sal_dense, sal=sal, s1=s1, off=off, s2=s2, nnz=nnz)


def gen_x_torch(M: int, K: int, device, seed: int):
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return torch.randn((M, K), generator=g, device=device).half()


# ------------------------------------------------------ element-wise masks
# The paper's recorded projection: four disjoint salience masks with orders
# [2, 2, 1, 1] covering 0.5 %, 3.1 %, 10.0 % and 86.5 % of the weights (the
# printed coverages add to 100.1 %; the largest is taken as the rest).
EW_ORDERS = (2, 2, 1, 1)
EW_COVERAGE = (0.005, 0.031, 0.100)
TENSOR_MASK, TENSOR_MU, TENSOR_A0, TENSOR_A1 = range(8, 12)


@dataclass
class EwWeights:
    """Inputs of one projection in the element-wise four-mask form (host numpy)."""
    N: int
    K: int
    T0: np.ndarray    # int8 [N][K]
    T1: np.ndarray    # int8 [N][K], 0 wherever the element's mask has order 1
    mask: np.ndarray  # uint8 [N][K], mask id 0..3 of every element
    mu: np.ndarray    # uint16 fp16 bits [N][4]
    a0: np.ndarray    # uint16 fp16 bits [N][4]
    a1: np.ndarray    # uint16 fp16 bits [N][2] (masks 0 and 1)


def gen_ew_weights(N: int, K: int, config: int = 0, layer: int = 0, proj: int = 0, seed: int = 0,
                   coverage=EW_COVERAGE) -> EwWeights:
    """Mask ids i.i.d. per element with the recorded coverages (mask 3 the
    rest); T0, T1 i.i.d. {-1, 0, +1} at 0.3 / 0.4 / 0.3, T1 zero outside the
    order-2 masks; mu ~ Normal(0, 1e-3), alpha0 and alpha1 ~ lognormal(-4,
    0.5), all rounded to fp16."""
    u = _rng(seed, config, layer, proj, TENSOR_MASK).random((N, K))
    c = np.cumsum(coverage)
    mask = (u >= c[0]).astype(np.uint8) + (u >= c[1]).astype(np.uint8) + (u >= c[2]).astype(np.uint8)
    T0 = _trits(_rng(seed, config, layer, proj, TENSOR_T1), (N, K))
    T1 = _trits(_rng(seed, config, layer, proj, TENSOR_T2), (N, K))
    T1 *= (mask <= 1).astype(np.int8)
    mu = _fp16_bits(_rng(seed, config, layer, proj, TENSOR_MU).normal(0.0, 1e-3, (N, 4)))
    a0 = _fp16_bits(_rng(seed, config, layer, proj, TENSOR_A0).lognormal(-4.0, 0.5, (N, 4)))
    a1 = _fp16_bits(_rng(seed, config, layer, proj, TENSOR_A1).lognormal(-4.0, 0.5, (N, 2)))
    return EwWeights(N, K, T0, T1, mask, mu, a0, a1)
