"""Seeded synthetic inputs for the gradient-sparsification workloads.

This module is the one piece shared by the CUDA path's tests/bench and by the
oracle's tests: it only draws random gradients of the right shapes and
distributions.  It holds none of the method's arithmetic (no probabilities,
no sampling decisions, no coding, no sums of sparse vectors).

Five workloads, after the paper's settings (section 5) and the sizes the
GPU library is measured on:

  c1  one fp32 vector, d = 65536: g_i = s_i m_i, s_i a fair sign, m_i ~
      LogNormal(0, 1.5); kappa = 0.1, 2 iterations, Philox seed 1, step 0.
  c2  M = 8 workers of an l2-regularised logistic regression (section 5.1,
      Eq. 14): each owns X (256 x 2^20, N(0,1) scaled per feature by
      (j+1)^-0.8), labels b = sign(X w*), shared w ~ N(0, 0.01); g is the
      minibatch gradient (natural log, lambda_2 = 1/(10 N), N = 8*256);
      kappa = 0.05, 2 iterations.
  c3  M = 16 workers, d = 2^24: g_i ~ Student-t(3), 1% of coordinates zeroed
      by an independent Bernoulli(0.01); kappa = 0.01, 3 iterations.
  c4  M = 8 workers, layer-wise: 161 tensors shaped like ResNet-50's
      parameters (25,557,032 values), each N(0, 1/fan_in); kappa = 0.02 per
      layer, 2 iterations.
  c5  M = 8 workers, d = 2^27: |g_i| ~ LogNormal(0, 2) with a fair sign, and
      0.1% outliers scaled by 100; fp32 and bf16 (round-to-nearest-even from
      the same fp32 values); kappa in {0.001, 0.01, 0.1}, 3 iterations.

Beside them, the training data of the section 5.1 experiment (gen_sec51)
and the minibatch indices of its SGD runs (minibatches).

Host (numpy) generators serve the CPU tests and reduced sizes; device
(torch) generators make the full-size inputs quickly on the GPU.  The two use
different random streams: a parity check always hands the same bytes to both
the CUDA path and the oracle.
"""
from dataclasses import dataclass, field
import math

import numpy as np


@dataclass(frozen=True)
class Workload:
    name: str
    M: int
    d: int
    kappa: float
    iters: int
    dtype: str = "f32"          # "f32" or "bf16" storage of g
    seed: int = 1               # Philox key
    step: int = 0
    data_seed: int = 0
    segmented: bool = False
    kappas: tuple = field(default_factory=tuple)


C1 = Workload("c1_d65536_M1_lognormal", M=1, d=65536, kappa=0.1, iters=2, data_seed=0)
C2 = Workload("c2_logreg_d1048576_M8", M=8, d=1 << 20, kappa=0.05, iters=2, data_seed=2)
C3 = Workload("c3_d16777216_M16_student_t3", M=16, d=1 << 24, kappa=0.01, iters=3, data_seed=3)
C4 = Workload("c4_resnet50_layerwise_M8", M=8, d=25557032, kappa=0.02, iters=2, data_seed=4, segmented=True)
C5 = Workload("c5_d134217728_M8_lognormal_outliers", M=8, d=1 << 27, kappa=0.01, iters=3, data_seed=5,
              kappas=(0.001, 0.01, 0.1))

WORKLOADS = {w.name: w for w in (C1, C2, C3, C4, C5)}


# ---------------------------------------------------------------------------
# ResNet-50 parameter tensor shapes (c4)
# ---------------------------------------------------------------------------
def resnet50_layers():
    """(name, numel, fan_in) of the 161 parameter tensors of a ResNet-50-like
    network: 7x7 stem, bottleneck stages (3, 4, 6, 3) with widths
    (64, 128, 256, 512) and x4 expansion, a 1x1 projection in each stage's
    first block, BN scale and shift after every conv, and a 2048 x 1000 FC
    layer with bias.  Conv fan_in = c_in*k*k; FC weight fan_in = 2048; BN
    vectors and the FC bias use their own length."""
    out = []

    def conv(name, cout, cin, k):
        out.append((name + ".weight", cout * cin * k * k, cin * k * k))

    def bn(name, c):
        out.append((name + ".weight", c, c))
        out.append((name + ".bias", c, c))

    conv("conv1", 64, 3, 7)
    bn("bn1", 64)
    inpl = 64
    for si, (blocks, width) in enumerate([(3, 64), (4, 128), (6, 256), (3, 512)]):
        for b in range(blocks):
            pre = f"layer{si + 1}.{b}"
            cout = width * 4
            conv(pre + ".conv1", width, inpl, 1)
            bn(pre + ".bn1", width)
            conv(pre + ".conv2", width, width, 3)
            bn(pre + ".bn2", width)
            conv(pre + ".conv3", cout, width, 1)
            bn(pre + ".bn3", cout)
            if b == 0:
                conv(pre + ".downsample", cout, inpl, 1)
                bn(pre + ".downsample_bn", cout)
            inpl = cout
    out.append(("fc.weight", 1000 * 2048, 2048))
    out.append(("fc.bias", 1000, 1000))
    return out


def resnet50_offsets():
    layers = resnet50_layers()
    off = np.zeros(len(layers) + 1, dtype=np.int64)
    off[1:] = np.cumsum([n for _, n, _ in layers])
    return off


# ---------------------------------------------------------------------------
# bf16 storage
# ---------------------------------------------------------------------------
def f32_to_bf16_bits(x):
    """Round-to-nearest-even fp32 -> bf16 bit patterns (uint16); NaN stays NaN."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounding = ((b >> 16) & 1) + 0x7FFF
    r = ((b + rounding) >> 16).astype(np.uint16)
    nan = np.isnan(np.asarray(x, dtype=np.float32))
    r[nan] = 0x7FC0
    return r


def bf16_bits_to_f32(bits):
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# ---------------------------------------------------------------------------
# Host generators (numpy)
# ---------------------------------------------------------------------------
def lognormal_signed(d, sigma, seed):
    rng = np.random.default_rng(seed)
    m = rng.lognormal(0.0, sigma, size=d)
    s = np.where(rng.random(d) < 0.5, -1.0, 1.0)
    return (s * m).astype(np.float32)


def gen_c1(d=65536, seed=0):
    return lognormal_signed(d, 1.5, seed)


def gen_student_t(M, d, seed0=3, zero_frac=0.01):
    g = np.empty((M, d), dtype=np.float32)
    for m in range(M):
        rng = np.random.default_rng(seed0 + m)
        row = rng.standard_t(3.0, size=d)
        row[rng.random(d) < zero_frac] = 0.0
        g[m] = row
    return g


def gen_c5(M, d, seed0=5, outlier_frac=0.001, outlier_scale=100.0):
    g = np.empty((M, d), dtype=np.float32)
    for m in range(M):
        rng = np.random.default_rng(seed0 * 1000 + m)
        mag = rng.lognormal(0.0, 2.0, size=d)
        mag[rng.random(d) < outlier_frac] *= outlier_scale
        sgn = np.where(rng.random(d) < 0.5, -1.0, 1.0)
        g[m] = (sgn * mag).astype(np.float32)
    return g


def gen_layerwise(M, layers=None, seed0=4):
    """c4 values: per layer N(0, 1/fan_in); `layers` defaults to ResNet-50."""
    layers = resnet50_layers() if layers is None else layers
    d = sum(n for _, n, _ in layers)
    g = np.empty((M, d), dtype=np.float32)
    off = np.zeros(len(layers) + 1, dtype=np.int64)
    off[1:] = np.cumsum([n for _, n, _ in layers])
    for m in range(M):
        rng = np.random.default_rng(seed0 * 1000 + m)
        for l, (_, n, fan_in) in enumerate(layers):
            g[m, off[l]:off[l + 1]] = rng.standard_normal(n) / math.sqrt(fan_in)
    return g, off


def gen_logreg(M, d, B=256, seed0=2, lam2=None):
    """c2 on the host at reduced size: the minibatch gradient of Eq. 14
    (natural log) for each of M workers."""
    rng = np.random.default_rng(seed0)
    N = M * B
    lam2 = 1.0 / (10.0 * N) if lam2 is None else lam2
    scale = (np.arange(d, dtype=np.float64) + 1.0) ** -0.8
    w_star = rng.standard_normal(d)
    w = rng.normal(0.0, 0.1, size=d)
    g = np.empty((M, d), dtype=np.float32)
    for m in range(M):
        X = rng.standard_normal((B, d)) * scale
        b = np.sign(X @ w_star)
        b[b == 0] = 1.0
        r = -b / (1.0 + np.exp(b * (X @ w))) / B
        g[m] = (X.T @ r + 2.0 * lam2 * w).astype(np.float32)
    return g


def gen_sec51(N=1024, d=2048, C1=0.6, C2=1.0 / 16.0, seed=0):
    """The synthetic data set of section 5.1: dense rows xbar_n ~ N(0, I), a
    magnitude vector Bbar ~ U[0,1]^d whose entries at or below C2 are scaled by
    C1, rows x_n = xbar_n * Bbar (element-wise), and labels
    y_n = sign(xbar_n^T wbar) with wbar ~ N(0, I) (a zero sign counts as +1).
    Returns fp32 X (N x d) and y (N)."""
    rng = np.random.default_rng(seed)
    xbar = rng.standard_normal((N, d))
    Bbar = rng.uniform(0.0, 1.0, d)
    Bbar = np.where(Bbar <= C2, C1 * Bbar, Bbar)
    wbar = rng.standard_normal(d)
    y = np.sign(xbar @ wbar)
    y[y == 0] = 1.0
    return (xbar * Bbar).astype(np.float32), y.astype(np.float32)


def minibatches(T, M, B, N, seed=0):
    """Row indices of T steps of M workers' minibatches of B, uniform with
    replacement (int32, T x M x B)."""
    rng = np.random.default_rng(seed + 7919)
    return rng.integers(0, N, size=(T, M, B)).astype(np.int32)


# ---------------------------------------------------------------------------
# Device generators (torch), for the full sizes
# ---------------------------------------------------------------------------
def _torch():
    import torch
    return torch


def device_student_t(M, d, seed0=3, zero_frac=0.01, device="cuda", out=None):
    """Student-t(3) rows built as Z / sqrt(chi2_3 / 3) with chi2_3 the sum of
    three squared normals; 1% of coordinates zeroed."""
    torch = _torch()
    out = torch.empty((M, d), dtype=torch.float32, device=device) if out is None else out
    for m in range(M):
        gen = torch.Generator(device=device)
        gen.manual_seed(seed0 + m)
        z = torch.randn(d, generator=gen, device=device)
        chi = torch.zeros(d, device=device)
        for _ in range(3):
            chi.add_(torch.randn(d, generator=gen, device=device).square_())
        row = z.div_(chi.div_(3.0).sqrt_())
        row.masked_fill_(torch.rand(d, generator=gen, device=device) < zero_frac, 0.0)
        out[m].copy_(row)
        del z, chi, row
    return out


def device_lognormal(M, d, sigma=2.0, seed0=5, outlier_frac=0.001, outlier_scale=100.0, device="cuda", out=None):
    torch = _torch()
    out = torch.empty((M, d), dtype=torch.float32, device=device) if out is None else out
    for m in range(M):
        gen = torch.Generator(device=device)
        gen.manual_seed(seed0 * 1000 + m)
        row = torch.randn(d, generator=gen, device=device).mul_(sigma).exp_()
        if outlier_frac > 0:
            hit = torch.rand(d, generator=gen, device=device) < outlier_frac
            row = torch.where(hit, row * outlier_scale, row)
        neg = torch.rand(d, generator=gen, device=device) < 0.5
        out[m].copy_(torch.where(neg, -row, row))
        del row, neg
    return out


def device_layerwise(M, seed0=4, device="cuda"):
    torch = _torch()
    layers = resnet50_layers()
    off = resnet50_offsets()
    d = int(off[-1])
    g = torch.empty((M, d), dtype=torch.float32, device=device)
    for m in range(M):
        gen = torch.Generator(device=device)
        gen.manual_seed(seed0 * 1000 + m)
        for l, (_, n, fan_in) in enumerate(layers):
            g[m, int(off[l]):int(off[l + 1])] = torch.randn(n, generator=gen, device=device) / math.sqrt(fan_in)
    return g, off


def device_logreg(M, d, B=256, seed0=2, device="cuda"):
    """c2 at full size on the GPU: per worker X (B x d fp32, 1 GiB at d=2^20)
    is drawn, used for one gradient of Eq. 14 (natural log), and dropped."""
    torch = _torch()
    gen = torch.Generator(device=device)
    gen.manual_seed(seed0)
    N = M * B
    lam2 = 1.0 / (10.0 * N)
    scale = (torch.arange(d, device=device, dtype=torch.float32) + 1.0).pow_(-0.8)
    w_star = torch.randn(d, generator=gen, device=device)
    w = torch.randn(d, generator=gen, device=device) * 0.1
    g = torch.empty((M, d), dtype=torch.float32, device=device)
    for m in range(M):
        X = torch.randn((B, d), generator=gen, device=device).mul_(scale)
        b = torch.sign(X @ w_star)
        b[b == 0] = 1.0
        r = -b / (1.0 + torch.exp(b * (X @ w))) / B
        g[m] = X.t() @ r + 2.0 * lam2 * w
        del X
    return g


def device_c1(d=65536, seed=0, device="cuda"):
    torch = _torch()
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    m = torch.randn(d, generator=gen, device=device).mul_(1.5).exp_()
    neg = torch.rand(d, generator=gen, device=device) < 0.5
    return torch.where(neg, -m, m).reshape(1, d)


def device_to_bf16(g):
    """Round-to-nearest-even copy of an fp32 device tensor as bf16."""
    torch = _torch()
    return g.to(torch.bfloat16)
