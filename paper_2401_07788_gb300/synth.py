"""Seeded synthetic inputs shaped like the paper's stage-boundary tensors.

This module only draws inputs; it holds none of the compression arithmetic.  Tests feed
the same tensors to the CUDA library and (copied to the host) to the CPU oracle; the
benchmark uses them as its workload.  The paper's data (CIFAR-10 activations of
ResNet-18, GPT-2 hidden states on Wikitext, §3.1 and §3.2) is not available here, so each
recipe reproduces the shapes and value distributions of those boundaries:

* cnn_small : ResNet-18 boundary at batch 32, [32, 64, 16, 16]; activations ReLU(N(0,1))
              (about half exact zeros), gradients N(0, sigma=1e-3); row = one sample.
* cnn       : batch 128, [128, 128, 16, 16]; same distributions; activations drift by
              0.1 * N(0,1) per step.
* lm        : GPT-2-small boundary, batch 8 x 1024 tokens x 768 hidden; hidden states
              N(0,1) with 0.5% of channels (4 of 768, chosen by the seed) scaled x20;
              gradients N(0, sigma=1e-4); drift 0.05 * N(0,1); row = one token.
* aqsgd     : per-sample buffer [4096, 512, 1024] from N(0,1); 16 ids per step drawn
              without replacement; x = buf[ids] + 0.05 * N(0,1).
* sweep     : single N(0,1) tensors of 2^20 .. 2^30 entries.

Standard deviations: "N(0, 1e-3)" in the workload description is read as sigma = 1e-3.
"""

from __future__ import annotations

import torch


def k_of(row_len: int, percent: int) -> int:
    """Entries kept per row for Top K% (whole percent): max(1, floor(row_len * K / 100))."""
    return max(1, (int(row_len) * int(percent)) // 100)


def generator(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def normal(shape, seed: int, device, std: float = 1.0, gen: torch.Generator | None = None):
    g = gen or generator(seed, device)
    x = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x


def relu_normal(shape, seed: int, device, gen: torch.Generator | None = None):
    return normal(shape, seed, device, gen=gen).clamp_min_(0.0)


def drift(x: torch.Tensor, sigma: float, gen: torch.Generator) -> torch.Tensor:
    """Next step's tensor: x + sigma * N(0,1)."""
    return x + sigma * torch.randn(x.shape, generator=gen, device=x.device, dtype=torch.float32)


def lm_hidden(seed: int, device, batch: int = 8, seq: int = 1024, hidden: int = 768,
              outlier_frac: float = 0.005, outlier_scale: float = 20.0):
    """Hidden states [batch*seq, hidden] with a fixed set of outlier channels."""
    g = generator(seed, device)
    x = torch.randn((batch * seq, hidden), generator=g, device=device, dtype=torch.float32)
    n_out = max(1, int(round(hidden * outlier_frac)))
    gc = generator(seed + 7919, "cpu")
    ch = torch.randperm(hidden, generator=gc)[:n_out].to(device)
    x[:, ch] *= outlier_scale
    return x


def sample_ids(num_samples: int, n: int, seed: int, device) -> torch.Tensor:
    """n distinct ids in [0, num_samples), drawn without replacement."""
    g = generator(seed, "cpu")
    return torch.randperm(num_samples, generator=g)[:n].to(torch.int64).to(device)


# Workloads (sizes as in the descriptions above)
CNN_SMALL = dict(shape=(32, 64, 16, 16), rows=32, row_len=16384, topk_percent=10, bits=8)
CNN = dict(shape=(128, 128, 16, 16), rows=128, row_len=32768, topk_percents=(5, 10, 30),
           bits=(2, 4, 8), steps=50, drift=0.1, seeds=tuple(range(10)))
LM = dict(rows=8192, row_len=768, topk_percent=10, bits=4, steps=20, drift=0.05)
AQSGD = dict(num_samples=4096, rows_per_sample=512, row_len=1024, ids_per_step=16,
             topk_percent=30, steps=100, noise=0.05)
SWEEP = dict(log2_sizes=tuple(range(20, 31)), row_lens=(768, 4096, 65536, None),
             topk_percents=(1, 10, 50), bits=(2, 4, 8))
