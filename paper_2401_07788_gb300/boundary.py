"""Compression block between pipeline stages (§2.1, Figure 1): the forward pass sends a
compressed activation across the cut and the backward pass a compressed gradient, so that
a model cut into stages trains as it would if the stages ran on separate devices that
exchange compressed messages.

``CompressionBoundary`` is a ``torch.nn.Module`` wrapping one such block.  Its forward
output is the decompressed activation (what the next stage receives); its backward
returns the decompressed gradient (what the previous stage receives).  Every compression
step runs in the library's kernels through the ``mpc_*`` calls; this module only reshapes
tensors into rows, keeps the feedback state between steps, routes the calls and reads the
reconstruction out of the feedback buffer.

Compressors (the operators of §2.2 - §2.5):

* ``Quant(bits, stochastic, feedback)``  min-max quantisation to 2^bits levels (§2.2),
  bits 1..16 (the paper uses 2, 4, 6, 8), round to nearest or stochastic; ``feedback``
  ``"aqsgd"`` quantises the change against a buffer kept per training sample, as the work
  §2.5 cites does.
* ``TopK(percent, feedback)``  TopK of §2.3, optionally with error feedback (§2.4):
  ``"none"``, ``"ef"`` (Seide: one global error buffer), ``"ef21"`` (the previously sent
  value), ``"aqsgd"`` (§2.5: one buffer per training sample; ``forward`` then takes the
  batch's sample ids).
* ``Reuse()`` (gradients only): the gradient is sent at the indices the activation's TopK
  kept (§3.2, Table 5, which fine-tuning needs to converge).
* ``None``: no compression in that direction.

What the next stage receives: the decompressed message for plain compression and for EF
(the receiver has no buffer of its own); the receiver's reconstruction for EF21 (its copy
of ``g``) and AQ-SGD (its copy of the sample's buffer rows), which equals the sender's
buffer after the update since both take the same fp32 additions.

Rows: ``rows="sample"`` treats each sample (all dims but the first) as one row, as for the
CNN boundaries; ``rows="last"`` treats the last dimension as the row (one token of a
transformer boundary).

Inference: in ``eval()`` mode the block is the identity unless ``compress_at_inference``
is set; the paper finds that models trained with compression score better when the
compression stays on at inference (§3.1).  At inference the forward compressor is applied
without feedback: EF, EF21 and AQ-SGD buffers are left as training left them.
"""

from __future__ import annotations

from dataclasses import dataclass

import torch

from . import (mpc_aqsgd_compress, mpc_aqsgd_quant_compress, mpc_ef21_topk_compress,
               mpc_ef_topk_compress, mpc_quant_compress, mpc_quant_decompress,
               mpc_topk_compress, mpc_topk_decompress, mpc_topk_gather)
from .synth import k_of

__all__ = ["Quant", "TopK", "Reuse", "CompressionBoundary", "with_boundaries"]


@dataclass(frozen=True)
class Quant:
    bits: int
    stochastic: bool = False
    feedback: str = "none"  # "none" | "aqsgd"

    def __post_init__(self):
        if self.feedback not in ("none", "aqsgd"):
            raise ValueError("quantisation feedback must be none or aqsgd")


@dataclass(frozen=True)
class TopK:
    percent: int
    feedback: str = "none"  # "none" | "ef" | "ef21" | "aqsgd"

    def __post_init__(self):
        if self.feedback not in ("none", "ef", "ef21", "aqsgd"):
            raise ValueError("feedback must be none, ef, ef21 or aqsgd")


@dataclass(frozen=True)
class Reuse:
    """Gradient compressed at the activation's TopK indices (backward only)."""


def _as_rows(t: torch.Tensor, rows: str) -> torch.Tensor:
    t = t.contiguous()
    if rows == "sample":
        return t.reshape(t.shape[0], -1) if t.dim() > 1 else t.reshape(1, -1)
    return t.reshape(-1, t.shape[-1])


class _BoundaryFn(torch.autograd.Function):
    @staticmethod
    def forward(ctx, x, block, sample_ids):
        y, idx = block._compress_forward(x, sample_ids)
        ctx.block = block
        ctx.idx = idx
        return y

    @staticmethod
    def backward(ctx, gy):
        return ctx.block._compress_backward(gy, ctx.idx), None, None


class CompressionBoundary(torch.nn.Module):
    """One compression block between two pipeline stages (§2.1, Figure 1)."""

    def __init__(self, forward=None, backward=None, rows: str = "sample",
                 compress_at_inference: bool = False, seed: int = 0,
                 aqsgd_samples: int = 0):
        super().__init__()
        if rows not in ("sample", "last"):
            raise ValueError("rows must be 'sample' or 'last'")
        if isinstance(forward, Reuse):
            raise ValueError("Reuse() compresses gradients only")
        if isinstance(backward, Reuse) and not isinstance(forward, TopK):
            raise ValueError("Reuse() needs a TopK forward compressor")
        if isinstance(backward, (TopK, Quant)) and backward.feedback != "none":
            raise ValueError("feedback applies to the forward (activation) compressor")
        if getattr(forward, "feedback", None) == "aqsgd" and aqsgd_samples < 1:
            raise ValueError("AQ-SGD needs aqsgd_samples, the number of training samples")
        self.fw = forward
        self.bw = backward
        self.rows = rows
        self.compress_at_inference = compress_at_inference
        self.seed = int(seed)
        self.aqsgd_samples = int(aqsgd_samples)
        self.step = 0
        self.state = None  # EF error, EF21 last sent value, or the AQ-SGD per-sample buffer
        self.sample_ids = None  # AQ-SGD: the batch's ids when forward is not given them

    def reset_state(self) -> None:
        self.state = None
        self.step = 0

    def forward(self, x: torch.Tensor, sample_ids: torch.Tensor | None = None) -> torch.Tensor:
        if not self.training and not self.compress_at_inference:
            return x
        return _BoundaryFn.apply(x, self, self.sample_ids if sample_ids is None else sample_ids)

    # -- the two directions ---------------------------------------------------------------

    def _seed(self, direction: int) -> int:
        return (((self.seed << 1) | direction) << 32) | (self.step & 0xffffffff)

    def _quant(self, rows2d: torch.Tensor, c: Quant, direction: int) -> torch.Tensor:
        codes, scale, minv = mpc_quant_compress(rows2d, c.bits, stochastic=c.stochastic,
                                                seed=self._seed(direction))
        return mpc_quant_decompress(codes, scale, minv, rows2d.shape[1], c.bits)

    def _compress_forward(self, x: torch.Tensor, sample_ids):
        c = self.fw
        if c is None:
            return x.clone(), None
        r = _as_rows(x.detach(), self.rows)
        R, L = r.shape
        idx = None
        fb = c.feedback if self.training else "none"
        if fb == "aqsgd":
            y, idx = self._aqsgd(r, c, sample_ids)
        elif isinstance(c, Quant):
            y = self._quant(r, c, 0)
        else:
            k = k_of(L, c.percent)
            if fb == "none":
                vals, idx = mpc_topk_compress(r, k)
            elif fb == "ef":
                if self.state is None or self.state.shape != r.shape:
                    self.state = torch.zeros_like(r)
                vals, idx = mpc_ef_topk_compress(r, self.state, k)
            elif fb == "ef21":
                if self.state is None or self.state.shape != r.shape:
                    self.state = torch.zeros_like(r)
                vals, idx = mpc_ef21_topk_compress(r, self.state, k)
            if fb == "ef21":
                y = self.state.clone()  # the receiver's g' = g + C(x - g)
            else:
                y = mpc_topk_decompress(vals, idx, L)
        if self.training:
            self.step += 1
        return y.reshape(x.shape), idx

    def _aqsgd(self, r: torch.Tensor, c, sample_ids):
        """AQ-SGD (§2.5): the change against the samples' buffer rows is compressed and
        both copies of the buffer take it; the next stage receives the updated rows."""
        if sample_ids is None:
            raise ValueError("AQ-SGD needs the batch's sample ids")
        R, L = r.shape
        ids = sample_ids.to(device=r.device, dtype=torch.int64).contiguous()
        if R % ids.numel():
            raise ValueError("rows must split evenly over the sample ids")
        n, rps = ids.numel(), R // ids.numel()
        shape = (self.aqsgd_samples, rps, L)
        if self.state is None or tuple(self.state.shape) != shape:
            self.state = torch.zeros(shape, device=r.device)
        idx = None
        if isinstance(c, Quant):
            mpc_aqsgd_quant_compress(r.reshape(n, rps, L), self.state, ids, c.bits,
                                     stochastic=c.stochastic, seed=self._seed(0))
        else:
            _, idx = mpc_aqsgd_compress(r.reshape(n, rps, L), self.state, ids,
                                        k_of(L, c.percent))
            idx = idx.reshape(R, -1)
        return self.state[ids].reshape(R, L), idx

    def _compress_backward(self, gy: torch.Tensor, idx):
        c = self.bw
        if c is None:
            return gy
        g = _as_rows(gy, self.rows)
        L = g.shape[1]
        if isinstance(c, Quant):
            out = self._quant(g, c, 1)
        elif isinstance(c, Reuse):
            out = mpc_topk_decompress(mpc_topk_gather(g, idx), idx, L)
        else:
            vals, ix = mpc_topk_compress(g, k_of(L, c.percent))
            out = mpc_topk_decompress(vals, ix, L)
        return out.reshape(gy.shape)


def with_boundaries(stages, make_boundary) -> torch.nn.Sequential:
    """A pipeline of stages with a compression block after every stage but the last
    (model-parallel degree len(stages): len(stages) - 1 blocks, §3.2 uses degree 4).
    ``make_boundary(i)`` returns the block after stage i."""
    mods = []
    for i, s in enumerate(stages):
        mods.append(s)
        if i + 1 < len(stages):
            mods.append(make_boundary(i))
    return torch.nn.Sequential(*mods)
