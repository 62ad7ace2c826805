"""Seeded synthetic inputs for the slot-loss workloads.

This module only draws random tensors and arranges them; it holds none of the loss
arithmetic, so both the GPU path and the CPU oracle can be fed from it.  All draws come from
one ``torch.Generator`` per call, seeded explicitly, in a fixed order.

Workloads (the paper's head shapes; its corpora are not available, so these stand in):
  tiny   fp32  d=256,  V=4096,   B=8,  A=64     W~N(0,0.02^2), Hd~N(0,1), Ht = Hd + 0.5 N(0,1)
  small  bf16  d=2048, V=32000,  B=16, A=256    same recipe, sigma 0.5
  vl7b   bf16  d=3584, V=152064, B=16, A=512    rollout buffer F [32, 2048, d] ~ N(0,1);
                                                Ht rows gathered from F; Hd = Ht + 0.5 N(0,1)
  text8b bf16  d=4096, V=151936, B=16, A=2048   rollout buffer F [16, 4096, d] (128 anchors per
                                                sample); Hd = Ht + sigma N(0,1), sigma in
                                                {0.25, 0.5, 1.0}
  erase  bf16  as text8b with sigma 0.5; corpus token = greedy target token, replaced by a
               uniform random token with probability 0.2 per position
  sharp  any of the above through ``sharpen``: the head scaled so that the logits reach a
         trained head's magnitude (|z| up to 30-40) instead of the random head's (|z| < 7)
"""

from __future__ import annotations

from dataclasses import dataclass

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    d: int
    V: int
    B: int
    A: int
    dtype: str                 # "bf16" or "f32"
    sigma: float = 0.5
    S: int = 0                 # rollout sequences (0: no feature buffer)
    L: int = 0                 # rollout sequence length
    replace_rate: float = 0.0  # erase workload: corpus-token replacement probability

    @property
    def N(self) -> int:
        return self.A * self.B

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32


WORKLOADS = {
    "tiny": Workload("tiny", 256, 4096, 8, 64, "f32"),
    "small": Workload("small", 2048, 32000, 16, 256, "bf16"),
    "vl7b": Workload("vl7b", 3584, 152064, 16, 512, "bf16", S=32, L=2048),
    "text8b": Workload("text8b", 4096, 151936, 16, 2048, "bf16", S=16, L=4096),
    "erase": Workload("erase", 4096, 151936, 16, 2048, "bf16", S=16, L=4096, replace_rate=0.2),
}

HEAD_STD = 0.02


def _gen(device, seed):
    return torch.Generator(device=device).manual_seed(int(seed))


def slot_batch(d, V, A, B, sigma=0.5, *, dtype=torch.bfloat16, device="cpu", seed=0):
    """Head and hidden states without a feature buffer.

    Draw order: W [d, V] ~ N(0, 0.02^2), Hd [N, d] ~ N(0, 1), noise [N, d] ~ N(0, 1);
    Ht = Hd + sigma * noise.  Returned in ``dtype`` (rounded once from fp32).
    """
    g = _gen(device, seed)
    N = A * B
    W = torch.randn(d, V, generator=g, device=device) * HEAD_STD
    Hd = torch.randn(N, d, generator=g, device=device)
    noise = torch.randn(N, d, generator=g, device=device)
    Ht = Hd + sigma * noise
    return dict(W=W.to(dtype), Hd=Hd.to(dtype), Ht=Ht.to(dtype))


def anchor_positions(A, S, L, B, *, device="cpu", g=None, seed=0):
    """Anchors spread evenly over S sequences (A/S per sequence, in order), start positions
    uniform in [1, L - B] so that every slot of the block lies inside its sequence."""
    g = g if g is not None else _gen(device, seed)
    per = max(1, A // S)
    seq = (torch.arange(A, device=device) // per).clamp_(max=S - 1).to(torch.int32)
    pos = torch.randint(1, L - B + 1, (A,), generator=g, device=device, dtype=torch.int32)
    return seq, pos


def rollout_batch(d, V, A, B, S, L, sigma=0.5, *, dtype=torch.bfloat16, device="cpu", seed=0,
                  chunk_rows=1 << 16):
    """Head, rollout feature buffer, anchor placement and drafter hidden states.

    Draw order: W [d, V], F [S, L, d] ~ N(0, 1), anchor start positions, noise [N, d].
    The drafter state of slot (a, s) is F[seq_a, pos_a + s] + sigma * noise, i.e. a noisy copy
    of the target feature the block reads; Ht itself is produced by the gather under test.
    """
    g = _gen(device, seed)
    N = A * B
    W = (torch.randn(d, V, generator=g, device=device) * HEAD_STD).to(dtype)
    F = torch.empty(S, L, d, dtype=dtype, device=device)
    flat = F.view(S * L, d)
    for r0 in range(0, S * L, chunk_rows):
        r1 = min(S * L, r0 + chunk_rows)
        flat[r0:r1] = torch.randn(r1 - r0, d, generator=g, device=device).to(dtype)
    seq, pos = anchor_positions(A, S, L, B, device=device, g=g)
    rows = (seq.long() * L + pos.long())[:, None] + torch.arange(B, device=device)[None, :]
    Hd = torch.empty(N, d, dtype=dtype, device=device)
    rows = rows.reshape(-1)
    for r0 in range(0, N, chunk_rows):
        r1 = min(N, r0 + chunk_rows)
        noise = torch.randn(r1 - r0, d, generator=g, device=device)
        Hd[r0:r1] = (flat[rows[r0:r1]].float() + sigma * noise).to(dtype)
    return dict(W=W, F=F, seq=seq, pos=pos, Hd=Hd)


def corpus_replacement(N, V, rate, *, device="cpu", seed=0):
    """Per-position replacement draw of the erase workload: (mask bool [N], tokens int32 [N]),
    tokens uniform over [0, V)."""
    g = _gen(device, seed + 7919)
    mask = torch.rand(N, generator=g, device=device) < rate
    tok = torch.randint(0, V, (N,), generator=g, device=device, dtype=torch.int32)
    return mask, tok


def corpus_tokens(greedy_tok, mask, tok):
    """Corpus token per row: the greedy target token, or the random one where replaced."""
    return torch.where(mask, tok, greedy_tok.to(torch.int32))



def sharpen(batch, scale=6.0):
    """A head whose logits reach a trained head's magnitude: W scaled by ``scale`` (rounded
    once to the input dtype), so that with d = 4096 the logits spread to |z| of 30-40 instead
    of the random head's |z| < 7.  Returns a new dict; the input dict is untouched."""
    W = batch["W"]
    return dict(batch, W=(W.float() * scale).to(W.dtype))
