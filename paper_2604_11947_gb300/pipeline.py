"""A decoder-only transformer split into pipeline stages with a ResBM boundary between
consecutive stages, simulated on one GPU (the boundary tensor is handed over in device memory).

Placement (Sec. 3.2, "Placement under pipeline parallelism" and "Preserving the identity path";
the bottleneck follows the feed-forward layer of the last block of a stage):

  last block l of a stage     h = x + Attn(norm(x))                 (x^Attn of the paper)
                              z = FFN(norm(h))                      (the feed-forward output)
                              b = h . P^id + E(z)                   (encode: the only tensor sent)
  first block l+1, reading A  x = b . P^id' + D(b)                  (decode, merge_identity = 1)
                              then the block as usual
  first block l+1, reading B  h = b . P^id' + Attn(norm(D(b)))      (decode, merge_identity = 0:
                              then the FFN half as usual             the pad is added after Attn)

P^id truncates to the first r columns on the send side and zero-pads on the receive side (Eq.
Pid_definition). The encoder and decoder run through the C ABI of libresbm.so
(resbm_encode_fwd / resbm_decode_fwd forward, resbm_decode_bwd / resbm_encode_bwd backward)
inside torch.autograd.Function; everything else (attention, SwiGLU feed-forward, RMSNorm, rotary
positions, embedding, loss) is plain PyTorch in bf16. There is no fallback: without the library
the boundary raises.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, replace

import torch
import torch.nn.functional as Fn

from . import resbm


@dataclass(frozen=True)
class PipelineConfig:
    layers: int = 24
    d: int = 2048
    heads: int = 16
    ffn: int = 5632
    vocab: int = 32000
    stages: int = 4
    r: object = 16           # bottleneck width (d / r compression): one int for every boundary, or a
                             # tuple of stages - 1 widths (a non-uniform r per boundary)
    m: object = 16           # hidden width of the encoder / decoder: an int, or one per boundary
    batch: int = 8
    seq: int = 2048
    act: str = "silu"
    wiring: str = "A"        # "A": decoder output merged with pad(b) and fed to the block;
                             # "B": D(b) feeds the attention branch, pad(b) its skip
    seed: int = 0
    flags: int = 0           # resbm descriptor flags of the boundaries (RESBM_FLAG_*)
    fuse_norm: bool = True   # the receiving block's pre-attention RMSNorm fused into the decoder

    def with_(self, **kw) -> "PipelineConfig":
        return replace(self, **kw)

    @property
    def tokens(self) -> int:
        return self.batch * self.seq

    def boundary_widths(self, k: int):
        """(r, m) of boundary k (between stage k and stage k + 1)."""
        pick = lambda v: int(v[k]) if isinstance(v, (tuple, list)) else int(v)
        return pick(self.r), pick(self.m)


# The workload the boundary's share of a training step is measured on: 24 layers, d = 2048,
# 16 heads, SwiGLU 5632, vocabulary 32000, 4 stages with r = 16 (128x), batch 8 x seq 2048.
PIPELINE = PipelineConfig()


class BoundaryTimer:
    """CUDA events around every boundary call on the launching stream (when enabled)."""

    def __init__(self):
        self.enabled = False
        self.pairs = []

    def start(self):
        if not self.enabled:
            return None
        ev = torch.cuda.Event(enable_timing=True)
        ev.record()
        return ev

    def stop(self, ev):
        if ev is None:
            return
        end = torch.cuda.Event(enable_timing=True)
        end.record()
        self.pairs.append((ev, end))

    def total_ms(self):
        torch.cuda.synchronize()
        return sum(a.elapsed_time(b) for a, b in self.pairs)

    def reset(self):
        self.pairs = []


class _Encode(torch.autograd.Function):
    """b = X[:, :r] + E(F): resbm_encode_fwd forward, resbm_encode_bwd backward (which also adds
    dB into the first r columns of the residual gradient of X)."""

    @staticmethod
    def forward(ctx, X, F, We1, We2, bnd):
        T = X.shape[0]
        desc = bnd.desc(T)
        B = torch.empty(T, bnd.r, dtype=X.dtype, device=X.device)
        P = torch.empty(T, bnd.m, dtype=torch.float32, device=X.device)
        ev = bnd.timer.start()
        resbm.resbm_encode_fwd(desc, X, F, We1, We2, B, P, bnd.workspace(T))
        bnd.timer.stop(ev)
        ctx.save_for_backward(F, P, We1, We2)
        ctx.bnd = bnd
        if bnd.capture is not None:
            bnd.capture.update(X=X.detach(), F=F.detach(), B=B.detach())
        return B

    @staticmethod
    def backward(ctx, dB):
        F, P, We1, We2 = ctx.saved_tensors
        bnd = ctx.bnd
        T, d = F.shape
        dB = dB.contiguous()
        dF = torch.empty_like(F)
        dX = torch.zeros(T, d, dtype=F.dtype, device=F.device)
        dWe1 = torch.empty(d, bnd.m, dtype=torch.float32, device=F.device)
        dWe2 = torch.empty(bnd.m, bnd.r, dtype=torch.float32, device=F.device)
        ev = bnd.timer.start()
        resbm.resbm_encode_bwd(bnd.desc(T), dB, F, P, We1, We2, dF, dX, dWe1, dWe2, bnd.workspace(T))
        bnd.timer.stop(ev)
        if bnd.capture is not None:
            bnd.capture.update(dB_in=dB.detach(), dF=dF, dX=dX, dWe1=dWe1, dWe2=dWe2)
        return dX, dF, dWe1.to(We1.dtype), dWe2.to(We2.dtype), None


class _Decode(torch.autograd.Function):
    """y = [merge] pad(b) + D(b): resbm_decode_fwd forward, resbm_decode_bwd backward."""

    @staticmethod
    def forward(ctx, B, Wd1, Wd2, bnd):
        T = B.shape[0]
        Y = torch.empty(T, bnd.d, dtype=B.dtype, device=B.device)
        ev = bnd.timer.start()
        resbm.resbm_decode_fwd(bnd.desc(T), B, Wd1, Wd2, Y, bnd.workspace(T))
        bnd.timer.stop(ev)
        ctx.save_for_backward(B, Wd1, Wd2)
        ctx.bnd = bnd
        if bnd.capture is not None:
            bnd.capture.update(B_dec=B.detach(), Y=Y.detach())
        return Y

    @staticmethod
    def backward(ctx, dY):
        B, Wd1, Wd2 = ctx.saved_tensors
        bnd = ctx.bnd
        T = B.shape[0]
        dY = dY.contiguous()
        dB = torch.empty_like(B)
        dWd1 = torch.empty(bnd.r, bnd.m, dtype=torch.float32, device=B.device)
        dWd2 = torch.empty(bnd.m, bnd.d, dtype=torch.float32, device=B.device)
        ev = bnd.timer.start()
        resbm.resbm_decode_bwd(bnd.desc(T), dY, B, Wd1, Wd2, dB, dWd1, dWd2, bnd.workspace(T))
        bnd.timer.stop(ev)
        if bnd.capture is not None:
            bnd.capture.update(dY=dY.detach(), dB=dB, dWd1=dWd1, dWd2=dWd2)
        return dB, dWd1.to(Wd1.dtype), dWd2.to(Wd2.dtype), None


NORM_EPS = 1e-5


class _DecodeNorm(torch.autograd.Function):
    """(y, n) = (D(b) [+ pad(b)], RMSNorm(y) * gamma): resbm_decode_fwd_rmsnorm forward (the
    receiving block's pre-attention norm fused into the decoder). Backward: resbm_rmsnorm_bwd adds
    the norm's gradient to dy (and gives dgamma), then resbm_decode_bwd on the sum."""

    @staticmethod
    def forward(ctx, B, Wd1, Wd2, gamma, bnd):
        T = B.shape[0]
        Y = torch.empty(T, bnd.d, dtype=B.dtype, device=B.device)
        N = torch.empty_like(Y)
        ev = bnd.timer.start()
        resbm.resbm_decode_fwd_rmsnorm(bnd.desc(T), B, Wd1, Wd2, gamma, NORM_EPS, Y, N, bnd.workspace(T))
        bnd.timer.stop(ev)
        ctx.save_for_backward(B, Wd1, Wd2, gamma, Y)
        ctx.bnd = bnd
        if bnd.capture is not None:
            bnd.capture.update(B_dec=B.detach(), Y=Y.detach(), N=N.detach(), gamma=gamma.detach())
        return Y, N

    @staticmethod
    def backward(ctx, dY, dN):
        B, Wd1, Wd2, gamma, Y = ctx.saved_tensors
        bnd = ctx.bnd
        T = B.shape[0]
        dgamma = None
        dB = torch.empty_like(B)
        dWd1 = torch.empty(bnd.r, bnd.m, dtype=torch.float32, device=B.device)
        dWd2 = torch.empty(bnd.m, bnd.d, dtype=torch.float32, device=B.device)
        ev = bnd.timer.start()
        if dN is not None:
            dy = torch.empty_like(Y)
            dg = torch.empty(bnd.d, dtype=torch.float32, device=B.device)
            resbm.resbm_rmsnorm_bwd(bnd.desc(T), Y, gamma, NORM_EPS, dN.contiguous(),
                                    None if dY is None else dY.contiguous(), dy, dg, bnd.workspace(T))
            dgamma = dg.to(gamma.dtype)
        else:
            dy = torch.zeros_like(Y) if dY is None else dY.contiguous()
        resbm.resbm_decode_bwd(bnd.desc(T), dy, B, Wd1, Wd2, dB, dWd1, dWd2, bnd.workspace(T))
        bnd.timer.stop(ev)
        if bnd.capture is not None:
            bnd.capture.update(dY=dy.detach(), dB=dB, dWd1=dWd1, dWd2=dWd2)
        return dB, dWd1.to(Wd1.dtype), dWd2.to(Wd2.dtype), dgamma, None


class Boundary(torch.nn.Module):
    """One ResBM boundary: the encoder on the sending stage, the decoder on the receiving one.
    Weights N(0, 1/fan_in), bf16."""

    def __init__(self, d, r, m, act, merge, timer, gen, device, flags=0):
        super().__init__()
        self.d, self.r, self.m, self.act, self.merge, self.flags = d, r, m, act, merge, flags
        self.timer = timer
        self.capture = None   # a dict that receives this boundary's tensors when set

        def w(rows, cols, fan_in):
            t = torch.randn(rows, cols, generator=gen, device=device, dtype=torch.float32) / math.sqrt(fan_in)
            return torch.nn.Parameter(t.to(torch.bfloat16))

        self.We1, self.We2 = w(d, m, d), w(m, r, m)
        self.Wd1, self.Wd2 = w(r, m, r), w(m, d, m)
        self._ws = {}

    def desc(self, T):
        return resbm.make_desc(T, self.d, self.r, self.m, "bf16", self.act, self.merge, self.flags)

    def workspace(self, T):
        ws = self._ws.get(T)
        if ws is None:
            desc = self.desc(T)
            n = max(resbm.resbm_workspace_bytes(desc, op) for op in
                    (resbm.RESBM_OP_ENCODE_FWD, resbm.RESBM_OP_DECODE_FWD, resbm.RESBM_OP_DECODE_BWD,
                     resbm.RESBM_OP_ENCODE_BWD, resbm.RESBM_OP_DECODE_FWD_RMSNORM, resbm.RESBM_OP_RMSNORM_BWD))
            ws = torch.empty(max(n, 1), dtype=torch.uint8, device=self.We1.device)
            self._ws = {T: ws}
        return ws

    def encode(self, h, z):
        return _Encode.apply(h, z, self.We1, self.We2, self)

    def decode(self, b):
        return _Decode.apply(b, self.Wd1, self.Wd2, self)

    def decode_norm(self, b, gamma):
        """(y, RMSNorm(y) * gamma) in one call: the receiving block's attention input with it."""
        return _DecodeNorm.apply(b, self.Wd1, self.Wd2, gamma, self)


def _rope_tables(seq, hd, device):
    inv = 1.0 / (10000.0 ** (torch.arange(0, hd, 2, device=device, dtype=torch.float32) / hd))
    ang = torch.outer(torch.arange(seq, device=device, dtype=torch.float32), inv)
    return ang.cos().to(torch.bfloat16), ang.sin().to(torch.bfloat16)


def _rope(x, cos, sin):
    # x: (batch, heads, seq, hd); rotate the two halves of every head
    x1, x2 = x.chunk(2, dim=-1)
    return torch.cat((x1 * cos - x2 * sin, x2 * cos + x1 * sin), dim=-1)


class Block(torch.nn.Module):
    """Pre-norm decoder block: attention (causal, rotary positions) and a SwiGLU feed-forward."""

    def __init__(self, cfg: PipelineConfig, gen, device):
        super().__init__()
        d, f = cfg.d, cfg.ffn
        self.heads, self.hd = cfg.heads, d // cfg.heads

        def w(rows, cols):
            t = torch.randn(rows, cols, generator=gen, device=device, dtype=torch.float32) * 0.02
            return torch.nn.Parameter(t.to(torch.bfloat16))

        self.n1 = torch.nn.Parameter(torch.ones(d, device=device, dtype=torch.bfloat16))
        self.n2 = torch.nn.Parameter(torch.ones(d, device=device, dtype=torch.bfloat16))
        self.wqkv, self.wo = w(3 * d, d), w(d, d)
        self.w1, self.w3, self.w2 = w(f, d), w(f, d), w(d, f)

    def attn(self, x, rope, normed=None):
        """Attention of the pre-norm block; normed: RMSNorm(x) * n1 when the caller has it."""
        bsz, seq, d = x.shape
        u = Fn.rms_norm(x, (d,), self.n1, NORM_EPS) if normed is None else normed
        qkv = Fn.linear(u, self.wqkv)
        q, k, v = qkv.view(bsz, seq, 3, self.heads, self.hd).permute(2, 0, 3, 1, 4)
        q, k = _rope(q, *rope), _rope(k, *rope)
        o = Fn.scaled_dot_product_attention(q, k, v, is_causal=True)
        return Fn.linear(o.transpose(1, 2).reshape(bsz, seq, d), self.wo)

    def ffn(self, h):
        u = Fn.rms_norm(h, (h.shape[-1],), self.n2, NORM_EPS)
        return Fn.linear(Fn.silu(Fn.linear(u, self.w1)) * Fn.linear(u, self.w3), self.w2)


class PipelineModel(torch.nn.Module):
    """The stages of the transformer with a Boundary between consecutive stages."""

    def __init__(self, cfg: PipelineConfig, device="cuda"):
        super().__init__()
        assert cfg.layers % cfg.stages == 0 and cfg.wiring in ("A", "B")
        self.cfg = cfg
        gen = torch.Generator(device=device)
        gen.manual_seed(cfg.seed)
        self.timer = BoundaryTimer()
        self.embed = torch.nn.Parameter(
            torch.randn(cfg.vocab, cfg.d, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16))
        self.blocks = torch.nn.ModuleList(Block(cfg, gen, device) for _ in range(cfg.layers))
        merge = 1 if cfg.wiring == "A" else 0
        for v in (cfg.r, cfg.m):
            assert not isinstance(v, (tuple, list)) or len(v) == cfg.stages - 1, "one width per boundary"
        self.bounds = torch.nn.ModuleList(Boundary(cfg.d, *cfg.boundary_widths(k), cfg.act, merge, self.timer, gen,
                                                   device, cfg.flags) for k in range(cfg.stages - 1))
        self.norm = torch.nn.Parameter(torch.ones(cfg.d, device=device, dtype=torch.bfloat16))
        self.head = torch.nn.Parameter(
            (torch.randn(cfg.vocab, cfg.d, generator=gen, device=device, dtype=torch.float32) * 0.02).to(torch.bfloat16))
        self._rope = {}

    def rope(self, seq, device):
        if seq not in self._rope:
            self._rope[seq] = _rope_tables(seq, self.cfg.d // self.cfg.heads, device)
        return self._rope[seq]

    def forward(self, tokens):
        """Mean next-token cross-entropy of a (batch, seq) tensor of token ids."""
        cfg = self.cfg
        bsz, seq = tokens.shape
        T, d = bsz * seq, cfg.d
        rope = self.rope(seq, tokens.device)
        per_stage = cfg.layers // cfg.stages
        x = Fn.embedding(tokens, self.embed)
        b = None
        for s in range(cfg.stages):
            for j in range(per_stage):
                blk = self.blocks[s * per_stage + j]
                if j == 0 and s > 0:   # receive: decode the boundary tensor of the previous stage
                    bnd = self.bounds[s - 1]
                    if cfg.fuse_norm:   # the block's attention norm comes out of the decoder
                        y, n = bnd.decode_norm(b, blk.n1)
                        y, n = y.view(bsz, seq, d), n.view(bsz, seq, d)
                    else:
                        y, n = bnd.decode(b).view(bsz, seq, d), None
                    if cfg.wiring == "A":
                        x = y                                       # pad(b) + D(b)
                        h = x + blk.attn(x, rope, n)
                    else:
                        h = Fn.pad(b, (0, d - bnd.r)).view(bsz, seq, d) + blk.attn(y, rope, n)   # pad(b) + Attn(D(b))
                else:
                    h = x + blk.attn(x, rope)
                z = blk.ffn(h)
                if j == per_stage - 1 and s < cfg.stages - 1:   # send: encode after the feed-forward
                    b = self.bounds[s].encode(h.reshape(T, d), z.reshape(T, d))
                else:
                    x = h + z
        logits = Fn.linear(Fn.rms_norm(x, (d,), self.norm, NORM_EPS), self.head)
        return Fn.cross_entropy(logits[:, :-1].reshape(-1, cfg.vocab).float(), tokens[:, 1:].reshape(-1))


def synthetic_tokens(cfg: PipelineConfig, device="cuda", seed=1):
    """Uniform random token ids in [0, vocab), shape (batch, seq)."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return torch.randint(0, cfg.vocab, (cfg.batch, cfg.seq), generator=g, device=device)


def train_step(model: PipelineModel, tokens):
    """One training step's forward and backward (gradients left in .grad); returns the loss."""
    model.zero_grad(set_to_none=True)
    loss = model(tokens)
    loss.backward()
    return loss


def time_steps(model: PipelineModel, tokens, steps, warmup):
    """Mean ms per training step and the boundary kernels' ms per step (CUDA events around every
    C-ABI call of the boundaries, on the launching stream)."""
    for _ in range(warmup):
        train_step(model, tokens)
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    model.timer.reset()
    model.timer.enabled = True
    start.record()
    for _ in range(steps):
        loss = train_step(model, tokens)
    end.record()
    torch.cuda.synchronize()
    model.timer.enabled = False
    step_ms = start.elapsed_time(end) / steps
    bnd_ms = model.timer.total_ms() / steps
    model.timer.reset()
    return step_ms, bnd_ms, float(loss.detach())


# ---- convergence on a learnable synthetic stream ----------------------------------------------
def markov_batches(cfg: PipelineConfig, n_batches, seed=2, branching=4, device="cuda"):
    """n_batches x (batch, seq) token ids drawn from a seeded random Markov chain: every token has
    `branching` possible successors with Dirichlet(1) probabilities, so the stream is learnable
    down to the chain's entropy rate. Returns (tokens on the GPU, entropy rate in nats)."""
    import numpy as np
    rng = np.random.default_rng(seed)
    succ = rng.integers(0, cfg.vocab, size=(cfg.vocab, branching))
    probs = rng.dirichlet(np.ones(branching), size=cfg.vocab)
    cum = np.cumsum(probs, axis=1)
    n = n_batches * cfg.batch
    out = np.empty((n, cfg.seq), np.int64)
    cur = rng.integers(0, cfg.vocab, size=n)
    for t in range(cfg.seq):
        out[:, t] = cur
        pick = np.minimum((rng.random(n)[:, None] > cum[cur]).sum(axis=1), branching - 1)
        cur = succ[cur, pick]
    # stationary entropy rate: the chain's per-token entropies weighted by visit frequency
    counts = np.bincount(out[:, :-1].ravel(), minlength=cfg.vocab).astype(np.float64)
    h = -(probs * np.log(probs)).sum(axis=1)
    rate = float((counts * h).sum() / counts.sum())
    return torch.from_numpy(out).view(n_batches, cfg.batch, cfg.seq).to(device), rate


def train_curve(cfg: PipelineConfig, data, steps, lr=1e-3, every=25):
    """AdamW on the model's parameters over `steps` batches of `data` (cycled); the loss at step
    0, every `every` steps and at the end (mean of the last `every` steps' losses)."""
    model = PipelineModel(cfg)
    opt = torch.optim.AdamW(model.parameters(), lr=lr, weight_decay=0.01)
    curve, window = [], []
    for s in range(steps):
        loss = train_step(model, data[s % data.shape[0]])
        opt.step()
        window.append(loss.detach())
        if s == 0 or (s + 1) % every == 0:
            curve.append((s + 1, float(torch.stack(window).mean())))
            window = []
    del model, opt
    return curve


# The convergence comparison: a 4-layer model in 2 stages (one boundary, r = 16, 32x) against the
# same model with no boundary (1 stage), on a 256-token Markov stream.
CONVERGENCE = PipelineConfig(layers=4, d=512, heads=8, ffn=1024, vocab=256, stages=2, r=16, m=16, batch=16,
                             seq=256)


def convergence(steps=300, lr=1e-3):
    """Loss curves of wiring A (pad(b) + D(b) into the block), wiring B (D(b) into the attention
    branch, pad(b) its skip) and the uncompressed model, on the same data and initial seed; a
    fresh batch every step, so the losses approach the stream's entropy rate from above."""
    data, rate = markov_batches(CONVERGENCE, steps)
    res = {"entropy_rate": rate, "steps": steps, "lr": lr}
    for name, cfg in (("A", CONVERGENCE), ("B", CONVERGENCE.with_(wiring="B")),
                      ("uncompressed", CONVERGENCE.with_(stages=1))):
        res[name] = train_curve(cfg, data, steps, lr)
    return res
