"""Seeded synthetic workloads for SPIRe speculation-round attention.

This module only draws inputs: shapes, random values, context lengths, page
tables and NaN poisoning.  It holds none of the attention arithmetic, and both
sides of every parity check (the CUDA library and the fp64 oracle) read the
very tensors it returns.

The paper measures on LongCrawl64 (Section 4), which is not available here and
not needed: the kernels' cost depends only on shapes and lengths.  These
inputs stand in for it:
  * K, V ~ N(0, 1) and Q ~ N(0, 1) / sqrt(D), all rounded to bf16, so the
    softmax scale is 1.0;
  * context lengths fixed, uniform or log-uniform per config, drawn with
    numpy.random.default_rng(seed);
  * paged caches of 64-token pages with a seeded random page permutation
    (an identity table for the tiny contiguous config);
  * optional NaN poisoning of every cache slot no query may see.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np
import torch

PAGE = 64


@dataclasses.dataclass(frozen=True)
class Config:
    name: str
    batch: int
    ctx_dist: str            # "fixed" | "list" | "uniform" | "loguniform"
    ctx_lo: int
    ctx_hi: int
    k: int                   # speculation depth (k+1 verify rows)
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    n_sink: int
    window: int
    seed: int
    paged_shuffle: bool = True
    ctx_list: tuple = ()
    windows: tuple = ()      # draft sweep only

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads


CONFIGS = {
    # Tiny correctness case: contiguous KV, 4 query heads over 1 KV head, D=64.
    "tiny": Config("tiny", 2, "list", 256, 300, 4, 4, 1, 64, 4, 64, 1,
                   paged_shuffle=False, ctx_list=(256, 300)),
    # Uniform long context: B=64, L=8192, k=4, 32/8 heads, D=128.
    "uniform8k": Config("uniform8k", 64, "fixed", 8192, 8192, 4, 32, 8, 128, 16, 512, 2),
    # Ragged serving mix: L log-uniform in [1024, 131072].
    "ragged": Config("ragged", 64, "loguniform", 1024, 131072, 4, 32, 8, 128, 16, 1024, 3),
    # Large batch, deeper speculation: B=256, L uniform in [16384, 32768], k=8, 64/8.
    "big": Config("big", 256, "uniform", 16384, 32768, 8, 64, 8, 128, 32, 2048, 4),
    # Draft sweep: B=512, L log-uniform in [4096, 262144], sink 16, three windows.
    "draft_sweep": Config("draft_sweep", 512, "loguniform", 4096, 262144, 4, 32, 8, 128,
                          16, 1024, 5, windows=(256, 1024, 4096)),
}


def sample_ctx_lens(cfg: Config, seed: int | None = None) -> np.ndarray:
    """Context lengths of a config, int32 [B]."""
    rng = np.random.default_rng(cfg.seed if seed is None else seed)
    B = cfg.batch
    if cfg.ctx_dist == "fixed":
        L = np.full(B, cfg.ctx_lo)
    elif cfg.ctx_dist == "list":
        L = np.array(cfg.ctx_list[:B])
    elif cfg.ctx_dist == "uniform":
        L = rng.integers(cfg.ctx_lo, cfg.ctx_hi + 1, size=B)
    elif cfg.ctx_dist == "loguniform":
        u = rng.uniform(math.log(cfg.ctx_lo), math.log(cfg.ctx_hi), size=B)
        L = np.floor(np.exp(u))
    else:
        raise ValueError(cfg.ctx_dist)
    return np.clip(L, cfg.ctx_lo, cfg.ctx_hi).astype(np.int32)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _randn_bf16(shape, gen, device, std: float = 1.0) -> torch.Tensor:
    x = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(torch.bfloat16)


def _randn_bf16_inplace(t: torch.Tensor, gen, chunk_elems: int = 1 << 28):
    """Fill a (possibly huge) bf16 tensor with N(0,1) in chunks."""
    flat = t.view(-1)
    for s in range(0, flat.numel(), chunk_elems):
        e = min(flat.numel(), s + chunk_elems)
        tmp = torch.randn(e - s, generator=gen, device=t.device, dtype=torch.float32)
        flat[s:e].copy_(tmp)
    return t


@dataclasses.dataclass
class VerifyInputs:
    q: torch.Tensor            # bf16 [B, k+1, Hq, D]
    k_cache: torch.Tensor      # bf16 [num_pages, Hkv, 64, D]
    v_cache: torch.Tensor
    block_table: torch.Tensor  # int32 [B, max_pages]
    ctx_lens: torch.Tensor     # int32 [B]
    k: int
    scale: float = 1.0

    @property
    def shape(self):
        B, kp1, Hq, D = self.q.shape
        return dict(batch=B, num_q_heads=Hq, num_kv_heads=self.k_cache.shape[1],
                    head_dim=D, page_size=self.k_cache.shape[2],
                    max_pages_per_seq=self.block_table.shape[1],
                    num_pages=self.k_cache.shape[0], softmax_scale=self.scale)


@dataclasses.dataclass
class DraftInputs:
    q: torch.Tensor            # bf16 [B, Hq, D]
    kv: torch.Tensor           # bf16 [B, 2, Hkv, S, D]
    ctx_lens: torch.Tensor     # int32 [B]
    n_sink: int
    window: int
    scale: float = 1.0

    @property
    def shape(self):
        B, Hq, D = self.q.shape
        return dict(batch=B, num_q_heads=Hq, num_kv_heads=self.kv.shape[2], head_dim=D,
                    page_size=PAGE, max_pages_per_seq=0, num_pages=0,
                    softmax_scale=self.scale)


def make_verify(ctx_lens, k: int, num_q_heads: int, num_kv_heads: int, head_dim: int,
                *, seed: int, device="cpu", shuffle: bool = True, poison: bool = False,
                spare_pages: int = 0, max_pages: int | None = None,
                q_std: float | None = None) -> VerifyInputs:
    """Paged verification inputs.

    ctx_lens  lengths L_b (including the k+1 block tokens).
    shuffle   seeded random physical page order (else pages in sequence order).
    poison    fill every cache slot that no query may see with NaN: the tail of
              each sequence's last page and every page no sequence references.
    """
    L = np.asarray(ctx_lens, dtype=np.int64)
    B = int(L.size)
    pages = (L + PAGE - 1) // PAGE
    mp = int(pages.max()) if B else 0
    if max_pages is not None:
        mp = max(mp, int(max_pages))
    num_pages = int(pages.sum()) + int(spare_pages)
    rng = np.random.default_rng(seed + 1000)
    order = rng.permutation(num_pages) if shuffle else np.arange(num_pages)
    bt = np.full((B, max(mp, 1)), -1, dtype=np.int32)
    off = 0
    for b in range(B):
        bt[b, :pages[b]] = order[off:off + pages[b]]
        off += pages[b]
    gen = _gen(seed, device)
    q_std = (1.0 / math.sqrt(head_dim)) if q_std is None else q_std
    q = _randn_bf16((B, k + 1, num_q_heads, head_dim), gen, device, q_std)
    kc = torch.empty((max(num_pages, 1), num_kv_heads, PAGE, head_dim), dtype=torch.bfloat16,
                     device=device)
    vc = torch.empty_like(kc)
    _randn_bf16_inplace(kc, gen)
    _randn_bf16_inplace(vc, gen)
    if poison and num_pages:
        used = np.zeros((max(num_pages, 1), PAGE), dtype=bool)
        for b in range(B):
            for p in range(pages[b]):
                n = min(PAGE, int(L[b]) - p * PAGE)
                used[bt[b, p], :n] = True
        bad = torch.from_numpy(~used).to(device)
        kc.permute(0, 2, 1, 3)[bad] = float("nan")
        vc.permute(0, 2, 1, 3)[bad] = float("nan")
    return VerifyInputs(q=q, k_cache=kc, v_cache=vc,
                        block_table=torch.from_numpy(bt).to(device),
                        ctx_lens=torch.from_numpy(L.astype(np.int32)).to(device), k=k)


def make_draft(ctx_lens, num_q_heads: int, num_kv_heads: int, head_dim: int,
               n_sink: int, window: int, *, seed: int, device="cpu",
               poison: bool = False, q_std: float | None = None) -> DraftInputs:
    """Bounded draft cache [B, 2, Hkv, n_sink + window, D] with random contents.

    poison  fill slots >= min(t_b, S), which hold no visible memory entry, with NaN.
    """
    t = np.asarray(ctx_lens, dtype=np.int64)
    B = int(t.size)
    S = n_sink + window
    gen = _gen(seed, device)
    q_std = (1.0 / math.sqrt(head_dim)) if q_std is None else q_std
    q = _randn_bf16((B, num_q_heads, head_dim), gen, device, q_std)
    kv = torch.empty((B, 2, num_kv_heads, S, head_dim), dtype=torch.bfloat16, device=device)
    _randn_bf16_inplace(kv, gen)
    if poison:
        for b in range(B):
            n = int(min(max(t[b], 0), S))
            if n < S:
                kv[b, :, :, n:, :] = float("nan")
    return DraftInputs(q=q, kv=kv, ctx_lens=torch.from_numpy(t.astype(np.int32)).to(device),
                       n_sink=n_sink, window=window)


@dataclasses.dataclass
class AppendInputs:
    x: torch.Tensor           # bf16 [n_act, B, d_model]: the token's activations
    mix_w: torch.Tensor       # fp32 [n_dl, n_act]: mixing weights (un-normalised)
    w_kv: torch.Tensor        # bf16 [n_dl, 2*Hkv*D, d_model]: key rows, then value rows
    pos: torch.Tensor         # int32 [B]: logical position of the new entry
    kv: torch.Tensor          # bf16 [n_dl, B, 2, Hkv, n_sink + window, D]: caches
    n_sink: int
    window: int


def make_append(pos, num_act: int, num_draft_layers: int, d_model: int, num_kv_heads: int,
                head_dim: int, n_sink: int, window: int, *, seed: int,
                device="cpu") -> AppendInputs:
    """Inputs of the feedback-memory append: N(0,1) activations and mixing
    weights, N(0, 1/d_model) projections (entries of order 1), caches filled
    with N(0,1) bf16 so that untouched slots are recognisable."""
    p = np.asarray(pos, dtype=np.int64)
    B = int(p.size)
    S = n_sink + window
    gen = _gen(seed, device)
    x = _randn_bf16((num_act, B, d_model), gen, device)
    mix_w = torch.randn((num_draft_layers, num_act), generator=gen, device=device,
                        dtype=torch.float32)
    F = 2 * num_kv_heads * head_dim
    w_kv = _randn_bf16((num_draft_layers, F, d_model), gen, device, 1.0 / math.sqrt(d_model))
    kv = torch.empty((num_draft_layers, B, 2, num_kv_heads, S, head_dim), dtype=torch.bfloat16,
                     device=device)
    _randn_bf16_inplace(kv, gen)
    return AppendInputs(x=x, mix_w=mix_w, w_kv=w_kv,
                        pos=torch.from_numpy(p.astype(np.int32)).to(device), kv=kv,
                        n_sink=n_sink, window=window)


@dataclasses.dataclass
class TokenInputs:
    p: torch.Tensor       # fp32 [B, k+1, V]: target distributions
    q: torch.Tensor       # fp32 [B, k, V]: draft distributions
    x: torch.Tensor       # int32 [B, k]: draft tokens, x_i drawn from q_i
    u: torch.Tensor       # fp32 [B, k]: uniforms in [0, 1)
    e: torch.Tensor       # fp32 [B, V]: Exp(1) variates


def make_tokens(batch: int, k: int, vocab: int, *, seed: int, device="cpu",
                logit_std: float = 2.0, draft_noise: float = 1.0) -> TokenInputs:
    """Distributions of one speculation round: target logits N(0, logit_std^2)
    per vocabulary entry, draft logits = target logits + N(0, draft_noise^2)
    (a draft that roughly agrees with the target), both through a softmax;
    draft tokens drawn from the draft distributions; uniforms and Exp(1)
    variates from the same seeded generator."""
    gen = _gen(seed, device)
    zt = torch.randn((batch, k + 1, vocab), generator=gen, device=device) * logit_std
    zd = zt[:, :k] + torch.randn((batch, k, vocab), generator=gen, device=device) * draft_noise
    p = torch.softmax(zt, dim=-1).float().contiguous()
    q = torch.softmax(zd, dim=-1).float().contiguous()
    if k > 0:
        x = torch.multinomial(q.reshape(batch * k, vocab), 1, generator=gen).reshape(batch, k)
    else:
        x = torch.zeros((batch, 0), dtype=torch.int64, device=device)
    u = torch.rand((batch, k), generator=gen, device=device)
    e = torch.empty((batch, vocab), device=device).exponential_(1.0, generator=gen)
    return TokenInputs(p=p, q=q, x=x.to(torch.int32).contiguous(), u=u.contiguous(),
                       e=e.contiguous())


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Raw bf16 bit patterns of a tensor as a host uint16 numpy array."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def draft_ctx_for_step(verify_ctx: np.ndarray, k: int, j: int) -> np.ndarray:
    """Memory entries visible to draft step j (0..k-1) of a round whose verify
    pass sees L_b cache entries: t = L_b - k + j."""
    return (np.asarray(verify_ctx, dtype=np.int64) - k + j).astype(np.int32)
