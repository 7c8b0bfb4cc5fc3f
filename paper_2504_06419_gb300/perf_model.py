"""The paper's performance model of speculative decoding (Section 2), fed
either by cost estimates or by measured kernel times.

A round of speculation is k draft passes and one verification pass over the
k+1 block tokens.  Its throughput relative to plain decoding is

    throughput multiplier = tau / delta_t,
    delta_t = (k * t_draft + t_verify) / t_target              (iteration time multiplier)

with tau the average number of tokens generated per round.  The
implementation-agnostic form replaces each latency by its forward cost,
max(FLOPs, (weight bytes + KV-cache bytes) * HOI), HOI being the hardware's
FLOPs per byte (compute and memory traffic assumed fully overlapped,
Section 2 and its footnote).  Section 5 turns a multiplier m into the
fraction 1 - 1/m of the decoding budget that speculation saves.

Everything here is host arithmetic; the measured times come from the
library's kernels (bench.py reports `detail.perf_model`).
"""
from __future__ import annotations

import dataclasses


def forward_cost(flops: float, weight_bytes: float, kv_bytes: float, hoi: float) -> float:
    """Cost of one forward pass in FLOP-equivalents: the larger of the compute
    cost and the memory cost (bytes moved times HOI)."""
    return max(float(flops), (float(weight_bytes) + float(kv_bytes)) * float(hoi))


def iteration_time_multiplier(k: int, c_draft: float, n_draft: float, kv_draft: float,
                              c_target: float, n_target: float, kv_target: float,
                              hoi: float) -> float:
    """delta_t from costs: k draft passes plus one verification pass over k+1
    tokens (k+1 times the target's FLOPs, the same bytes), over one target pass.

    c_* are the FLOPs of one single-token forward pass, n_* the weight bytes,
    kv_* the KV-cache bytes read by a pass."""
    draft = forward_cost(c_draft, n_draft, kv_draft, hoi)
    verify = forward_cost((k + 1) * c_target, n_target, kv_target, hoi)
    target = forward_cost(c_target, n_target, kv_target, hoi)
    return (k * draft + verify) / target


def measured_delta_t(k: int, t_draft: float, t_verify: float, t_target: float) -> float:
    """delta_t from measured latencies (any one unit): k draft steps, one
    verification of k+1 tokens, one plain decoding step."""
    return (k * float(t_draft) + float(t_verify)) / float(t_target)


def throughput_multiplier(tau: float, delta_t: float) -> float:
    return float(tau) / float(delta_t)


def decoding_cost_saved(budget_units: float, multiplier: float) -> float:
    """Units of a decoding budget saved by running at `multiplier` times the
    throughput of plain decoding (Section 5)."""
    return float(budget_units) * (1.0 - 1.0 / float(multiplier))


@dataclasses.dataclass(frozen=True)
class ForwardCosts:
    flops: float          # FLOPs of the pass
    weight_bytes: float   # model weights read
    kv_bytes: float       # KV cache read


def transformer_forward_costs(params: float, layers: int, q_width: int, kv_width: int,
                              batch: int, ctx: int, tokens: int = 1,
                              kv_limit: int | None = None, bytes_per_param: float = 2.0,
                              bytes_per_kv: float = 2.0) -> ForwardCosts:
    """Costs of one forward pass of `tokens` new tokens per sequence for a batch
    of `batch` sequences with `ctx` cached entries each.

    params     body parameters (embedding / unembedding ignored, as Section 5 does)
    q_width    query width per layer (heads x head_dim); kv_width likewise for K / V
    kv_limit   cache entries a token may attend (n_sink + window for a
               StreamingLLM draft, Section 3.1); None = the whole context
    FLOPs: 2 per parameter per token plus 4 * q_width per attended entry per
    layer (scores and weighted values); bytes: the weights once and the K and V
    of every attended entry."""
    attended = ctx if kv_limit is None else min(ctx, kv_limit)
    flops = 2.0 * params * batch * tokens + 4.0 * layers * q_width * attended * batch * tokens
    kv = 2.0 * layers * kv_width * attended * batch * bytes_per_kv
    return ForwardCosts(flops, params * bytes_per_param, kv)
