"""Seeded synthetic inputs for the elbow-routed MoE layer.

This module only draws random numbers and lays them out; it holds none of the
routing, dispatch or expert arithmetic. Both the CPU oracle and the CUDA path
are fed from here, so that the two sides see bit-identical inputs.

The workloads stand in for the paper's OLMoE-1B-7B evaluation (64 experts,
top-8, d_model 2048, SwiGLU intermediate 1024, 16 MoE layers; Sec. 2, App. A.4),
whose weights and benchmark prompts are not available. Token vectors follow the
signal-noise picture of Sec. 2.2: a token is a sum of a few routing-relevant
directions (one per "signal" expert) plus isotropic noise, so that its sorted
router probabilities have a head of high-confidence experts and a flat tail.

Recipe (numpy PCG64, seed fixed per workload, draws in this order):
  1. router weights W_r[N, d] ~ N(0, 1/sqrt(d)) (std), rounded to bf16;
     unit directions W_hat[j] = W_r[j] / ||W_r[j]|| from the fp32 draws.
  2. tokens: |S_t| ~ U{1..12}; S_t = first |S_t| experts of a uniformly random
     permutation; a_j ~ U(2, 5);  x_t = sum_j a_j W_hat[j] + N(0, 0.3^2) per
     coordinate, rounded to bf16.  For the wide-router workload a fraction of
     tokens (20 %) is "flat": |S_t| ~ U{24..40}, a_j ~ U(0.5, 1).
  3. expert weights W_gu[N, 2I, d] (rows [0, I) gate, rows [I, 2I) up) and
     W_d[N, d, I], all ~ N(0, 0.02^2), rounded to bf16; expert e draws from its
     own stream PCG64(SeedSequence([seed, e])).
Routing-only stress logits: l = N(0, 1) + U(2, 5) on a random 1..12 experts per
token, drawn directly in fp32.

bf16 tensors are carried as uint16 bit patterns (round to nearest even).
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

__all__ = [
    "WORKLOADS",
    "bf16_bits",
    "bf16_bits_to_f32",
    "router_weights",
    "tokens",
    "expert_weights",
    "boosted_logits",
    "stack_inputs",
    "stack_expert_seed",
    "layer_inputs",
]

# Named workloads (shapes of the paper's OLMoE setting, App. A.4).
WORKLOADS = {
    # small layer: the oracle runs it in seconds
    "layer_t64": dict(T=64, d=2048, N=64, I=1024, K=8, seed=1001),
    # routing-only stress: 1,048,576 tokens x 64 fp32 logits
    "route_t1m": dict(T=1048576, N=64, K=8, seed=1002),
    # one OLMoE-shaped layer at prefill scale
    "layer_t16k": dict(T=16384, d=2048, N=64, I=1024, K=8, seed=1003),
    # wider router with 20 % flat tokens
    "layer_wide": dict(T=8192, d=4096, N=128, I=1536, K=8, seed=1004, flat_frac=0.2),
    # 16-layer stack, residual between layers; layer l uses seed 5000 + l
    "stack16_t4k": dict(T=4096, d=2048, N=64, I=1024, K=8, L=16, seed=1005),
}


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest, ties to even
    (finite inputs)."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    r = (u >> 16) & np.uint32(1)
    r += np.uint32(0x7FFF)
    r += u
    r >>= 16
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> fp32 (exact)."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def router_weights(rng: np.random.Generator, N: int, d: int):
    """W_r ~ N(0, 1/sqrt(d)) as bf16 bits, plus fp32 unit rows W_hat."""
    w = rng.standard_normal((N, d), dtype=np.float32) * np.float32(1.0 / np.sqrt(d))
    w_hat = w / np.linalg.norm(w, axis=1, keepdims=True)
    return bf16_bits(w), w_hat.astype(np.float32)


def _subsets(rng: np.random.Generator, T: int, N: int, lo: int, hi: int):
    """Per token: size ~ U{lo..hi}; members = first `size` of a random permutation."""
    size = rng.integers(lo, hi + 1, size=T)
    order = np.argsort(rng.random((T, N), dtype=np.float32), axis=1)
    rank = np.empty_like(order)
    np.put_along_axis(rank, order, np.arange(N)[None, :].repeat(T, 0), axis=1)
    return rank < size[:, None]  # [T, N] bool membership


def tokens(rng: np.random.Generator, T: int, w_hat: np.ndarray, flat_frac: float = 0.0):
    """Token matrix x[T, d] (bf16 bits) built from the signal-noise recipe."""
    N, d = w_hat.shape
    member = _subsets(rng, T, N, 1, min(12, N))
    amp = rng.uniform(2.0, 5.0, size=(T, N)).astype(np.float32)
    if flat_frac > 0.0:
        flat = rng.random(T) < flat_frac
        fmember = _subsets(rng, T, N, min(24, N), min(40, N))
        famp = rng.uniform(0.5, 1.0, size=(T, N)).astype(np.float32)
        member = np.where(flat[:, None], fmember, member)
        amp = np.where(flat[:, None], famp, amp)
    coef = np.where(member, amp, np.float32(0.0)).astype(np.float32)
    x = np.empty((T, d), dtype=np.uint16)
    step = 4096
    for t0 in range(0, T, step):
        t1 = min(T, t0 + step)
        sig = coef[t0:t1] @ w_hat
        noise = rng.standard_normal((t1 - t0, d), dtype=np.float32) * np.float32(0.3)
        x[t0:t1] = bf16_bits(sig + noise)
    return x


def expert_weights(seed: int, N: int, d: int, I: int):
    """W_gu[N, 2I, d] (gate rows then up rows) and W_d[N, d, I], bf16 bits.

    Expert e draws from its own stream PCG64(SeedSequence([seed, e])) (W_gu
    first, then W_d), so the result does not depend on the thread count."""
    wgu = np.empty((N, 2 * I, d), dtype=np.uint16)
    wd = np.empty((N, d, I), dtype=np.uint16)
    s = np.float32(0.02)

    def one(e):
        g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, e])))
        wgu[e] = bf16_bits(g.standard_normal((2 * I, d), dtype=np.float32) * s)
        wd[e] = bf16_bits(g.standard_normal((d, I), dtype=np.float32) * s)

    with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
        list(ex.map(one, range(N)))
    return wgu, wd


def stack_inputs(T: int, d: int, N: int, L: int, seed: int):
    """Inputs of an L-layer stack: the tokens x_0 and layer 0's router follow the
    layer recipe (seed); layer l >= 1 draws its own router from
    PCG64(SeedSequence([seed, l])). Experts: expert_weights(seed * 100 + l, ...)."""
    first = layer_inputs(T=T, d=d, N=N, I=0, seed=seed, with_experts=False)
    routers = [first["w_router"]]
    for l in range(1, L):
        g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, l])))
        routers.append(router_weights(g, N, d)[0])
    return first["x"], routers


def stack_expert_seed(seed: int, l: int) -> int:
    return seed * 100 + l


def boosted_logits(rng: np.random.Generator, T: int, N: int, chunk: int = 1 << 17):
    """fp32 logits: N(0,1) baseline + U(2,5) boost on a random 1..12 experts."""
    out = np.empty((T, N), dtype=np.float32)
    for t0 in range(0, T, chunk):
        t1 = min(T, t0 + chunk)
        n = t1 - t0
        base = rng.standard_normal((n, N), dtype=np.float32)
        member = _subsets(rng, n, N, 1, min(12, N))
        boost = rng.uniform(2.0, 5.0, size=(n, N)).astype(np.float32)
        out[t0:t1] = base + np.where(member, boost, np.float32(0.0))
    return out


def layer_inputs(T: int, d: int, N: int, I: int, seed: int, flat_frac: float = 0.0,
                 with_experts: bool = True):
    """All inputs of one MoE layer: x, W_r, W_gu, W_d (bf16 bits)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    wr, w_hat = router_weights(rng, N, d)
    x = tokens(rng, T, w_hat, flat_frac)
    out = dict(x=x, w_router=wr)
    if with_experts:
        out["w_gate_up"], out["w_down"] = expert_weights(seed, N, d, I)
    return out
