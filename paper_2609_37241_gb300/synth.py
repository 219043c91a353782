"""Seeded synthetic inputs shaped like the decode workloads the paper evaluates.

This module only draws random data and builds buffers; it holds none of the method's
arithmetic. Both the CUDA path and the CPU oracle consume what it returns: activations
as bit patterns (numpy uint16 for bf16/fp16, uint32 for fp32), so the two sides read
identical bytes. Conversion of the fp32 draws to bf16/fp16 is torch's CPU cast (round
to nearest even).

Workloads (the paper evaluates Qwen3-8B and DeepSeek-V2-Lite decoding at batch size one,
§4.1; no weights or datasets are used here -- activations are N(0,1), norm weights
N(1, 0.1), positions uniform without replacement):
  * llama decode layer:  H 4096, 32 q heads, 8 kv heads, D 128, I 14336, theta 5e5,
                         KV cache [8, 8192, 128]
  * qwen3 decode layer:  H 4096, 32/8 heads, D 128, I 12288, theta 1e6, q/k norm, 36 layers
  * guard stress:        T ~ Zipf(1.2) truncated to [1, 512]; 10% fp16; 5% row-strided
  * bandwidth sweep:     T = 2^0 .. 2^15, H 8192, I 28672
"""
import numpy as np
import torch

BF16, FP16, FP32 = 1, 2, 3
CACHE_SENTINEL = 0x5A5A  # bit pattern pre-filled into KV caches (a finite bf16/fp16 value)

LLAMA = dict(H=4096, Hq=32, Hkv=8, D=128, S=8192, I=14336, theta=500000.0, qknorm=False,
             eps=1e-6)
QWEN3 = dict(H=4096, Hq=32, Hkv=8, D=128, S=8192, I=12288, theta=1000000.0, qknorm=True,
             eps=1e-6, layers=36)
SWEEP = dict(H=8192, I=28672, eps=1e-6)
STRESS = dict(H=4096, n_calls=100_000, zipf_a=1.2, t_lo=1, t_hi=512, p_fp16=0.10,
              p_strided=0.05, pad=64, eps=1e-6)

_TORCH_DT = {BF16: torch.bfloat16, FP16: torch.float16, FP32: torch.float32}


def rng(seed=0):
    return np.random.default_rng(seed)


def to_bits(f32, dtype):
    """Cast float32 values to `dtype` (torch, RNE) and return their bit patterns."""
    t = torch.from_numpy(np.ascontiguousarray(f32, np.float32))
    if dtype == FP32:
        return t.numpy().view(np.uint32).copy()
    return t.to(_TORCH_DT[dtype]).view(torch.int16).numpy().view(np.uint16).copy()


def bits_to_torch(bits, dtype):
    """CPU torch tensor of `dtype` holding exactly these bit patterns."""
    if dtype == FP32:
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.float32).copy())
    raw = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16).copy())
    return raw.view(_TORCH_DT[dtype])


def torch_to_bits(t, dtype):
    """Bit patterns of a torch tensor (any device) as numpy."""
    t = t.detach().contiguous().cpu()
    if dtype == FP32:
        return t.view(torch.int32).numpy().view(np.uint32).copy()
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def act(g, shape, dtype, mean=0.0, std=1.0):
    """Activation bits drawn from N(mean, std) in fp32, then cast."""
    return to_bits(g.normal(mean, std, size=shape).astype(np.float32), dtype)


def gamma(g, n):
    """Norm weight, fp32 ~ N(1, 0.1)."""
    return g.normal(1.0, 0.1, size=n).astype(np.float32)


def positions(g, T, S):
    """T distinct cache positions, uniform in [0, S)."""
    return g.choice(S, size=T, replace=False).astype(np.int32)


def cache(Hkv, S, D):
    """KV cache bits pre-filled with the sentinel."""
    return np.full((Hkv, S, D), CACHE_SENTINEL, np.uint16)


def layer_inputs(g, T, cfg, dtype=BF16):
    """One decoder layer's chain inputs (bits) for T tokens; the GEMM outputs that the
    chain consumes (q/k/v, attention output, gate and up) are synthetic N(0,1)."""
    H, Hq, Hkv, D, S, I = cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]
    d = dict(
        h=act(g, (T, H), dtype), r0=act(g, (T, H), dtype), gamma_attn=gamma(g, H),
        q=act(g, (T, Hq, D), dtype), k=act(g, (T, Hkv, D), dtype), v=act(g, (T, Hkv, D), dtype),
        pos=positions(g, T, S), k_cache=cache(Hkv, S, D), v_cache=cache(Hkv, S, D),
        attn_out=act(g, (T, H), dtype), gamma_mlp=gamma(g, H),
        g=act(g, (T, I), dtype), u=act(g, (T, I), dtype),
    )
    if cfg.get("qknorm"):
        d["gamma_q"] = gamma(g, D)
        d["gamma_k"] = gamma(g, D)
    return d


def zipf_tokens(g, n, a, lo, hi):
    """n token counts from Zipf(a) truncated to [lo, hi] (p(k) proportional to k^-a)."""
    k = np.arange(lo, hi + 1, dtype=np.float64)
    p = k ** (-a)
    p /= p.sum()
    return g.choice(k.astype(np.int64), size=n, p=p)


def stress_trace(g, cfg=STRESS):
    """(T, dtype, strided) per call of the dynamic-shape guard stress."""
    n = cfg["n_calls"]
    T = zipf_tokens(g, n, cfg["zipf_a"], cfg["t_lo"], cfg["t_hi"])
    dt = np.where(g.random(n) < cfg["p_fp16"], FP16, BF16).astype(np.int32)
    strided = (g.random(n) < cfg["p_strided"])
    return T, dt, strided


def act_device(shape, dtype, seed, device="cuda", mean=0.0, std=1.0):
    """Large activation drawn on the device by torch's seeded generator (N(mean, std) in
    fp32, then cast): for full-size workloads where host generation would dominate."""
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    t = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
    if std != 1.0 or mean != 0.0:
        t = t * std + mean
    return t.to(_TORCH_DT[dtype])


def gamma_device(n, seed, device="cuda"):
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    return torch.randn(n, generator=gen, device=device, dtype=torch.float32) * 0.1 + 1.0
