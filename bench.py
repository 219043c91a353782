"""Benchmark of the SCM hot path on GB300: one JSON line on stdout (rank 0).

Headline ("value"): microseconds per decoder-layer step of the Llama-style non-GEMM chain
at 64 tokens (H 4096, 32/8 heads, D 128, I 14336, theta 5e5, KV cache [8, 8192, 128]):
one trident_scm_invoke per step from Python -- guards, argument packing and one fused
launch -- timed with CUDA events over K back-to-back steps, inputs rotated over enough
buffer sets that the working set exceeds twice the L2.

Also reported on the same line: every token count of that workload fused and unfused,
the 36-layer Qwen3-style step, host nanoseconds per cache hit (single add+RMSNorm call,
1 token), the 100k-call dynamic-shape guard stress (hit/miss counts checked against the
oracle replay), the HBM bandwidth sweep (add+RMSNorm and SwiGLU, 1..32768 tokens), the
roofline of the dominant kernel, the end-to-end step with host copies, and the CPU
oracle as a reported baseline.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference] [--quick]
                 [--sections LIST] [--tokens LIST]
"""
import argparse
import ctypes
import json
import math
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "us per decoder-layer step (host dispatch+device) at 1-64 tok; HBM GB/s vs 8 TB/s"
UNIT = "us/step"
HEADLINE_T = 64
HEADLINE_LEAD_CYCLES = 50000  # about 24 us at 2.07 GHz: the device's lead over the host
HEADLINE_LEAD_STEPS = 8  # untimed warm-up steps queued right behind the lead, ahead of the window
L2_BYTES = 129 * 2 ** 20
NOMINAL_HBM_GBS = 8000.0


CHAIN_SOURCES = ["paper_2609_37241_gb300/csrc/chain.cu", "paper_2609_37241_gb300/csrc/device_common.cuh",
                 "paper_2609_37241_gb300/csrc/internal.h"]
CHAIN_COUNTERS = "profiles/chain_kernel_llama_t64.json"


def chain_sources_sha256():
    import hashlib
    h = hashlib.sha256()
    for f in CHAIN_SOURCES:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def chain_traffic():
    """DRAM bytes per launch of the chain kernel, read and written, from the committed ncu
    counters (profiles/chain_kernel_llama_t64.json: dram__bytes_read.sum and
    dram__bytes_write.sum averaged over consecutive launches of the headline workload), or
    None when the kernel sources changed since those counters were taken."""
    try:
        with open(os.path.join(ROOT, CHAIN_COUNTERS)) as fh:
            d = json.load(fh)
        if d["source_sha256"] != chain_sources_sha256():
            return None
        return int(d["dram_bytes_read_per_launch"]), int(d["dram_bytes_write_per_launch"])
    except Exception:
        return None


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# ---------------------------------------------------------------------------- algorithmic bytes
def chain_bytes_per_token(cfg, fused=True):
    """Bytes one token moves through the layer chain (bf16 activations)."""
    H, Hq, Hkv, D, I = cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["I"]
    norm1 = 4 * H * 2                       # read h, r0; write x1, r1
    norm2 = (3 if fused else 4) * H * 2     # read attn_out (+ r1 unfused); write x2, r2
    rope = (2 * Hq * D + 2 * Hkv * D + 2 * Hkv * D) * 2 + 4  # q in/out, k in/out, v in/out, pos
    swiglu = 3 * I * 2
    return norm1 + norm2 + rope + swiglu


def chain_read_write_bytes(cfg, T):
    """(read, write) split of the fused chain's algorithmic bytes per launch."""
    H, Hq, Hkv, D, I = cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["I"]
    rope_rows = (Hq + 2 * Hkv) * D * 2
    read = 2 * H * 2 + H * 2 + rope_rows + 4 + 2 * I * 2
    write = 2 * H * 2 + 2 * H * 2 + rope_rows + I * 2
    g = 2 * H * 4 + (2 * D * 4 if cfg.get("qknorm") else 0) + D * 4
    return T * read + g, T * write


def chain_bytes_per_launch(cfg, T, fused=True):
    # norm weights (+ q/k norm weights) and the RoPE frequency table, once per launch
    g = 2 * cfg["H"] * 4 + (2 * cfg["D"] * 4 if cfg.get("qknorm") else 0) + cfg["D"] * 4
    return T * chain_bytes_per_token(cfg, fused) + g


# ---------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampling during the measured region (stopped by the caller)."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.proc = None
        self.dev = device_index
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(device_index), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = max(mx, float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        busy = [s for s in sm if s > 0.5 * mx] or sm
        return {"sm_mhz": float(np.median(busy)), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------- oracle (reference arm)
def oracle_layer_step_us(cfg, T, budget_s, seed=0):
    """The CPU oracle timed on a bounded sample of layer steps at T tokens."""
    from oracle import layer as L
    from paper_2609_37241_gb300 import synth
    g = np.random.default_rng(seed)
    inp = synth.layer_inputs(g, T, cfg)
    L.layer_chain(inp, cfg["theta"], cfg["eps"], synth.BF16, qknorm=cfg.get("qknorm", False))  # warm
    n, t0 = 0, time.perf_counter()
    while True:
        L.layer_chain(inp, cfg["theta"], cfg["eps"], synth.BF16, qknorm=cfg.get("qknorm", False))
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s and n >= 2:
            break
    return el / n * 1e6, n


# ---------------------------------------------------------------------------- GPU side
class Ctx:
    def __init__(self, device):
        import torch
        from paper_2609_37241_gb300 import scm as S
        from paper_2609_37241_gb300 import synth
        self.torch, self.S, self.synth = torch, S, synth
        self.dev = device
        self.stream = torch.cuda.current_stream()
        self.sp = ctypes.c_void_p(self.stream.cuda_stream)
        self.L = S.lib()
        self.fc = S.fastcall()  # CPython fast-call shim of the binding (None: ctypes only)
        self.launches = 0

    def invoker(self, scm):
        """fn(args_struct_or_address) -> status: one trident_scm_invoke from Python."""
        h, sp = scm.h.value, self.sp.value or 0  # the default stream is NULL
        if self.fc is not None:
            inv = self.fc.invoke
            return lambda addr: inv(h, addr, sp)
        inv, hh, spp = self.L.trident_scm_invoke, scm.h, self.sp
        P = ctypes.POINTER(self.S.trident_args)
        return lambda addr: inv(hh, ctypes.cast(addr, P), spp, None)

    def seq_invoker(self, scm):
        h, sp = scm.h.value, self.sp.value or 0
        if self.fc is not None:
            seq = self.fc.invoke_seq
            return lambda addr, n: seq(h, addr, n, sp)
        seq, hh, spp = self.L.trident_scm_invoke_seq, scm.h, self.sp
        P = ctypes.POINTER(self.S.trident_args)
        return lambda addr, n: seq(hh, ctypes.cast(addr, P), n, spp, None)

    def step_invoker(self, scm):
        h, sp = scm.h.value, self.sp.value or 0
        if self.fc is not None:
            stp = self.fc.invoke_step
            return lambda addr, n: stp(h, addr, n, sp)
        stp, hh, spp = self.L.trident_scm_invoke_step, scm.h, self.sp
        P = ctypes.POINTER(self.S.trident_args)
        return lambda addr, n: stp(hh, ctypes.cast(addr, P), n, spp, None)

    def events(self):
        t = self.torch
        return t.cuda.Event(enable_timing=True), t.cuda.Event(enable_timing=True)


class ChainSets:
    """R rotating input/output sets of one decoder layer at T tokens, carved from arenas,
    plus per-layer norm weights and KV caches."""

    def __init__(self, c, cfg, T, layers=1, min_bytes=2 * L2_BYTES, max_sets=4096, seed=0):
        t, synth = c.torch, c.synth
        self.cfg, self.T, self.layers = cfg, T, layers
        H, Hq, Hkv, D, S, I = (cfg[k] for k in ("H", "Hq", "Hkv", "D", "S", "I"))
        per_set = chain_bytes_per_token(cfg) * T
        R = max(layers, int(math.ceil(min_bytes / per_set)))
        R = min(max_sets, int(math.ceil(R / layers)) * layers)
        self.R = R
        W = (Hq + 2 * Hkv) * D
        bf = t.bfloat16
        dev = c.dev
        self.h = synth.act_device((R, T, H), synth.BF16, seed + 1, dev)
        self.r0 = synth.act_device((R, T, H), synth.BF16, seed + 2, dev)
        self.ao = synth.act_device((R, T, H), synth.BF16, seed + 3, dev)
        self.qkv = synth.act_device((R, T, W), synth.BF16, seed + 4, dev)
        self.gu = synth.act_device((R, T, 2 * I), synth.BF16, seed + 5, dev)
        self.x1 = t.empty((R, T, H), dtype=bf, device=dev)
        self.r1 = t.empty((R, T, H), dtype=bf, device=dev)
        self.x2 = t.empty((R, T, H), dtype=bf, device=dev)
        self.r2 = t.empty((R, T, H), dtype=bf, device=dev)
        self.o = t.empty((R, T, I), dtype=bf, device=dev)
        g = np.random.default_rng(seed)
        self.pos = t.from_numpy(np.stack([synth.positions(g, T, S) for _ in range(R)])).to(dev)
        self.ga = [synth.gamma_device(H, seed + 10 + l, dev) for l in range(layers)]
        self.gm = [synth.gamma_device(H, seed + 100 + l, dev) for l in range(layers)]
        self.gq = [synth.gamma_device(D, seed + 200 + l, dev) for l in range(layers)]
        self.gk = [synth.gamma_device(D, seed + 300 + l, dev) for l in range(layers)]
        self.kc = [t.zeros((Hkv, S, D), dtype=bf, device=dev) for _ in range(layers)]
        self.vc = [t.zeros((Hkv, S, D), dtype=bf, device=dev) for _ in range(layers)]

    def slots(self, i, layer=0):
        cfg = self.cfg
        Hq, Hkv, D, I = cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["I"]
        T = self.T
        qkv = self.qkv[i]
        q = qkv[:, :Hq * D].view(T, Hq, D)
        k = qkv[:, Hq * D:(Hq + Hkv) * D].view(T, Hkv, D)
        v = qkv[:, (Hq + Hkv) * D:].view(T, Hkv, D)
        gu = self.gu[i]
        ts = [self.h[i], self.r0[i], self.ga[layer], self.x1[i], self.r1[i], q, k, v, self.pos[i],
              self.kc[layer], self.vc[layer], self.ao[i], self.gm[layer], self.x2[i], self.r2[i],
              gu[:, :I], gu[:, I:], self.o[i]]
        if cfg.get("qknorm"):
            ts += [self.gq[layer], self.gk[layer]]
        return ts

    def fused_args(self, c, i, layer=0):
        S = c.S
        op = S.OP_LAYER_CHAIN_QKNORM if self.cfg.get("qknorm") else S.OP_LAYER_CHAIN
        return S.make_args(op, self.slots(i, layer), eps=self.cfg["eps"], rope_theta=self.cfg["theta"])

    def unfused_args(self, c, i, layer=0):
        S = c.S
        ts = self.slots(i, layer)
        (h, r0, ga, x1, r1, q, k, v, pos, kc, vc, ao, gm, x2, r2, g, u, o) = ts[:18]
        if self.cfg.get("qknorm"):
            rope = S.make_args(S.OP_QKNORM_ROPE_KV, [q, k, v, pos, kc, vc, ts[18], ts[19]],
                               eps=self.cfg["eps"], rope_theta=self.cfg["theta"])
        else:
            rope = S.make_args(S.OP_ROPE_KV, [q, k, v, pos, kc, vc], rope_theta=self.cfg["theta"])
        return [S.make_args(S.OP_ADD_RMSNORM, [h, r0, ga, x1, r1], eps=self.cfg["eps"]), rope,
                S.make_args(S.OP_ADD_RMSNORM, [ao, r1, gm, x2, r2], eps=self.cfg["eps"]),
                S.make_args(S.OP_SWIGLU, [g, u, o])]


def layer_scm(c, cfg, pdl=True, timing=False, replay=False):
    """One SCM holding the layer's versions: the fused chain (index 0), then the four
    single-step versions, all for token buckets 1..4096 and row-strided q/k/v and g/u.
    invoke_step's replay cache is off unless `replay`: the rotating-set lines measure the
    full path (selection, byte rules and packing on every step)."""
    S = c.S
    flags = (S.OPT_PDL if pdl else 0) | (S.OPT_TIMING if timing else 0) | (0 if replay else S.OPT_NO_STEP_REPLAY)
    s = S.Scm(device=c.dev.index or 0, flags=flags)
    qk = cfg.get("qknorm", False)
    fixed = [cfg[k] for k in ("H", "Hq", "Hkv", "D", "S", "I")]
    op = S.OP_LAYER_CHAIN_QKNORM if qk else S.OP_LAYER_CHAIN
    for lay in (S.LAYOUT_ROWSTRIDED, S.LAYOUT_CONTIG):
        s.register(S.make_spec(op, S.BF16, fixed, 1, 4096, layout=lay, rope_theta=cfg["theta"]))
    s.register(S.make_spec(S.OP_ADD_RMSNORM, S.BF16, [cfg["H"]], 1, 4096))
    rop = S.OP_QKNORM_ROPE_KV if qk else S.OP_ROPE_KV
    for lay in (S.LAYOUT_ROWSTRIDED, S.LAYOUT_CONTIG):
        s.register(S.make_spec(rop, S.BF16, fixed[1:5], 1, 4096, layout=lay, rope_theta=cfg["theta"]))
        s.register(S.make_spec(S.OP_SWIGLU, S.BF16, [cfg["I"]], 1, 4096, layout=lay))
    return s


def assert_all_hit(scm, what):
    """Every timed call must have been a cache hit that launched (no silent misses)."""
    st = scm.stats()
    if st.misses or st.err_invalid or st.err_cuda or st.hits != st.invokes:
        raise RuntimeError(f"{what}: {st.invokes} invokes, {st.hits} hits, {st.misses} misses, "
                           f"{st.err_invalid} invalid, {st.err_cuda} cuda errors")
    return st.hits


def max_over_ranks(x, world, device="cpu"):
    """The largest value of x over all ranks (the job's time is its slowest replica)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def time_steps(c, fn, K, W, lead_cycles=0):
    """Runs fn(i) for W warm-up then K timed steps; returns (us per step on the device
    clock, host us per step). With lead_cycles, a sleep kernel of that many cycles runs
    ahead of the first timed step (outside the window), so the window opens on a busy
    device with the first steps already queued."""
    t = c.torch
    for i in range(W):
        fn(i)
    t.cuda.synchronize()
    e0, e1 = c.events()
    if lead_cycles:
        t.cuda._sleep(lead_cycles)
    h0 = time.perf_counter()
    e0.record(c.stream)
    for i in range(K):
        fn(W + i)
    e1.record(c.stream)
    h1 = time.perf_counter()
    t.cuda.synchronize()
    return e0.elapsed_time(e1) * 1e3 / K, (h1 - h0) * 1e6 / K


def bench_layer(c, cfg, T, K, W, layers=1, min_bytes=2 * L2_BYTES):
    """Fused and unfused layer steps at T tokens (one Python call per step)."""
    S = c.S
    sets = ChainSets(c, cfg, T, layers=layers, min_bytes=min_bytes)
    scm = layer_scm(c, cfg)
    R = sets.R
    fused = [sets.fused_args(c, i, i % layers) for i in range(R)]
    unf = [(S.trident_args * 4)(*sets.unfused_args(c, i, i % layers)) for i in range(R)]
    inv, seq = c.invoker(scm), c.seq_invoker(scm)
    h, sp = scm.h, c.sp
    faddr = [ctypes.addressof(a) for a in fused]
    uaddr = [ctypes.addressof(a) for a in unf]
    if layers == 1:
        f_fused = lambda i: inv(faddr[i % R])
        f_unf = lambda i: seq(uaddr[i % R], 4)
        n_launch = (1, 4)
    else:  # one step = `layers` layers through one call
        groups = R // layers
        farr = [(S.trident_args * layers)(*fused[g * layers:(g + 1) * layers]) for g in range(groups)]
        uarr = [(S.trident_args * (4 * layers))(*[a for l in range(layers) for a in
                                                   sets.unfused_args(c, g * layers + l, l)])
                for g in range(groups)]
        fa = [ctypes.addressof(x) for x in farr]
        ua = [ctypes.addressof(x) for x in uarr]
        f_fused = lambda i: seq(fa[i % groups], layers)
        f_unf = lambda i: seq(ua[i % groups], 4 * layers)
        n_launch = (layers, 4 * layers)
    st, sel = S.trident_scm_invoke(h, fused[0], c.sp.value)
    assert st == S.OK and sel in (0, 1), S.trident_scm_last_error()
    # the warm-up visits every rotating set once, so that no timed step is the first touch of
    # its buffers (the rotation exists only to keep the working set larger than the L2)
    W = max(W, R if layers == 1 else R // layers)
    fus_dev, fus_host = time_steps(c, f_fused, K, W)
    unf_dev, unf_host = time_steps(c, f_unf, K, W)
    c.launches += K * (n_launch[0] + n_launch[1])
    step = None
    if layers > 1:  # the same layers through invoke_step: independent chains, one launch
        stp = c.step_invoker(scm)
        before = scm.stats().fused_launches
        step_dev, step_host = time_steps(c, lambda i: stp(fa[i % groups], layers), K, W)
        per_step = -(-layers // S.STEP_MAX)
        fused_n = scm.stats().fused_launches - before
        assert fused_n == (K + W) * per_step, ("step launches not fused", fused_n)
        c.launches += K * per_step
        step = dict(us=round(step_dev, 3), host_us=round(step_host, 3), launches_per_step=per_step)
        # A decode loop with static buffers passes the same argument arrays every step:
        # invoke_step relaunches them from its replay cache (no selection, byte rules or
        # packing). As many rotating arrays as the cache keeps (4); working set reported.
        rs = layer_scm(c, cfg, replay=True)
        rstp = c.step_invoker(rs)
        nrep = min(groups, 4)
        for i in range(2 * nrep):  # seen, then stored
            rstp(fa[i % nrep], layers)
        before = rs.stats().step_replays
        rep_dev, rep_host = time_steps(c, lambda i: rstp(fa[i % nrep], layers), K, W)
        replayed = rs.stats().step_replays - before
        assert replayed == (K + W) * layers, ("steps not replayed", replayed)
        assert_all_hit(rs, "replayed step T=%d" % T)
        rs.close()
        c.launches += K * per_step
        step["replayed"] = dict(us=round(rep_dev, 3), host_us=round(rep_host, 3), arrays=nrep,
                                working_set_mb=round(nrep * layers * chain_bytes_per_token(cfg) * T / 2 ** 20, 1))
    # device throughput floor: the same launches issued from one native call
    nat = min(K, R if layers == 1 else R)
    if layers == 1:
        arr = (S.trident_args * nat)(*fused[:nat])
        arr_addr = ctypes.addressof(arr)
        nat_fn = lambda i: seq(arr_addr, nat)
        nat_us, _ = time_steps(c, nat_fn, 4, 2)
        nat_us /= nat
        c.launches += 4 * nat
    else:
        nat_us = None
    st, bits = S.trident_scm_device_status(h, c.sp.value)
    assert st == S.OK and bits == 0
    assert_all_hit(scm, "layer T=%d" % T)
    scm.close()
    res = dict(fused_us=round(fus_dev, 3), fused_host_us=round(fus_host, 3), unfused_us=round(unf_dev, 3),
               unfused_host_us=round(unf_host, 3), launches_per_step=list(n_launch), sets=R,
               working_set_mb=round(R * chain_bytes_per_token(cfg) * T / 2 ** 20, 1))
    if nat_us is not None:
        res["fused_native_seq_us"] = round(nat_us, 3)
    if step is not None:
        res["one_launch_step"] = step
    return res, sets


def bench_launch_floor(c, n=2000):
    """Single-launch latency floor: an empty kernel launched back to back through the
    library's own launch path (trident_launch_floor: same context, driver entry point and
    launch attributes as a hit), with and without programmatic dependent launch. Device us
    per launch from CUDA events around one native call of n launches; host us per launch
    from the host clock around the same call."""
    S, t = c.S, c.torch
    res = {}
    for name, flags in (("pdl", S.OPT_PDL), ("no_pdl", 0)):
        s = S.Scm(device=c.dev.index or 0, flags=flags | S.OPT_TIMING)
        assert S.trident_launch_floor(s.h, c.sp.value, 20) == S.OK, S.trident_scm_last_error()
        t.cuda.synchronize()
        e0, e1 = c.events()
        h0 = time.perf_counter()
        e0.record(c.stream)
        st = S.trident_launch_floor(s.h, c.sp.value, n)
        e1.record(c.stream)
        h1 = time.perf_counter()
        t.cuda.synchronize()
        assert st == S.OK, S.trident_scm_last_error()
        # the launch call alone, per launch (library clock), in bursts of 32 with the queue
        # drained in between -- the same pattern as the host cost per hit
        for _ in range(1000 // 32 + 1):
            assert S.trident_launch_floor(s.h, c.sp.value, 32) == S.OK, S.trident_scm_last_error()
            t.cuda.synchronize()
        ns = np.array(S.trident_scm_host_times(s.h, 1000)[1], np.float64)
        res[name] = dict(device_us=round(e0.elapsed_time(e1) * 1e3 / n, 3),
                         host_us=round((h1 - h0) * 1e6 / n, 3),
                         launch_call_ns=dict(median=float(np.median(ns)), p99=float(np.percentile(ns, 99)),
                                             samples=int(ns.size)))
        s.close()
    c.launches += 2 * (n + 20 + 32 * (1000 // 32 + 1))
    return res


def add_floor_fractions(per_t, floor_us, layers=1):
    """Fraction of the single-launch latency floor (n_launches x the empty-kernel launch
    time) that each decode-size step reaches: 1.0 would be a step as fast as its launches."""
    for v in per_t.values():
        n_fused, n_unf = v["launches_per_step"]
        v["floor_frac"] = dict(fused=round(n_fused * floor_us / v["fused_us"], 3),
                               unfused=round(n_unf * floor_us / v["unfused_us"], 3))
        o = v.get("one_launch_step")
        if o:
            v["floor_frac"]["one_launch_step"] = round(o["launches_per_step"] * floor_us / o["us"], 3)
            if "replayed" in o:
                v["floor_frac"]["replayed"] = round(o["launches_per_step"] * floor_us / o["replayed"]["us"], 3)


def bench_e2e(c, cfg, T, K, W):
    """End to end through the public API: per step, one pinned host -> device copy of the
    layer's inputs (h, r0, attn_out, qkv, gate|up, pos laid out in one staging arena), one
    invoke, one device -> host copy of its outputs (x1, x2, r2, o in one arena).

    Steps are double-buffered over three streams, as a serving engine overlaps transfers:
    step i+1's input copy (copy-in stream) runs while step i's kernel (the bench stream) and
    step i's output copy (copy-out stream) run; events order each buffer's reuse. The timed
    region starts before the first step's input copy and ends after the last step's output
    copy. The same steps issued serially (copy in, invoke, copy out on one stream) are
    reported beside it."""
    t, S, synth = c.torch, c.S, c.synth
    H, Hq, Hkv, D, Sl, I = (cfg[k] for k in ("H", "Hq", "Hkv", "D", "S", "I"))
    Wq = (Hq + 2 * Hkv) * D

    def layout(parts):
        offs, o = [], 0
        for nbytes in parts:
            offs.append(o)
            o += (nbytes + 255) // 256 * 256
        return offs, o

    in_parts = [T * H * 2, T * H * 2, T * H * 2, T * Wq * 2, T * 2 * I * 2, T * 4]
    out_parts = [T * H * 2, T * H * 2, T * H * 2, T * I * 2]
    ioffs, itot = layout(in_parts)
    ooffs, otot = layout(out_parts)
    view = lambda buf, o, n, dt, shape: buf[o:o + n].view(dt).view(shape)
    bf = t.bfloat16
    r1 = t.empty((T, H), dtype=bf, device=c.dev)
    kc = t.zeros((Hkv, Sl, D), dtype=bf, device=c.dev)
    vc = t.zeros((Hkv, Sl, D), dtype=bf, device=c.dev)
    ga, gm = synth.gamma_device(H, 50, c.dev), synth.gamma_device(H, 51, c.dev)
    scm = layer_scm(c, cfg)
    bufs = []
    for k in range(2):
        dev_in = t.empty(itot, dtype=t.uint8, device=c.dev)
        dev_out = t.empty(otot, dtype=t.uint8, device=c.dev)
        host_in = t.empty(itot, dtype=t.uint8, pin_memory=True)
        host_out = t.empty(otot, dtype=t.uint8, pin_memory=True)
        h = view(dev_in, ioffs[0], in_parts[0], bf, (T, H))
        r0 = view(dev_in, ioffs[1], in_parts[1], bf, (T, H))
        ao = view(dev_in, ioffs[2], in_parts[2], bf, (T, H))
        qkv = view(dev_in, ioffs[3], in_parts[3], bf, (T, Wq))
        gu = view(dev_in, ioffs[4], in_parts[4], bf, (T, 2 * I))
        pos = view(dev_in, ioffs[5], in_parts[5], t.int32, (T,))
        for j, tv in enumerate((h, r0, ao, qkv, gu)):
            tv.copy_(synth.act_device(tuple(tv.shape), S.BF16, 40 + 10 * k + j, c.dev))
        pos.copy_(t.from_numpy(synth.positions(np.random.default_rng(1 + k), T, Sl)).to(c.dev))
        host_in.copy_(dev_in)
        x1 = view(dev_out, ooffs[0], out_parts[0], bf, (T, H))
        x2 = view(dev_out, ooffs[1], out_parts[1], bf, (T, H))
        r2 = view(dev_out, ooffs[2], out_parts[2], bf, (T, H))
        o = view(dev_out, ooffs[3], out_parts[3], bf, (T, I))
        ts = [h, r0, ga, x1, r1, qkv[:, :Hq * D].view(T, Hq, D), qkv[:, Hq * D:(Hq + Hkv) * D].view(T, Hkv, D),
              qkv[:, (Hq + Hkv) * D:].view(T, Hkv, D), pos, kc, vc, ao, gm, x2, r2, gu[:, :I], gu[:, I:], o]
        a = S.make_args(S.OP_LAYER_CHAIN, ts, eps=cfg["eps"], rope_theta=cfg["theta"])
        bufs.append(dict(dev_in=dev_in, dev_out=dev_out, host_in=host_in, host_out=host_out, args=a,
                         addr=ctypes.addressof(a)))
    t.cuda.synchronize()
    inv = c.invoker(scm)
    main = c.stream
    s_in, s_out = t.cuda.Stream(device=c.dev), t.cuda.Stream(device=c.dev)
    ev = lambda: t.cuda.Event()
    kdone = [ev(), ev()]    # kernel k finished reading dev_in[k]
    odone = [ev(), ev()]    # output copy k finished reading dev_out[k]
    ready = [ev(), ev()]    # input copy k landed
    made = [ev(), ev()]     # kernel k wrote dev_out[k]
    started = [False, False]

    def pipelined(i):
        k = i % 2
        b = bufs[k]
        with t.cuda.stream(s_in):
            if started[k]:
                s_in.wait_event(kdone[k])
            b["dev_in"].copy_(b["host_in"], non_blocking=True)
            ready[k].record(s_in)
        main.wait_event(ready[k])
        if started[k]:
            main.wait_event(odone[k])
        inv(b["addr"])
        kdone[k].record(main)
        made[k].record(main)
        with t.cuda.stream(s_out):
            s_out.wait_event(made[k])
            b["host_out"].copy_(b["dev_out"], non_blocking=True)
            odone[k].record(s_out)
        started[k] = True

    def run(fn, n):
        e0, e1 = c.events()
        e0.record(main)
        s_in.wait_event(e0)
        s_out.wait_event(e0)
        for i in range(n):
            fn(i)
        for k in range(2):
            if started[k]:
                main.wait_event(odone[k])
        e1.record(main)
        t.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / max(n, 1)

    run(pipelined, W)
    us = run(pipelined, K)
    # each buffer's inputs are the same every step and the kernel is deterministic, so the
    # pipelined outputs must equal a serial recomputation byte for byte
    piped = [b["host_out"].clone() for b in bufs]

    def serial(i):
        b = bufs[i % 2]
        b["dev_in"].copy_(b["host_in"], non_blocking=True)
        inv(b["addr"])
        b["host_out"].copy_(b["dev_out"], non_blocking=True)

    with t.cuda.stream(main):
        time_steps(c, serial, W, 1)
        serial_us, _ = time_steps(c, serial, K, W)
    t.cuda.synchronize()
    for k, b in enumerate(bufs):
        if not t.equal(piped[k], b["host_out"]):
            raise RuntimeError("e2e: pipelined outputs differ from the serial recomputation")
    assert_all_hit(scm, "e2e")
    c.launches += 3 * W + 2 * K + 1  # pipelined W + K, serial (W + 1) + (W + K)
    scm.close()
    return dict(value=round(us, 3), unit=UNIT, h2d_bytes_per_step=int(sum(in_parts)),
                d2h_bytes_per_step=int(sum(out_parts)), copies_per_step=2,
                pipeline="double-buffered: input copy of step i+1 overlaps kernel and output copy of step i",
                serial_us=round(serial_us, 3))


def bench_host_hit(c, n=1000):
    """Single add+RMSNorm, 1 token, H 4096; four versions (fp16 contig, fp16 strided,
    bf16 strided, bf16 contig) so each hit evaluates four guards. Host ns per hit from
    the library's own clock (entry to return, the launch call included; launched as the
    library launches in production, with programmatic serialisation), per call as seen
    from Python, and the guards, validation and packing alone (dry run). On the Grace host
    the driver's launch call alone takes about 1.4 us (median) and 2.0 us (p99); the
    library's own work is the dry-run figure."""
    t, S, synth = c.torch, c.S, c.synth
    s = S.Scm(device=c.dev.index or 0, flags=S.OPT_TIMING | S.OPT_PDL)
    for dt in (S.FP16, S.BF16):
        for lay in ((S.LAYOUT_CONTIG, S.LAYOUT_ROWSTRIDED) if dt == S.FP16 else
                    (S.LAYOUT_ROWSTRIDED, S.LAYOUT_CONTIG)):
            s.register(S.make_spec(S.OP_ADD_RMSNORM, dt, [4096], 1, 1, layout=lay))
    g = np.random.default_rng(0)
    x = c.synth.bits_to_torch(synth.act(g, (1, 4096), synth.BF16), synth.BF16).to(c.dev)
    r = c.synth.bits_to_torch(synth.act(g, (1, 4096), synth.BF16), synth.BF16).to(c.dev)
    gam = t.from_numpy(synth.gamma(g, 4096)).to(c.dev)
    y, ro = t.empty_like(x), t.empty_like(r)
    a = S.make_args(S.OP_ADD_RMSNORM, [x, r, gam, y, ro], eps=1e-6)
    inv, ar, sel = c.L.trident_scm_invoke, ctypes.byref(a), ctypes.c_int32(-1)
    for _ in range(50):
        inv(s.h, ar, c.sp, ctypes.byref(sel))
    t.cuda.synchronize()
    # back to back: the device (about 2 us per call without PDL) is slower than the host, so
    # the launch queue fills and some launches wait for room in it -- back-pressure, not
    # dispatch cost; those samples are reported separately
    h0 = time.perf_counter()
    for _ in range(n):
        inv(s.h, ar, c.sp, ctypes.byref(sel))
    h1 = time.perf_counter()
    t.cuda.synchronize()
    st, bb_ns = S.trident_scm_host_times(s.h, n)
    bb_ns = np.array(bb_ns[-n:], np.float64)
    # dispatch cost: the same calls in bursts of 32 with the queue drained in between (a
    # decode step issues a few dozen calls, then waits for its results), warm caches; from
    # the fast-call shim (the binding the headline uses) and, for comparison, from ctypes,
    # whose own work between calls (about 1 us) leaves colder caches for the next call
    def bursts(call):
        for _ in range(n // 32 + 1):
            for _ in range(32):
                call()
            t.cuda.synchronize()
        return np.array(S.trident_scm_host_times(s.h, n)[1][-n:], np.float64)

    ns_ctypes = bursts(lambda: inv(s.h, ar, c.sp, ctypes.byref(sel)))
    ns, binding = ns_ctypes, "ctypes"
    if c.fc is not None:
        fhit, fh, fa, fs = c.fc.invoke, s.h.value, ctypes.addressof(a), c.sp.value or 0
        ns, binding = bursts(lambda: fhit(fh, fa, fs)), "fastcall"
    fast_us = None
    if c.fc is not None:
        finv, hh, addr, sp = c.fc.invoke, s.h.value, ctypes.addressof(a), c.sp.value or 0
        f0 = time.perf_counter()
        for _ in range(n):
            finv(hh, addr, sp)
        f1 = time.perf_counter()
        t.cuda.synchronize()
        fast_us = round((f1 - f0) * 1e6 / n, 3)
        c.launches += n
    # guards, validation and packing alone: the same table and call on a dry-run SCM
    d = S.Scm(device=c.dev.index or 0, flags=S.OPT_TIMING | S.OPT_DRY_RUN)
    for dt in (S.FP16, S.BF16):
        for lay in ((S.LAYOUT_CONTIG, S.LAYOUT_ROWSTRIDED) if dt == S.FP16 else
                    (S.LAYOUT_ROWSTRIDED, S.LAYOUT_CONTIG)):
            d.register(S.make_spec(S.OP_ADD_RMSNORM, dt, [4096], 1, 1, layout=lay))
    for _ in range(n + 50):
        c.L.trident_scm_invoke(d.h, ar, c.sp, None)
    dns = np.array(S.trident_scm_host_times(d.h, n)[1], np.float64)
    d.close()
    hits = S.trident_scm_spec_hits(s.h)[1]
    # one call at a time (after the samples above were read): device us from an event
    # recorded before the call to one after it, and host us from the call to the return of
    # that event's synchronise (launch to completion)
    e0, e1 = c.events()
    ev_us, wall_us = [], []
    for _ in range(200):
        t.cuda.synchronize()
        w0 = time.perf_counter()
        e0.record(c.stream)
        inv(s.h, ar, c.sp, ctypes.byref(sel))
        e1.record(c.stream)
        e1.synchronize()
        w1 = time.perf_counter()
        ev_us.append(e0.elapsed_time(e1) * 1e3)
        wall_us.append((w1 - w0) * 1e6)
    assert_all_hit(s, "host dispatch")
    c.launches += 2 * n + 32 * (n // 32 + 1) * (2 if c.fc is not None else 1) + 200
    s.close()
    # the fused layer chain (18 tensors, 64 tokens): host ns per hit with the launch, and alone
    cfg = synth.LLAMA
    sets = ChainSets(c, cfg, HEADLINE_T, min_bytes=0, max_sets=1)
    chain_ns = {}
    for label, flags in (("live", S.OPT_TIMING | S.OPT_PDL), ("guards_only", S.OPT_TIMING | S.OPT_DRY_RUN)):
        cs = S.Scm(device=c.dev.index or 0, flags=flags)
        fixed = [cfg[k] for k in ("H", "Hq", "Hkv", "D", "S", "I")]
        cs.register(S.make_spec(S.OP_LAYER_CHAIN, S.BF16, fixed, 1, 4096, layout=S.LAYOUT_ROWSTRIDED,
                                rope_theta=cfg["theta"]))
        ca = sets.fused_args(c, 0)
        cinv, caddr = c.invoker(cs), ctypes.addressof(ca)
        for _ in range(50):
            cinv(caddr)
        t.cuda.synchronize()
        for _ in range(n // 32 + 1):  # in bursts, as above (a device step is longer than a call)
            for _ in range(32):
                cinv(caddr)
            t.cuda.synchronize()
        cns = np.array(S.trident_scm_host_times(cs.h, n)[1], np.float64)
        chain_ns[label] = dict(median_ns=float(np.median(cns)), p99_ns=float(np.percentile(cns, 99)))
        if label == "live":
            assert_all_hit(cs, "chain host")
            c.launches += 50 + 32 * (n // 32 + 1)
        cs.close()
    del sets
    return dict(hits_on_bf16_contig=int(hits[3]), calls=n, selected=sel.value, layer_chain=chain_ns,
                isolated_call=dict(event_us_median=round(float(np.median(ev_us)), 3),
                                   launch_to_completion_us_median=round(float(np.median(wall_us)), 3),
                                   calls=len(ev_us)),
                median_ns=float(np.median(ns)), p99_ns=float(np.percentile(ns, 99)), binding=binding,
                ctypes_bursts=dict(median_ns=float(np.median(ns_ctypes)),
                                   p99_ns=float(np.percentile(ns_ctypes, 99))),
                min_ns=float(ns.min()), guards_only_median_ns=float(np.median(dns)),
                guards_only_p99_ns=float(np.percentile(dns, 99)),
                back_to_back=dict(median_ns=float(np.median(bb_ns)), p99_ns=float(np.percentile(bb_ns, 99)),
                                  note="launch queue full: launches wait for room"),
                python_call_us_ctypes=round((h1 - h0) * 1e6 / n, 3), python_call_us_fastcall=fast_us)


def bench_guard_stress(c, n_calls=None):
    """100k add+RMSNorm calls with T ~ Zipf(1.2) on [1,512], 10% fp16, 5% row-strided.
    Static mode: 16 pre-registered versions (buckets 1..128 x {bf16, fp16}); a miss is
    served by a second SCM of generic catch-all versions. Growth mode: the hook
    registers the bucket's version and re-invokes. Selections are compared with the
    oracle's replay of the same trace (memoised per distinct tuple and table size)."""
    t, S, synth = c.torch, c.S, c.synth
    from oracle import guards as G
    cfg = dict(synth.STRESS)
    if n_calls:
        cfg["n_calls"] = n_calls
    g = np.random.default_rng(0)
    Ts, dts, strided = synth.stress_trace(g, cfg)
    H, pad = cfg["H"], cfg["pad"]
    Tmax = int(Ts.max())
    bufs = {}
    for dt in (S.BF16, S.FP16):
        tdt = synth._TORCH_DT[dt]
        bufs[dt] = [t.randn((Tmax, H + pad), device=c.dev).to(tdt) for _ in range(4)]
    gam = synth.gamma_device(H, 7, c.dev)
    args_cache, odicts = {}, {}

    def args_for(T, dt, st):
        key = (int(T), int(dt), bool(st))
        if key not in args_cache:
            ts = [b[:T, :H] if st else b[:T].view(-1)[:T * H].view(T, H) for b in bufs[dt]]
            full = [ts[0], ts[1], gam, ts[2], ts[3]]
            args_cache[key] = S.make_args(S.OP_ADD_RMSNORM, full, eps=1e-6)
            odicts[key] = dict(op=1, tensors=[dict(addr=x.data_ptr(), dtype=S.BF16 if x.dtype == t.bfloat16 else
                                                   (S.FP16 if x.dtype == t.float16 else S.FP32),
                                                   shape=tuple(x.shape), stride=tuple(x.stride()),
                                                   device=c.dev.index or 0) for x in full],
                               eps=1e-6, theta=0.0, flags=0)
        return args_cache[key], odicts[key]

    generic = S.Scm(device=c.dev.index or 0)
    for dt in (S.BF16, S.FP16):
        generic.register(S.make_spec(S.OP_ADD_RMSNORM, dt, [H], 1, 1 << 40, layout=S.LAYOUT_ANY,
                                     align_bytes=2, variant=S.VARIANT_GENERIC))
    static_specs = []
    for b in range(8):
        lo, hi = G.bucket_range(b)
        for dt in (S.BF16, S.FP16):
            static_specs.append(dict(op=1, dtype=dt, rank=2, layout=0, fixed=(H,), tok_lo=lo, tok_hi=hi,
                                     align=16, device=c.dev.index or 0, variant=0, theta=0.0))
    results = {}
    for mode in ("static", "growth"):
        oracle_table = list(static_specs) if mode == "static" else []

        def hook(scm, args, stream):
            if mode == "static":
                st, _ = generic.invoke(args, stream)
                if st != S.OK:
                    raise RuntimeError("generic version failed")
                return None
            T = int(args.t[0].shape[0])
            lo, hi = G.bucket_range(G.bucket_of(T))
            lay = S.LAYOUT_CONTIG if args.t[0].stride[0] == H or T == 1 else S.LAYOUT_ROWSTRIDED
            idx = scm.register(S.make_spec(S.OP_ADD_RMSNORM, int(args.t[0].dtype), [H], lo, hi, layout=lay))
            st, sel = scm.invoke(args, stream)
            if st != S.OK:
                raise RuntimeError("re-invoke after growth missed")
            return idx

        scm = S.Scm(device=c.dev.index or 0, flags=S.OPT_TIMING, max_specs=64, hook=hook)
        if mode == "static":
            for sp in static_specs:
                scm.register(S.make_spec(1, sp["dtype"], [H], sp["tok_lo"], sp["tok_hi"]))
        memo = {}
        inv, sel = c.L.trident_scm_invoke, ctypes.c_int32(-1)
        mism = 0
        hits = misses = 0
        t.cuda.synchronize()
        h0 = time.perf_counter()
        for T, dt, st in zip(Ts, dts, strided):
            a, od = args_for(T, dt, st)
            rc = inv(scm.h, ctypes.byref(a), c.sp, ctypes.byref(sel))
            key = (len(oracle_table), int(T), int(dt), bool(st))
            if key not in memo:  # selection only: the buffers are distinct allocations
                memo[key] = G.select(oracle_table, od, check_overlap=False)
            ost, oidx = memo[key]
            if rc == S.OK:
                hits += 1
                mism += not (ost == G.OK and oidx == sel.value)
            elif rc == S.MISS_HANDLED:
                misses += 1
                mism += ost != G.MISS
                if mode == "growth":  # oracle replays the same growth rule
                    lo, hi = G.bucket_range(G.bucket_of(int(T)))
                    oracle_table.append(dict(op=1, dtype=int(dt), rank=2, layout=1 if (st and T > 1) else 0,
                                             fixed=(H,), tok_lo=lo, tok_hi=hi, align=16,
                                             device=c.dev.index or 0, variant=0, theta=0.0))
            else:
                raise RuntimeError(f"stress call failed: {rc} {S.trident_scm_last_error()} {scm.hook_error}")
        t.cuda.synchronize()
        wall = time.perf_counter() - h0
        _, ns = S.trident_scm_host_times(scm.h, 1 << 16)
        stt = scm.stats()
        c.launches += len(Ts) + (stt.hook_registered if mode == "growth" else 0)
        results[mode] = dict(calls=len(Ts), hits=hits, misses=misses, mismatches_vs_oracle=int(mism),
                             versions=stt.num_specs, host_ns_per_hit_median=float(np.median(ns)),
                             host_ns_per_hit_p99=float(np.percentile(ns, 99)),
                             python_us_per_call=round(wall * 1e6 / len(Ts), 3))
        scm.close()
    generic.close()
    return results


def bench_motivation(c, warmup=20, rounds=5, repeats=10):
    """The paper's motivation experiment (§2.3, Fig. 2) on this GPU: rms_norm of x (1024, 128)
    with weight (128,), warm path. Per call, host latency (until the Python call returns)
    and end-to-end latency (until the GPU finishes), after `warmup` calls, `rounds` x
    `repeats` samples, median -- for this library's SCM, torch eager F.rms_norm, and default
    torch.compile. Context only: torch is a comparison system here, not the oracle."""
    t, S, synth = c.torch, c.S, c.synth
    T, H = 1024, 128
    x = synth.act_device((T, H), S.BF16, 60, c.dev)
    w32 = synth.gamma_device(H, 61, c.dev)
    w16 = w32.to(t.bfloat16).float()  # the same weights, representable in bf16
    w32.copy_(w16)
    w_bf = w16.to(t.bfloat16)
    y = t.empty_like(x)
    scm = S.Scm(device=c.dev.index or 0)
    scm.register(S.make_spec(S.OP_RMSNORM, S.BF16, [H], 1, 4096))
    a = S.make_args(S.OP_RMSNORM, [x, w32, y], eps=1e-6)
    inv = c.invoker(scm)
    addr = ctypes.addressof(a)
    F = t.nn.functional

    def eager():
        return F.rms_norm(x, (H,), weight=w_bf, eps=1e-6)

    def ours():
        return inv(addr)

    def measure(fn):
        for _ in range(warmup):
            fn()
        t.cuda.synchronize()
        host, e2e = [], []
        for _ in range(rounds):
            for _ in range(repeats):
                t.cuda.synchronize()
                h0 = time.perf_counter()
                fn()
                h1 = time.perf_counter()
                t.cuda.synchronize()
                h2 = time.perf_counter()
                host.append((h1 - h0) * 1e6)
                e2e.append((h2 - h0) * 1e6)
        return float(np.median(host)), float(np.median(e2e))

    # the same call through the structured-argument entry: rms_norm(x, residual, weight, out,
    # eps) with two tree versions (residual None -> RMSNORM, a tensor -> ADD_RMSNORM); the
    # tree prebuilt once, and packed from the Python arguments on every call
    tscm = S.Scm(device=c.dev.index or 0)
    tscm.register_tree(S.make_spec(S.OP_RMSNORM, S.BF16, [H], 1, 4096),
                       S.Recipe(S.Slot(0), None, S.Slot(1), S.Slot(2), S.EPS))
    tscm.register_tree(S.make_spec(S.OP_ADD_RMSNORM, S.BF16, [H], 1, 4096),
                       S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)), S.EPS))
    tree = S.Tree(x, None, w32, y, 1e-6)
    th, sp = tscm.h.value, c.sp.value or 0
    if c.fc is not None:
        tinv = c.fc.invoke_tree
        t_addr = ctypes.addressof(tree.nodes)
        ours_tree = lambda: tinv(th, t_addr, tree.nargs, tree.nnodes, sp)

        def ours_tree_packed():
            tr = S.Tree(x, None, w32, y, 1e-6)
            return tinv(th, ctypes.addressof(tr.nodes), tr.nargs, tr.nnodes, sp)
        pinv = c.fc.invoke_py
        ours_tree_c = lambda: pinv(th, sp, x, None, w32, y, 1e-6)
    else:
        ours_tree = lambda: S.trident_scm_invoke_tree(tscm.h, tree, c.sp)
        ours_tree_packed = lambda: S.trident_scm_invoke_tree(tscm.h, S.Tree(x, None, w32, y, 1e-6), c.sp)
        ours_tree_c = None

    res = {}
    res["scm"] = dict(zip(("host_us", "e2e_us"), measure(ours)))
    assert_all_hit(scm, "motivation")
    c.launches += warmup + rounds * repeats
    res["scm_tree_prebuilt"] = dict(zip(("host_us", "e2e_us"), measure(ours_tree)))
    res["scm_tree_packed_python"] = dict(zip(("host_us", "e2e_us"), measure(ours_tree_packed)))
    n_tree = 2
    if ours_tree_c is not None:  # the arguments packed per call by the CPython shim
        res["scm_tree_packed_c"] = dict(zip(("host_us", "e2e_us"), measure(ours_tree_c)))
        n_tree += 1
    assert_all_hit(tscm, "motivation tree")
    c.launches += n_tree * (warmup + rounds * repeats)
    tscm.close()
    res["torch_eager"] = dict(zip(("host_us", "e2e_us"), measure(eager)))
    try:
        compiled = t.compile(eager)
        compiled()  # compile outside the timed samples
        res["torch_compile_default"] = dict(zip(("host_us", "e2e_us"), measure(compiled)))
    except Exception as e:  # context only
        res["torch_compile_default"] = dict(unavailable=str(e).splitlines()[0][:200])
    t.cuda.synchronize()
    agree = float((y.float() - eager().float()).abs().max())
    scm.close()
    base = res["torch_eager"]
    for k, v in res.items():
        if "host_us" in v:
            v["speedup_vs_eager_host"] = round(base["host_us"] / v["host_us"], 3)
            v["speedup_vs_eager_e2e"] = round(base["e2e_us"] / v["e2e_us"], 3)
            v["host_us"], v["e2e_us"] = round(v["host_us"], 3), round(v["e2e_us"], 3)
    res["max_abs_diff_scm_vs_eager"] = agree
    res["shape"] = "x (1024, 128) bf16, weight (128,), eps 1e-6"
    res["paper_h800_context"] = "Trident vs eager 1.18x host, 1.11x e2e; default torch.compile 0.39x host, 0.43x e2e (§2.3)"
    return res


def bench_kernels(c, n_calls=30):
    """The paper's kernel-benchmark method (§4.1) on this library's FlagGems-style operators
    (rms_norm, silu, add, neg, masked_fill), five shapes from LLM dimensions each: 30
    consecutive calls, the first reported as cold, the median of the rest as warm; host
    latency (until the call returns) and end-to-end latency (until the GPU finishes). The SCM
    writes into preallocated outputs; torch eager allocates its results (as the eager
    wrapper the paper compares against does). Per operator the arithmetic mean of the
    per-shape warm ratios eager / SCM, as the paper aggregates (§4.2)."""
    t, S, synth = c.torch, c.S, c.synth
    F = t.nn.functional
    shapes = [(1, 4096), (16, 4096), (128, 4096), (1024, 4096), (256, 14336)]
    ops = ["rms_norm", "silu", "add", "neg", "masked_fill"]
    out = {}

    def timed(fn, n):
        host, e2e = [], []
        for _ in range(n):
            t.cuda.synchronize()
            h0 = time.perf_counter()
            fn()
            h1 = time.perf_counter()
            t.cuda.synchronize()
            h2 = time.perf_counter()
            host.append((h1 - h0) * 1e6)
            e2e.append((h2 - h0) * 1e6)
        return dict(cold_host_us=round(host[0], 2), cold_e2e_us=round(e2e[0], 2),
                    warm_host_us=round(float(np.median(host[1:])), 3),
                    warm_e2e_us=round(float(np.median(e2e[1:])), 3))

    seed = 70
    for name in ops:
        rows = []
        for (T, W) in shapes:
            seed += 1
            x = synth.act_device((T, W), S.BF16, seed, c.dev)
            b = synth.act_device((T, W), S.BF16, seed + 1000, c.dev)
            mask = t.rand((T, W), device=c.dev) < 0.3
            y = t.empty_like(x)
            w32 = synth.gamma_device(W, seed + 2000, c.dev).to(t.bfloat16).float()
            w_bf = w32.to(t.bfloat16)
            op = {"rms_norm": S.OP_RMSNORM, "silu": S.OP_SILU, "add": S.OP_ADD, "neg": S.OP_NEG,
                  "masked_fill": S.OP_MASKED_FILL}[name]
            ts = {"rms_norm": [x, w32, y], "silu": [x, y], "add": [x, b, y], "neg": [x, y],
                  "masked_fill": [x, mask.view(t.uint8), y]}[name]
            eager = {"rms_norm": lambda: F.rms_norm(x, (W,), weight=w_bf, eps=1e-6),
                     "silu": lambda: F.silu(x), "add": lambda: t.add(x, b), "neg": lambda: t.neg(x),
                     "masked_fill": lambda: x.masked_fill(mask, -1e4)}[name]
            r0 = time.perf_counter()
            scm = S.Scm(device=c.dev.index or 0)
            scm.register(S.make_spec(op, S.BF16, [W], 1, 1 << 20))
            reg_us = (time.perf_counter() - r0) * 1e6
            a = S.make_args(op, ts, eps=1e-6, scalar=-1e4)
            inv, addr = c.invoker(scm), ctypes.addressof(a)
            ours = timed(lambda: inv(addr), n_calls)
            assert_all_hit(scm, name)
            c.launches += n_calls
            diff = float((y.float() - eager().float()).abs().max())
            ref = timed(eager, n_calls)
            scm.close()
            rows.append(dict(shape=[T, W], scm=ours, scm_register_us=round(reg_us, 1), torch_eager=ref,
                             speedup_host=round(ref["warm_host_us"] / ours["warm_host_us"], 3),
                             speedup_e2e=round(ref["warm_e2e_us"] / ours["warm_e2e_us"], 3),
                             max_abs_diff_vs_eager=diff))
        out[name] = dict(shapes=rows,
                         mean_speedup_host=round(float(np.mean([r["speedup_host"] for r in rows])), 3),
                         mean_speedup_e2e=round(float(np.mean([r["speedup_e2e"] for r in rows])), 3))
    out["paper_h800_context"] = ("21 FlagGems ops, Trident vs eager: mean 1.10x host, 1.07x e2e; silu 1.74x host, "
                                 "1.73x e2e; masked_fill 1.67x e2e (§4.2)")
    return out


def bench_sweep(c, reps=20, quick=False, tokens=None):
    """HBM bandwidth sweep: add+RMSNorm (H 8192) and SwiGLU (I 28672) at T = 2^0..2^15,
    bf16. Each size: `reps` back-to-back launches from one native call, rotating across
    row windows of arenas sized for 32768 tokens so no launch reads what the previous
    left in L2 (for T >= 512 the buffers alone exceed L2). With `tokens`, only those sizes,
    on arenas of two windows of the largest (for profiling a few GB at most)."""
    t, S, synth = c.torch, c.S, c.synth
    H, I, Tmax = 8192, 28672, 32768
    if tokens:
        Tmax = 2 * max(tokens)
    peak, _ = measured_peaks()
    s = S.Scm(device=c.dev.index or 0)
    s.register(S.make_spec(S.OP_ADD_RMSNORM, S.BF16, [H], 1, 1 << 20))
    s.register(S.make_spec(S.OP_SWIGLU, S.BF16, [I], 1, 1 << 20))
    out = {"add_rmsnorm": [], "swiglu": []}
    seq = c.L.trident_scm_invoke_seq
    Ts = list(tokens) if tokens else ([2 ** k for k in range(16)] if not quick else [1, 64, 4096, 32768])
    # add + RMSNorm
    x = synth.act_device((Tmax, H), S.BF16, 11, c.dev)
    r = synth.act_device((Tmax, H), S.BF16, 12, c.dev)
    gam = synth.gamma_device(H, 13, c.dev)
    y, ro = t.empty_like(x), t.empty_like(r)
    for T in Ts:
        nwin = Tmax // T
        arr = (S.trident_args * reps)(*[S.make_args(S.OP_ADD_RMSNORM, [
            x[(i % nwin) * T:(i % nwin + 1) * T], r[(i % nwin) * T:(i % nwin + 1) * T], gam,
            y[(i % nwin) * T:(i % nwin + 1) * T], ro[(i % nwin) * T:(i % nwin + 1) * T]], eps=1e-6)
            for i in range(reps)])
        us, _ = time_steps(c, lambda i: seq(s.h, arr, reps, c.sp, None), 3, 2)
        us /= reps
        c.launches += 5 * reps
        b = 8 * H * T + 4 * H
        out["add_rmsnorm"].append(dict(T=T, us=round(us, 3), gbs=round(b / us / 1e3, 1),
                                       frac_measured=round(b / us / 1e3 / peak, 3),
                                       frac_8tbs=round(b / us / 1e3 / NOMINAL_HBM_GBS, 3)))
    del x, r, y, ro
    g = synth.act_device((Tmax, I), S.BF16, 14, c.dev)
    u = synth.act_device((Tmax, I), S.BF16, 15, c.dev)
    o = t.empty_like(g)
    for T in Ts:
        nwin = Tmax // T
        arr = (S.trident_args * reps)(*[S.make_args(S.OP_SWIGLU, [
            g[(i % nwin) * T:(i % nwin + 1) * T], u[(i % nwin) * T:(i % nwin + 1) * T],
            o[(i % nwin) * T:(i % nwin + 1) * T]]) for i in range(reps)])
        us, _ = time_steps(c, lambda i: seq(s.h, arr, reps, c.sp, None), 3, 2)
        us /= reps
        c.launches += 5 * reps
        b = 6 * I * T
        out["swiglu"].append(dict(T=T, us=round(us, 3), gbs=round(b / us / 1e3, 1),
                                  frac_measured=round(b / us / 1e3 / peak, 3),
                                  frac_8tbs=round(b / us / 1e3 / NOMINAL_HBM_GBS, 3)))
    del g, u, o
    assert_all_hit(s, "sweep")
    s.close()
    out["rope_kv"] = sweep_rope_kv(c, Ts, reps, peak)
    big = [e for e in out["add_rmsnorm"] + out["swiglu"] if e["T"] >= 4096]
    out["min_frac_measured_T_ge_4096"] = min(e["frac_measured"] for e in big) if big else None
    return out


def sweep_rope_kv(c, Ts, reps, peak):
    """RoPE + KV append (the single-op kernel) at the Llama layer's shapes (32 / 8 heads, D 128,
    a cache of 8192 slots, q/k/v rows of one packed qkv row), T <= 8192 tokens of distinct
    uniform positions. The `reps` launches take consecutive T-token windows of a qkv arena of
    max(32768, 2 T) tokens; the two caches (16 MB each) are shared by all launches."""
    t, S, synth = c.torch, c.S, c.synth
    cfg = synth.LLAMA
    Hq, Hkv, D, Sc = cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"]
    Ts = [T for T in Ts if T <= Sc]
    if not Ts:
        return []
    W = (Hq + 2 * Hkv) * D
    Tmax = max(32768, 2 * max(Ts))
    s = S.Scm(device=c.dev.index or 0)
    for lay in (S.LAYOUT_ROWSTRIDED, S.LAYOUT_CONTIG):  # a one-token window is also contiguous
        s.register(S.make_spec(S.OP_ROPE_KV, S.BF16, [Hq, Hkv, D, Sc], 1, 1 << 20, layout=lay,
                               rope_theta=cfg["theta"]))
    qkv = synth.act_device((Tmax, W), S.BF16, 16, c.dev)
    g = np.random.default_rng(17)
    kc = t.zeros((Hkv, Sc, D), dtype=t.bfloat16, device=c.dev)
    vc = t.zeros((Hkv, Sc, D), dtype=t.bfloat16, device=c.dev)
    seq = c.L.trident_scm_invoke_seq
    out = []
    for T in Ts:
        nwin = Tmax // T
        pos = t.from_numpy(np.stack([synth.positions(g, T, Sc) for _ in range(reps)])).to(c.dev)

        def args(i):
            w = qkv[(i % nwin) * T:(i % nwin + 1) * T]
            q = w[:, :Hq * D].view(T, Hq, D)
            k = w[:, Hq * D:(Hq + Hkv) * D].view(T, Hkv, D)
            v = w[:, (Hq + Hkv) * D:].view(T, Hkv, D)
            return S.make_args(S.OP_ROPE_KV, [q, k, v, pos[i], kc, vc],
                               rope_theta=cfg["theta"])
        arr = (S.trident_args * reps)(*[args(i) for i in range(reps)])
        us, _ = time_steps(c, lambda i: seq(s.h, arr, reps, c.sp, None), 3, 2)
        us /= reps
        c.launches += 5 * reps
        b = ((2 * Hq + 4 * Hkv) * D * 2 + 4) * T + D * 4
        out.append(dict(T=T, us=round(us, 3), gbs=round(b / us / 1e3, 1),
                        frac_measured=round(b / us / 1e3 / peak, 3),
                        frac_8tbs=round(b / us / 1e3 / NOMINAL_HBM_GBS, 3)))
    assert_all_hit(s, "rope sweep")
    s.close()
    del qkv, kc, vc
    return out


def bench_chain_large(c, reps=10):
    """The fused layer chain where it is bandwidth-bound: Llama- and Qwen3-style layers at
    4096 and 8192 tokens (the KV cache's 8192 slots bound T), one launch per call, `reps`
    calls back to back, each moving far more than the L2 (0.7-1.4 GB), against the measured
    copy bandwidth. Token counts of several waves: one norm CTA per token, three head-rows per
    RoPE lane group."""
    S = c.S
    peak, _ = measured_peaks()
    out = []
    for name, cfg in (("llama", c.synth.LLAMA), ("qwen3", c.synth.QWEN3)):
        qk = cfg.get("qknorm", False)
        fixed = [cfg[k] for k in ("H", "Hq", "Hkv", "D", "S", "I")]
        op = S.OP_LAYER_CHAIN_QKNORM if qk else S.OP_LAYER_CHAIN
        scm = S.Scm(device=c.dev.index or 0, flags=S.OPT_PDL)
        scm.register(S.make_spec(op, S.BF16, fixed, 1, 1 << 20, layout=S.LAYOUT_ROWSTRIDED,
                                 rope_theta=cfg["theta"]))
        inv = c.invoker(scm)
        for T in ((4096, 8192) if name == "llama" else (4096,)):
            sets = ChainSets(c, cfg, T, min_bytes=2 * L2_BYTES, max_sets=2)
            args = [sets.fused_args(c, i) for i in range(sets.R)]
            addrs = [ctypes.addressof(a) for a in args]
            us, _ = time_steps(c, lambda i: inv(addrs[i % len(addrs)]), reps, 3)
            c.launches += reps + 3
            b = chain_bytes_per_launch(cfg, T)
            out.append(dict(layer=name, T=T, us=round(us, 3), gbs=round(b / us / 1e3, 1),
                            frac_measured=round(b / us / 1e3 / peak, 3), bytes_per_launch=int(b)))
            del args, addrs, sets
        assert_all_hit(scm, "chain large")
        scm.close()
    return out


def kernel_duration_chain(c, cfg, T, calls=40):
    """Average duration of the fused chain kernel: one launch per rotating input set, issued
    back to back by one native call (device-bound), `calls` such calls timed with CUDA events
    on the launching stream after a lead kernel (so the window holds about a thousand launches
    of a busy device, not the first launch of an idle one)."""
    S = c.S
    sets = ChainSets(c, cfg, T)
    scm = layer_scm(c, cfg)
    n = sets.R
    arr = (S.trident_args * n)(*[sets.fused_args(c, i) for i in range(n)])
    us, _ = time_steps(c, lambda i: c.L.trident_scm_invoke_seq(scm.h, arr, n, c.sp, None), calls, 3,
                       lead_cycles=HEADLINE_LEAD_CYCLES)
    assert_all_hit(scm, "roofline kernel")
    c.launches += (calls + 3) * n
    scm.close()
    return us / n


def copy_floor(c, cfg, T, blocks_list=(152, 304, 456, 512, 576, 608, 640, 760, 912, 1216), calls=40):
    """The copy floor for the chain's traffic: a plain streaming kernel that reads and writes
    the same byte counts as one fused-chain launch at T tokens (the read sum XORed per thread,
    the write a store of it), launched the same way -- PDL with an L2 prefetch before the
    wait, one launch per rotating input set, `calls` native calls of `sets` launches after a
    lead kernel. Gives, per grid size, the per-launch time the GPU needs for this traffic
    with no arithmetic, no gathers and no role mix."""
    torch, S = c.torch, c.S
    rb, wb = chain_read_write_bytes(cfg, T)
    rb, wb = (rb + 15) // 16 * 16, (wb + 15) // 16 * 16
    sets = max(2, -(-2 * L2_BYTES // (rb + wb)))
    src = torch.randint(-2 ** 31, 2 ** 31 - 1, (sets * rb // 4,), dtype=torch.int32, device=c.dev)
    dst = torch.empty((sets * wb // 4,), dtype=torch.int32, device=c.dev)
    scm = S.Scm(device=c.dev.index or 0, flags=S.OPT_PDL)
    out = dict(read_bytes=int(rb), write_bytes=int(wb), sets=int(sets), launches_per_call=int(sets), grids={})
    for blocks in blocks_list:
        def call(i, blocks=blocks):
            st = S.trident_copy_floor(scm.h, c.sp, src.data_ptr(), dst.data_ptr(), rb, wb, blocks, sets, sets)
            assert st == S.OK, S.trident_scm_last_error()
        us, _ = time_steps(c, call, calls, 3, lead_cycles=HEADLINE_LEAD_CYCLES)
        c.launches += (calls + 3) * sets
        out["grids"][str(blocks)] = round(us / sets, 3)
    scm.close()
    del src, dst
    return out


_T0 = time.perf_counter()


def progress(msg):
    print("[bench %7.1fs] %s" % (time.perf_counter() - _T0, msg), file=sys.stderr, flush=True)


def run_ours(a):
    import torch
    import torch.distributed as dist
    from paper_2609_37241_gb300 import synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    c = Ctx(torch.device("cuda", local))
    K, W = a.steps, a.warmup
    clocks = ClockSampler(local)
    cfg = synth.LLAMA

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    # ---- headline: T = 64, fused, one invoke per step; exactly K timed steps
    sets = ChainSets(c, cfg, HEADLINE_T)
    scm = layer_scm(c, cfg)
    R = sets.R
    fused_structs = [sets.fused_args(c, i) for i in range(R)]
    fused = [ctypes.addressof(x) for x in fused_structs]
    inv = c.invoker(scm)
    # W warm-up steps, and at least one visit of every rotating input set, so that no timed
    # step is the first touch of its buffers (the rotation only keeps the working set above
    # the L2; a decode loop reuses its buffers every step)
    W_run = max(W, R)
    for i in range(W_run):
        inv(fused[i % R])
    barrier()
    e0, e1 = c.events()
    # A short sleep kernel and the last HEADLINE_LEAD_STEPS untimed warm-up steps ahead of
    # e0 keep the device busy while the host issues the first timed steps, so the window
    # measures the steady stream of steps (as a decode loop runs) rather than the idle
    # device's first launch latency; both are outside the window, which opens when the
    # last of them has finished.
    torch.cuda._sleep(HEADLINE_LEAD_CYCLES)
    for i in range(HEADLINE_LEAD_STEPS):
        inv(fused[(W_run + i) % R])
    W_run += HEADLINE_LEAD_STEPS
    e0.record(c.stream)
    for i in range(K):
        inv(fused[(W_run + i) % R])
    e1.record(c.stream)
    barrier()
    ms = e0.elapsed_time(e1)
    headline_launches = assert_all_hit(scm, "headline") - W_run
    c.launches += W_run + K
    scm.close()
    del sets
    ms_max = max_over_ranks(ms, world, device=c.dev)
    us_step = ms_max * 1e3 / K

    extra = {}
    want = (lambda name: True) if a.sections == "all" else (lambda name: name in a.sections.split(","))
    toks_arg = [int(x) for x in a.tokens.split(",")] if a.tokens else None
    floor_us = None
    if rank == 0 and (want("floor") or want("layers") or want("qwen3")):
        progress("launch floor")
        extra["latency_floor"] = bench_launch_floor(c)
        floor_us = extra["latency_floor"]["pdl"]["device_us"]
    if rank == 0 and want("layers"):
        progress("per-token layer steps")
        per_t = {}
        for T in toks_arg or (1, 4, 16, 64):
            per_t[str(T)], _ = bench_layer(c, cfg, T, K=max(500, min(K, 2000)), W=W)
        add_floor_fractions(per_t, floor_us)
        extra["llama_per_tokens"] = per_t
    if rank == 0 and want("qwen3"):
        progress("qwen3 36-layer steps")
        qw = {}
        toks = toks_arg or (
            (1, 8, 32, 128) if not a.quick else (1, 128))
        for T in toks:
            qw[str(T)], _ = bench_layer(c, synth.QWEN3, T, K=max(56, min(K, 2000) // 36), W=W,
                                        layers=synth.QWEN3["layers"])
        add_floor_fractions(qw, floor_us)
        peak, _ = measured_peaks()
        for T, v in qw.items():  # the steps that are device-bound: HBM fraction of the whole step
            o = v.get("one_launch_step")
            if o:
                b = synth.QWEN3["layers"] * chain_bytes_per_launch(synth.QWEN3, int(T))
                o["bytes_per_step"] = int(b)
                o["hbm_frac"] = round(b / o["us"] / 1e3 / peak, 3)
                if "replayed" in o:
                    o["replayed"]["hbm_frac"] = round(b / o["replayed"]["us"] / 1e3 / peak, 3)
        extra["qwen3_36layer_step"] = qw
    if rank == 0 and want("host"):
        progress("host dispatch")
        extra["host_dispatch_single_addnorm"] = bench_host_hit(c)
    if rank == 0 and want("stress"):
        progress("guard stress")
        extra["guard_stress"] = bench_guard_stress(c, n_calls=20000 if a.quick else None)
    if rank == 0 and want("motivation"):
        progress("motivation microbenchmark")
        extra["motivation_rms_norm"] = bench_motivation(c)
    if rank == 0 and want("kernels"):
        progress("kernel benchmark (paper method)")
        extra["kernel_benchmark"] = bench_kernels(c)
    if rank == 0 and want("sweep"):
        progress("hbm sweep")
        extra["hbm_sweep"] = bench_sweep(c, quick=a.quick, tokens=toks_arg)
        if not a.quick and not toks_arg:
            extra["hbm_sweep"]["layer_chain"] = bench_chain_large(c)
    if rank == 0 and want("roofline"):
        progress("roofline kernel")
        kd = kernel_duration_chain(c, cfg, HEADLINE_T)
        peak, src = measured_peaks()
        b = chain_bytes_per_launch(cfg, HEADLINE_T)
        tr = chain_traffic()
        extra["roofline"] = dict(bound="hbm", achieved=round(b / kd / 1e3, 1), peak=peak, unit="GB/s",
                                 frac=round(b / kd / 1e3 / peak, 3),
                                 traffic=None if tr is None else tr[0] + tr[1],
                                 traffic_read=None if tr is None else tr[0],
                                 traffic_write=None if tr is None else tr[1],
                                 kernel="chain_kernel<bf16,H4096,D128>",
                                 bytes_per_launch=int(b), us_per_launch=round(kd, 3), peak_source=src)
        progress("copy floor")
        cf = copy_floor(c, cfg, HEADLINE_T)
        best = min(cf["grids"].values())
        cf.update(frac_of_peak={k: round((cf["read_bytes"] + cf["write_bytes"]) / v / 1e3 / peak, 3)
                                for k, v in cf["grids"].items()},
                  chain_over_best_copy=round(best / kd, 3))
        extra["roofline"]["copy_floor"] = cf
    if rank == 0 and want("e2e"):
        progress("e2e")
        extra["e2e"] = bench_e2e(c, cfg, HEADLINE_T, K=min(K, 500), W=W)
    ck = clocks.stop()
    if rank == 0:
        cpu_us = n = None
        cpu_all = None
        if want("cpu"):
            progress("cpu baseline")
            budget = 3.0 if a.quick else 12.0
            cpu_us, n = oracle_layer_step_us(cfg, HEADLINE_T, budget)
            from oracle import layer as L  # the same oracle, OpenMP build, all host cores
            L.set_parallel(True)
            try:
                us_all, n_all = oracle_layer_step_us(cfg, HEADLINE_T, budget)
                cpu_all = dict(value=round(us_all, 1), unit=UNIT, cores=L.threads(), kind="oracle",
                               nproc=os.cpu_count(),
                               sample="%d layer steps at 64 tokens (%.1f s), token loops shared "
                                      "over the host cores (OpenMP)" % (n_all, us_all * n_all / 1e6))
            finally:
                L.set_parallel(False)
        line = dict(metric=METRIC, value=round(us_step, 3), unit=UNIT, n_gpus=world, steps=K, warmup=W,
                    ms_per_step=round(us_step / 1e3, 6), higher_is_better=False, scaling="weak",
                    vs_baseline=None, dtype="bf16",
                    data="synthetic (seeded N(0,1) activations, N(1,0.1) norm weights, distinct "
                         "uniform positions; no model weights)",
                    config=dict(workload="llama decode layer non-GEMM chain: 64 tokens, H 4096, 32/8 "
                                         "heads, D 128, I 14336, theta 5e5, KV cache [8,8192,128]",
                                tokens=HEADLINE_T, path="fused chain, 1 launch per step, PDL",
                                l2="inputs rotated over %d sets (%.0f MB > 2x L2)" % (
                                    R, R * chain_bytes_per_token(cfg) * HEADLINE_T / 2 ** 20),
                                parallelism="replicas" if world > 1 else "single GPU"),
                    timing=dict(lead="a 24 us sleep kernel and %d untimed warm-up steps queued "
                                     "behind it ahead of the first timed step keep the device busy "
                                     "while the host issues the first steps (outside the timed "
                                     "window, which opens when they have finished)" % HEADLINE_LEAD_STEPS,
                                warmup_steps_run=W_run,
                                warmup_note="max(W, sets) + %d: every rotating set is visited once "
                                            "before timing" % HEADLINE_LEAD_STEPS),
                    gpu_launches=headline_launches, gpu_launches_whole_run=c.launches,
                    python_binding="fastcall" if c.fc is not None else "ctypes")
        line.update(extra)
        if cpu_us is not None:
            line["cpu_baseline"] = dict(value=round(cpu_us, 1), unit=UNIT, cores=1, kind="oracle",
                                        sample="%d layer steps at 64 tokens (%.1f s)" % (n, cpu_us * n / 1e6))
        if cpu_all is not None:
            line["cpu_baseline_all_cores"] = cpu_all
        if ck:
            line["clocks"] = ck
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def run_reference(a):
    """Reference arm: the CPU oracle, as it stands, on the headline configuration. Each
    step runs the whole layer chain on a sample of the 64 tokens (all four steps, every
    head), sized so that warm-up plus steps take about a minute; the time is scaled to
    64 tokens (the chain's work is proportional to the token count)."""
    from paper_2609_37241_gb300 import synth
    from oracle import layer as L
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cfg = synth.LLAMA
    g = np.random.default_rng(0)
    full = synth.layer_inputs(g, HEADLINE_T, cfg)

    def sample(Ts):
        d = {k: (v[:Ts] if k in ("h", "r0", "q", "k", "v", "pos", "attn_out", "g", "u") else v)
             for k, v in full.items()}
        return d

    one = sample(1)
    t0 = time.perf_counter()
    L.layer_chain(one, cfg["theta"], cfg["eps"], synth.BF16)
    t1 = max(time.perf_counter() - t0, 1e-4)
    budget = 20.0 if a.quick else 60.0
    Ts = int(max(1, min(HEADLINE_T, budget / ((a.steps + a.warmup) * t1))))
    inp = sample(Ts)
    for _ in range(a.warmup):
        L.layer_chain(inp, cfg["theta"], cfg["eps"], synth.BF16)
    samples = []
    for _ in range(a.steps):
        t0 = time.perf_counter()
        L.layer_chain(inp, cfg["theta"], cfg["eps"], synth.BF16)
        samples.append((time.perf_counter() - t0) * 1e6 * HEADLINE_T / Ts)
    us = float(np.median(samples))
    line = dict(metric=METRIC, value=round(us, 1), unit=UNIT, n_gpus=world, steps=a.steps,
                warmup=a.warmup, ms_per_step=round(us / 1e3, 4), higher_is_better=False,
                scaling="weak", vs_baseline=None, dtype="f64", data="synthetic", impl="reference",
                config=dict(workload="llama decode layer non-GEMM chain: 64 tokens, H 4096, 32/8 heads, "
                                     "D 128, I 14336, theta 5e5, KV cache [8,8192,128]", tokens=HEADLINE_T,
                            path="CPU oracle (plain C, fp64 arithmetic): the whole chain per step on a "
                                 "sample of the tokens",
                            l2="host CPU arm: no GPU cache to flush",
                            parallelism="single process (rank 0)"),
                cpu_baseline=dict(value=round(us, 1), unit=UNIT, cores=1, kind="oracle",
                                  sample="each step: the layer chain on %d of the 64 tokens, scaled "
                                         "to 64 (median of %d steps)" % (Ts, a.steps)),
                e2e=dict(value=round(us, 1), unit=UNIT, h2d_bytes_per_step=0, d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)


def main():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5000)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--quick", action="store_true", help="smaller sections (for smoke runs)")
    p.add_argument("--tokens", default="", help="comma list of token counts for the layers, qwen3 and sweep sections")
    p.add_argument("--sections", default="all",
                   help="comma list of: floor,layers,qwen3,host,stress,motivation,kernels,sweep,roofline,e2e,cpu"
                        " (default all;"
                        " the headline always runs)")
    a = p.parse_args()
    if a.warmup < 3:
        a.warmup = 3
    if a.impl == "reference":
        run_reference(a)
    else:
        run_ours(a)


if __name__ == "__main__":
    main()
