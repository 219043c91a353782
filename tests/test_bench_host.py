"""Host-side pieces of bench.py that the roofline line rests on (no GPU).

The algorithmic bytes of the fused layer chain are counted here by hand from what one token
moves through the chain (both norms, RoPE with the KV append, SwiGLU), and the committed ncu
DRAM counters are checked against those bytes while they belong to the current sources.
"""
import json
import os

import pytest

import bench
from paper_2609_37241_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def hand_bytes_per_token(H, Hq, Hkv, D, I):
    """Bytes one token moves through the fused chain, bf16 activations.

    first add+RMSNorm: read h and r0, write x1 and r1 (4 rows of H);
    second add+RMSNorm: read attn_out, write x2 and r2 (r1 stays on chip: 3 rows of H);
    RoPE + KV append: read and write q (Hq heads), k and v (Hkv heads each, written into the
    caches), read one int32 position; SwiGLU: read gate and up, write the output (3 rows of I).
    """
    norms = (4 + 3) * H * 2
    rope = 2 * (Hq + Hkv + Hkv) * D * 2 + 4
    swiglu = 3 * I * 2
    return norms + rope + swiglu


@pytest.mark.parametrize("cfg", [synth.LLAMA, synth.QWEN3], ids=["llama", "qwen3"])
def test_chain_bytes_per_token_by_hand(cfg):
    want = hand_bytes_per_token(cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["I"])
    assert bench.chain_bytes_per_token(cfg) == want


def test_llama_bytes_per_token_is_the_stated_figure():
    assert bench.chain_bytes_per_token(synth.LLAMA) == 167_940
    assert bench.chain_bytes_per_launch(synth.LLAMA, 64) == 10_781_440


@pytest.mark.parametrize("cfg", [synth.LLAMA, synth.QWEN3], ids=["llama", "qwen3"])
@pytest.mark.parametrize("T", [1, 4, 16, 64, 4096])
def test_read_write_split_adds_up(cfg, T):
    r, w = bench.chain_read_write_bytes(cfg, T)
    assert r + w == bench.chain_bytes_per_launch(cfg, T)
    # every output row is written once: x1, r1, x2, r2, the rotated q/k, k/v cache rows, SwiGLU
    H, Hq, Hkv, D, I = (cfg[k] for k in ("H", "Hq", "Hkv", "D", "I"))
    assert w == T * (4 * H + (Hq + 2 * Hkv) * D + I) * 2


def test_unfused_chain_rereads_r1():
    cfg = synth.LLAMA
    assert bench.chain_bytes_per_token(cfg, fused=False) - bench.chain_bytes_per_token(cfg) == 2 * cfg["H"]


def test_committed_dram_counters_match_the_algorithmic_bytes():
    """The ncu counters bench.py reports as roofline.traffic: read and written bytes per launch
    of the 64-token Llama chain. While they belong to the current chain sources, each part is
    within 10 % of its algorithmic count (no re-reads, no lost writes)."""
    with open(os.path.join(ROOT, bench.CHAIN_COUNTERS)) as fh:
        d = json.load(fh)
    r_alg, w_alg = bench.chain_read_write_bytes(synth.LLAMA, 64)
    assert d["algorithmic_bytes_read_per_launch"] == r_alg
    assert d["algorithmic_bytes_write_per_launch"] == w_alg
    got = bench.chain_traffic()
    if got is None:
        assert d["source_sha256"] != bench.chain_sources_sha256()
        pytest.skip("chain sources changed since the counters were taken")
    rd, wr = got
    assert abs(rd - r_alg) <= 0.1 * r_alg and abs(wr - w_alg) <= 0.1 * w_alg


def _run_reference(env_extra):
    import subprocess
    import sys
    env = dict(os.environ, **env_extra)
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                           "--steps", "3", "--warmup", "3", "--quick"],
                          capture_output=True, text=True, env=env, cwd=ROOT, timeout=600)


def test_reference_arm_prints_one_line_on_the_headline_workload(built_lib):
    """The reference arm (the CPU oracle, as it stands) prints exactly one JSON line with the
    GPU arm's metric, unit and direction, the headline workload, and its CPU-baseline and
    end-to-end objects; under a multi-rank launch only rank 0 prints."""
    r = _run_reference({"RANK": "0", "WORLD_SIZE": "1"})
    assert r.returncode == 0, r.stderr
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["higher_is_better"] is False and d["steps"] == 3 and d["warmup"] == 3
    assert set(d["config"]) == {"workload", "tokens", "path", "l2", "parallelism"}
    assert d["config"]["tokens"] == bench.HEADLINE_T
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"] > 0
    assert d["e2e"] == dict(value=d["value"], unit=d["unit"], h2d_bytes_per_step=0, d2h_bytes_per_step=0)
    r1 = _run_reference({"RANK": "1", "WORLD_SIZE": "2"})
    assert r1.returncode == 0 and not [ln for ln in r1.stdout.splitlines() if ln.startswith("{")]
