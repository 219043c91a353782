"""trident_scm_invoke_step on the host (dry-run SCM, no GPU): which chunks run as one
launch, against the oracle's per-call selection and its brute-force independence test,
and the sequential contract (misses, errors, NOT_RUN) when a chunk cannot be fused."""
import random

import pytest

from oracle import guards as G
from tests import cases

NOT_RUN = -2
LLAMA_SMALL = dict(H=4096, Hq=2, Hkv=1, D=128, S=4, I=64)
ACT_SLOTS = (0, 1, 3, 4, 11, 13, 14)  # h, r0, x1, r1, attn_out, x2, r2: [T, H] each


@pytest.fixture()
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def chain_call(k, T=1, dtype="bf16", op=5, theta=5e5):
    """Chain call number k: its own buffers, 2^40 bytes away from call k+1's."""
    d = dict(op=op, T=T, dtype=dtype, theta=theta, **LLAMA_SMALL)
    a = cases.make_chain_args(d)
    for t in a["tensors"]:
        t["addr"] += k << 40
    return a


def chain_spec(dtype="bf16", op=5, tok=(1, 64), theta=5e5):
    fx = LLAMA_SMALL
    return cases.make_spec(dict(op=op, dtype=dtype, tok=list(tok), theta=theta,
                                fixed=[fx["H"], fx["Hq"], fx["Hkv"], fx["D"], fx["S"], fx["I"]]))


def run_step(S, table, calls, flags=0, hook=None):
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN | flags, hook=hook)
    for sp in table:
        s.register(cases.lib_spec(sp))
    arr = (S.trident_args * len(calls))(*[cases.lib_args(c) for c in calls])
    st, sel = s.invoke_step(arr)
    stats = s.stats()
    s.close()
    return st, sel, stats


def test_independent_chains_share_one_launch(S):
    table = [chain_spec()]
    calls = [chain_call(k) for k in range(3)]
    assert G.calls_independent(calls)
    st, sel, stats = run_step(S, table, calls)
    assert (st, sel) == (S.OK, [0, 0, 0])
    assert (stats.fused_launches, stats.fused_calls) == (1, 3)
    assert (stats.invokes, stats.hits, stats.misses) == (3, 3, 0)


def test_dependent_chains_run_in_order(S):
    # call 1's residual input is call 0's second residual output (the decoder's residual
    # stream): the calls must run one after the other
    table = [chain_spec()]
    calls = [chain_call(k) for k in range(3)]
    calls[1]["tensors"][1] = dict(calls[0]["tensors"][14])
    assert not G.calls_independent(calls)
    st, sel, stats = run_step(S, table, calls)
    assert (st, sel) == (S.OK, [0, 0, 0])
    assert (stats.fused_launches, stats.fused_calls, stats.hits) == (0, 0, 3)


def test_shared_inputs_do_not_prevent_fusion(S):
    # every layer reading the same positions and the same gamma is still independent
    table = [chain_spec()]
    calls = [chain_call(k) for k in range(4)]
    for c in calls[1:]:
        for slot in (2, 8, 12):  # gamma_attn, pos, gamma_mlp
            c["tensors"][slot] = dict(calls[0]["tensors"][slot])
    assert G.calls_independent(calls)
    st, sel, stats = run_step(S, table, calls)
    assert st == S.OK and stats.fused_launches == 1 and stats.fused_calls == 4


@pytest.mark.parametrize("seed", range(24))
def test_random_aliasing_matches_oracle(S, seed):
    """Random cross-call and in-call aliasing of the [T, H] slots (whole tensors or
    views shifted by a row fragment); the library's fuse decision and statuses are the
    oracle's."""
    rng = random.Random(seed)
    table = [chain_spec()]
    m = rng.choice((2, 3))
    calls = [chain_call(k) for k in range(m)]
    for _ in range(rng.choice((0, 1, 1, 2))):
        i, j = rng.randrange(m), rng.randrange(m)
        si, sj = rng.choice(ACT_SLOTS), rng.choice(ACT_SLOTS)
        if (i, si) == (j, sj):
            continue
        src = dict(calls[j]["tensors"][sj])
        if rng.random() < 0.3:  # a view shifted by 64 elements (still 16-byte aligned)
            src["addr"] += 128
        calls[i]["tensors"][si] = src
    want = [G.select(table, c) for c in calls]
    st, sel, stats = run_step(S, table, calls)
    if all(w == (G.OK, 0) for w in want):
        fused = G.calls_independent(calls)
        assert (st, sel) == (S.OK, [0] * m)
        assert stats.fused_launches == (1 if fused else 0)
    else:
        k = next(i for i, w in enumerate(want) if w != (G.OK, 0))
        assert want[k][0] == G.INVALID  # aliasing can only break a launch precondition
        assert st == S.ERR_INVALID
        assert sel == [0] * k + [-1] + [NOT_RUN] * (m - k - 1)
        assert stats.fused_launches == 0 and stats.hits == k


def test_miss_stops_the_step_at_its_position(S):
    table = [chain_spec(tok=(1, 1))]
    calls = [chain_call(0), chain_call(1, T=2), chain_call(2)]
    st, sel, stats = run_step(S, table, calls)
    assert (st, sel) == (S.MISS, [0, -1, NOT_RUN])
    assert (stats.fused_launches, stats.hits, stats.misses) == (0, 1, 1)


def test_hook_handles_a_miss_inside_a_step(S):
    table = [chain_spec(tok=(1, 1))]

    def hook(scm, args, stream):
        idx = scm.register(cases.lib_spec(chain_spec(tok=(2, 2))))
        assert scm.invoke(args, stream)[0] == S.OK
        return idx

    calls = [chain_call(0), chain_call(1, T=2), chain_call(2)]
    st, sel, stats = run_step(S, table, calls, hook=hook)
    assert (st, sel) == (S.MISS_HANDLED, [0, 1, 0])
    assert stats.fused_launches == 0 and stats.hook_calls == 1


def test_different_kernels_are_not_fused(S):
    table = [chain_spec("bf16"), chain_spec("fp16"), chain_spec("bf16", op=6)]
    calls = [chain_call(0, dtype="bf16"), chain_call(1, dtype="fp16")]
    st, sel, stats = run_step(S, table, calls)
    assert (st, sel, stats.fused_launches) == (S.OK, [0, 1], 0)
    q = [chain_call(0, op=6), chain_call(1)]
    st, sel, stats = run_step(S, table, q)
    assert (st, sel, stats.fused_launches) == (S.OK, [2, 0], 0)


def test_theta_may_differ_between_fused_calls(S):
    table = [chain_spec(theta=5e5), chain_spec(theta=1e6)]
    calls = [chain_call(0, theta=5e5), chain_call(1, theta=1e6)]
    st, sel, stats = run_step(S, table, calls)
    assert (st, sel, stats.fused_launches) == (S.OK, [0, 1], 1)


def test_long_steps_are_chunked(S):
    table = [chain_spec()]
    calls = [chain_call(k) for k in range(50)]
    st, sel, stats = run_step(S, table, calls)
    assert st == S.OK and sel == [0] * 50
    assert (stats.fused_launches, stats.fused_calls) == (2, 50)
    # a single call, and a last chunk of one call, take the one-call path
    st, sel, stats = run_step(S, table, calls[:49])
    assert (stats.fused_launches, stats.fused_calls, stats.hits) == (1, 48, 49)
    st, sel, stats = run_step(S, table, calls[:1])
    assert (st, stats.fused_launches, stats.hits) == (S.OK, 0, 1)


def test_failed_fused_launch_reports_the_chunk(S):
    table = [chain_spec()]
    calls = [chain_call(k) for k in range(50)]
    st, sel, stats = run_step(S, table, calls, flags=S.OPT_FAIL_LAUNCHES)
    assert st == S.ERR_CUDA
    assert sel == [0] * 48 + [NOT_RUN] * 2
    assert stats.err_cuda == 1 and stats.hits == 0 and stats.fused_launches == 0


def test_non_chain_ops_take_the_sequential_path(S):
    norm = cases.make_spec(dict(op=1, fixed=[4096], tok=[1, 64]))
    a = cases.make_args(dict(op=1, T=1, H=4096))
    b = cases.make_args(dict(op=1, T=1, H=4096))
    for t in b["tensors"]:
        t["addr"] += 1 << 40
    st, sel, stats = run_step(S, [norm], [a, b])
    assert (st, sel, stats.fused_launches, stats.hits) == (S.OK, [0, 0], 0, 2)


def test_scattered_layouts_take_the_sorting_path(S):
    """30 calls whose tensors sit at addresses permuted independently per slot (more than
    24 ascending runs, so the extents are sorted rather than merged): independent calls
    fuse; one call reading another's output makes the step run call by call."""
    rng = random.Random(7)
    table = [chain_spec()]
    n = 30
    calls = [chain_call(0) for _ in range(n)]
    for slot in range(18):
        perm = list(range(n))
        rng.shuffle(perm)
        for k in range(n):
            calls[k]["tensors"][slot]["addr"] += perm[k] << 40
    assert len({(t["addr"]) for c in calls for t in c["tensors"]}) == n * 18
    st, sel, stats = run_step(S, table, calls)
    assert (st, stats.fused_launches, stats.fused_calls) == (S.OK, 1, n)
    calls[17]["tensors"][1] = dict(calls[4]["tensors"][14])  # r0 of call 17 = r2 of call 4
    st, sel, stats = run_step(S, table, calls)
    assert (st, sel, stats.fused_launches, stats.hits) == (S.OK, [0] * n, 0, n)
