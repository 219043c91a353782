"""invoke_step's replay cache on the host (dry-run SCM, no GPU): a chunk whose argument
bytes repeat is relaunched from the stored parameters from its third occurrence on, and
every step's status, selections, fused decision and statistics equal those of an SCM with
the cache off (which runs selection, the byte rules and packing every time)."""
import random
import threading

import pytest

from oracle import guards as G
from tests import cases
from tests.test_step_host import ACT_SLOTS, chain_call, chain_spec

NOT_RUN = -2


@pytest.fixture()
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def make_scm(S, table, flags=0, hook=None):
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN | flags, hook=hook)
    for sp in table:
        s.register(cases.lib_spec(sp))
    return s


def arr(S, calls):
    return (S.trident_args * len(calls))(*[cases.lib_args(c) for c in calls])


def test_third_repeat_replays(S):
    table = [chain_spec()]
    a = arr(S, [chain_call(k) for k in range(5)])
    s = make_scm(S, table)
    seen = []
    for _ in range(4):
        seen.append(s.invoke_step(a))
        st = s.stats()
    assert seen == [(S.OK, [0] * 5)] * 4
    assert st.step_replays == 2 * 5  # steps 3 and 4
    assert (st.invokes, st.hits, st.fused_launches, st.fused_calls) == (20, 20, 4, 20)
    assert st.guard_evals == 2 * 5  # only the two full-path steps evaluated guards
    s.close()


def test_cache_off_never_replays(S):
    table = [chain_spec()]
    a = arr(S, [chain_call(k) for k in range(3)])
    s = make_scm(S, table, flags=S.OPT_NO_STEP_REPLAY)
    for _ in range(5):
        assert s.invoke_step(a) == (S.OK, [0] * 3)
    st = s.stats()
    assert st.step_replays == 0 and st.fused_launches == 5 and st.guard_evals == 15
    s.close()


def test_any_changed_byte_takes_the_full_path(S):
    """After the chunk is stored, a copy that differs in one pointer (now a dependency), in
    eps (not guarded, but packed) or in theta (guarded) is not replayed."""
    table = [chain_spec(theta=5e5), chain_spec(theta=1e6)]
    calls = [chain_call(k) for k in range(3)]
    s = make_scm(S, table)
    for _ in range(3):
        assert s.invoke_step(arr(S, calls)) == (S.OK, [0] * 3)
    assert s.stats().step_replays == 3
    dep = [dict(c, tensors=[dict(t) for t in c["tensors"]]) for c in calls]
    dep[1]["tensors"][1] = dict(dep[0]["tensors"][14])  # call 1 reads call 0's r2
    assert s.invoke_step(arr(S, dep)) == (S.OK, [0] * 3)
    st = s.stats()
    assert (st.step_replays, st.fused_launches) == (3, 3)  # ran call by call
    eps = [dict(c, eps=1e-3) for c in calls]
    assert s.invoke_step(arr(S, eps)) == (S.OK, [0] * 3)
    assert s.stats().step_replays == 3 and s.stats().fused_launches == 4
    th = [dict(c, theta=1e6) for c in calls]
    assert s.invoke_step(arr(S, th)) == (S.OK, [1] * 3)
    assert s.stats().step_replays == 3
    s.close()


def test_table_growth_keeps_replays_valid(S):
    """Versions appended after a chunk was stored cannot change its first matches: the
    replayed selections still equal the oracle's over the grown table."""
    table = [chain_spec(tok=(1, 64))]
    calls = [chain_call(k) for k in range(4)]
    s = make_scm(S, table)
    for _ in range(2):
        s.invoke_step(arr(S, calls))
    grown = table + [chain_spec(tok=(1, 1)), chain_spec()]
    for sp in grown[1:]:
        s.register(cases.lib_spec(sp))
    assert s.invoke_step(arr(S, calls)) == (S.OK, [G.select(grown, c)[1] for c in calls])
    assert s.stats().step_replays == 4
    s.close()


def test_least_recently_used_entry_is_replaced(S):
    """Five repeating steps with four entries: each step stays correct; a step used again
    after four others were stored has been evicted and takes the full path once more."""
    table = [chain_spec()]
    steps = [arr(S, [chain_call(10 * j + k) for k in range(2)]) for j in range(5)]
    s = make_scm(S, table)
    for j in range(5):  # seen, then stored
        s.invoke_step(steps[j])
        s.invoke_step(steps[j])
    assert s.stats().step_replays == 0
    for j in (1, 2, 3, 4):  # the four most recent entries replay
        assert s.invoke_step(steps[j]) == (S.OK, [0, 0])
    assert s.stats().step_replays == 8
    assert s.invoke_step(steps[0]) == (S.OK, [0, 0])  # evicted: full path (and stored again)
    assert s.stats().step_replays == 8
    assert s.invoke_step(steps[0]) == (S.OK, [0, 0])
    assert s.stats().step_replays == 10
    s.close()


def test_failed_launches_are_never_stored(S):
    table = [chain_spec()]
    a = arr(S, [chain_call(k) for k in range(3)])
    s = make_scm(S, table, flags=S.OPT_FAIL_LAUNCHES)
    for _ in range(4):
        st, sel = s.invoke_step(a)
        assert st == S.ERR_CUDA and sel == [0] * 3
    st = s.stats()
    assert (st.step_replays, st.err_cuda, st.hits) == (0, 4, 0)
    s.close()


@pytest.mark.parametrize("seed", range(6))
def test_random_step_streams_equal_the_cache_off_path(S, seed):
    """A stream of steps drawn from a small pool (independent chunks, chunks with a
    cross-call dependency, chunks with an invalid in-call alias, chunks that miss): every
    result and the final statistics other than the replay and guard-evaluation counts
    equal those of an SCM with the cache off."""
    rng = random.Random(seed)
    table = [chain_spec(tok=(1, 4))]
    pool = []
    for j in range(7):
        m = rng.choice((2, 3, 5))
        calls = [chain_call(20 * j + k) for k in range(m)]
        kind = rng.choice(("indep", "indep", "indep", "dep", "alias", "miss"))
        if kind == "dep":
            calls[1]["tensors"][1] = dict(calls[0]["tensors"][14])
        elif kind == "alias":
            i, si, sj = rng.randrange(m), rng.choice(ACT_SLOTS), rng.choice(ACT_SLOTS)
            if si != sj:
                calls[i]["tensors"][si] = dict(calls[i]["tensors"][sj])
        elif kind == "miss":
            calls[m - 1] = chain_call(20 * j + m - 1, T=8)
        pool.append(arr(S, calls))
    on, off = make_scm(S, table), make_scm(S, table, flags=S.OPT_NO_STEP_REPLAY)
    for _ in range(60):
        a = pool[rng.randrange(len(pool))]
        assert on.invoke_step(a) == off.invoke_step(a)
    x, y = on.stats(), off.stats()
    assert x.step_replays > 0
    for f in ("invokes", "hits", "misses", "err_invalid", "err_cuda", "fused_launches", "fused_calls"):
        assert getattr(x, f) == getattr(y, f), f
    assert y.step_replays == 0 and x.guard_evals < y.guard_evals
    on.close()
    off.close()


def test_concurrent_replays(S):
    """Threads stepping the same SCM at once: a thread that finds the cache in use takes the
    full path; every call is counted once and every step selects the same versions."""
    table = [chain_spec()]
    steps = [arr(S, [chain_call(10 * j + k) for k in range(3)]) for j in range(3)]
    s = make_scm(S, table)
    bad = []

    def run(t):
        for i in range(300):
            if s.invoke_step(steps[(i + t) % 3]) != (S.OK, [0, 0, 0]):
                bad.append(t)

    th = [threading.Thread(target=run, args=(t,)) for t in range(4)]
    for t in th:
        t.start()
    for t in th:
        t.join()
    st = s.stats()
    assert not bad
    assert (st.invokes, st.hits, st.fused_launches) == (3600, 3600, 1200)
    assert 0 < st.step_replays <= 3600
    s.close()
