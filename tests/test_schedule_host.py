"""The score kernel's work split (score_schedule through wino_score_plan_host), on the CPU: every
(row block, vocabulary tile) goes to exactly one CTA pair, the pairs of a group carry tile counts within
one of each other, the records per row fit the workspace, the ring fits shared memory and keeps one CTA per
SM, and the benchmark shapes get the splits the kernel was tuned on."""
import itertools
import math

import pytest

import paper_2605_16941_gb300 as wino

SMEM_MAX = 227 * 1024        # dynamic shared memory a CTA may request
SMEM_OVERHEAD = 1024 + 256   # ring alignment slack + barrier block
SM_SHARED = 228 * 1024       # shared memory of one SM

DEVICES = [(152, 76), (148, 74), (132, 66), (152, 72), (8, 4), (2, 1)]
ROWS = [1, 64, 128, 255, 256, 257, 512, 1024, 2048, 4096, 32768, 1 << 24]
VOCABS = [2, 1000, 32640, 32641, 126464, 134400, 1 << 27]


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2605_16941_gb300 import build
    build.build()


def _owners(plan):
    """(row block, tile) -> pairs that compute it, following the split the kernel walks."""
    own = {}
    pairs = plan["ctas"] // 2
    for c in range(pairs):
        grp, col = c % plan["n_groups"], c // plan["n_groups"]
        for mb in range(grp, plan["n_mb"], plan["n_groups"]):
            for vt in range(col, plan["n_vt"], plan["G"]):
                own.setdefault((mb, vt), []).append(c)
    return own


@pytest.mark.parametrize("sm,pairs", DEVICES, ids=[f"sm{a}_p{b}" for a, b in DEVICES])
def test_split_invariants(sm, pairs):
    units = min(pairs, sm // 2)
    for N, V in itertools.product(ROWS, VOCABS):
        p = wino.wino_score_plan_host(N, 4096, V, sm, pairs)
        assert p["bn"] % 16 == 0 and 128 <= p["bn"] <= 256, p
        assert p["n_vt"] == math.ceil(V / p["bn"]) and p["n_mb"] == math.ceil(N / 256), p
        assert 1 <= p["n_groups"] <= min(p["n_mb"], units), p
        assert 1 <= p["G"] <= min(p["n_vt"], p["records_per_row"]), p
        assert p["n_groups"] * p["G"] <= units and p["ctas"] == 2 * p["n_groups"] * p["G"], p
        assert p["records_per_row"] == min(math.ceil(V / 128), 256), p
        assert p["two"] == (1 if p["n_mb"] >= 2 else 0), p
        assert p["stage_bytes"] == 16384 + (1 + p["two"]) * p["bn"] * 64, p
        ring = p["stages"] * p["stage_bytes"]
        assert 2 <= p["stages"] <= 7 and ring + SMEM_OVERHEAD <= SMEM_MAX, p
        assert 2 * (ring + SMEM_OVERHEAD) > SM_SHARED, p  # never two CTAs (two TMEM owners) on one SM
        # the workspace holds G records per row
        assert wino.wino_workspace_size(N, 4096, V) >= N * p["G"] * 16


@pytest.mark.parametrize("N,V", [(64, 1000), (256, 126464), (300, 5000), (1024, 126464), (2048, 134400),
                                 (4096, 32641), (8192, 1000)])
def test_every_tile_once_and_balanced(N, V):
    p = wino.wino_score_plan_host(N, 4096, V)
    own = _owners(p)
    assert sorted(own) == sorted(itertools.product(range(p["n_mb"]), range(p["n_vt"])))
    assert all(len(v) == 1 for v in own.values())
    for g in range(p["n_groups"]):  # within a group, tiles per pair and row block differ by at most one
        counts = [len(range(c // p["n_groups"], p["n_vt"], p["G"])) for c in range(g, p["ctas"] // 2, p["n_groups"])]
        assert max(counts) - min(counts) <= 1


def test_benchmark_shapes():
    """The splits the measurements were taken with on a GB300 (152 SMs, 76 resident pairs)."""
    b1 = wino.wino_score_plan_host(256, 4096, 126464)
    assert (b1["bn"], b1["n_vt"], b1["n_groups"], b1["G"], b1["two"], b1["stages"]) == (240, 527, 1, 76, 0, 7)
    for V, tiles in ((126464, 26), (134400, 28)):
        b8 = wino.wino_score_plan_host(2048, 4096, V)
        assert (b8["bn"], b8["n_groups"], b8["G"], b8["two"], b8["stages"]) == (256, 4, 19, 1, 4)
        assert math.ceil(b8["n_vt"] / b8["G"]) == tiles
    loop = wino.wino_score_plan_host(1024, 4096, 126464)
    assert (loop["bn"], loop["n_groups"], loop["G"], loop["two"]) == (256, 4, 19, 1)


def test_plan_host_argument_errors():
    for args in ((256, 4096, 126464, 1, 76), (256, 4096, 126464, 152, 0), (0, 4096, 126464, 152, 76),
                 (256, 4096, 1, 152, 76)):
        with pytest.raises(wino.WinoError):
            wino.wino_score_plan_host(*args)
