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
        wb = p["bn"] * 64  # W bytes per CTA and K slice of one tile
        # a pass stage's third slot: the second tile's W, or the partner row block's H (16 KB) when a group
        # owns more than one row block (row-pair sweeps)
        third = (16384 if p["n_mb"] > p["n_groups"] and wb < 16384 else wb) if p["two"] else 0
        assert p["stage_bytes"] == 16384 + wb + third, p
        ring = p["stages"] * p["stage_bytes"]
        assert 2 <= p["stages"] <= 7 and ring + SMEM_OVERHEAD <= SMEM_MAX, p
        assert 2 * (ring + SMEM_OVERHEAD) > SM_SHARED, p  # never two CTAs (two TMEM owners) on one SM
        # the workspace holds G records per row
        assert wino.wino_workspace_size(N, 4096, V) >= N * p["G"] * 16


def _walk(plan):
    """The items each CTA pair computes, in the order the score kernel's three roles walk them: per pair a
    list of items, each a list of (row block, tile, accumulator); and the vocabulary sweeps per group."""
    pairs = plan["ctas"] // 2
    ng, G, n_mb, n_vt, two = plan["n_groups"], plan["G"], plan["n_mb"], plan["n_vt"], plan["two"]
    items, sweeps = {}, {}
    for c in range(pairs):
        grp, col = c % ng, c // ng
        out = items.setdefault(c, [])
        for mb in range(grp, n_mb, 2 * ng if two else ng):
            sweeps[grp] = sweeps.get(grp, 0) + (1 if col == 0 else 0)
            mb2 = mb + ng
            if two and mb2 < n_mb:  # row-pair sweep: one tile of both blocks per item
                for vt in range(col, n_vt, G):
                    out.append([(mb, vt, 0), (mb2, vt, 1)])
            elif two:  # tile-pair sweep of a block without a partner
                for vt in range(col, n_vt, 2 * G):
                    out.append([(mb, vt, 0)] + ([(mb, vt + G, 1)] if vt + G < n_vt else []))
            else:  # single tiles, alternating accumulators
                for vt in range(col, n_vt, G):
                    out.append([(mb, vt, len(out) & 1)])
    return items, sweeps


@pytest.mark.parametrize("N,V", [(64, 1000), (256, 126464), (300, 5000), (768, 126464), (1024, 126464),
                                 (1280, 126464), (2048, 134400), (4096, 32641), (8192, 1000)])
def test_every_tile_once_and_balanced(N, V):
    p = wino.wino_score_plan_host(N, 4096, V)
    own = _owners(p)
    assert sorted(own) == sorted(itertools.product(range(p["n_mb"]), range(p["n_vt"])))
    assert all(len(v) == 1 for v in own.values())
    # the kernel's walk computes the same (row block, tile) set, each once, both accumulators of a pass
    # holding different tiles
    items, sweeps = _walk(p)
    walked = [(mb, vt) for its in items.values() for it in its for mb, vt, _ in it]
    assert sorted(walked) == sorted(own)
    assert all(len({acc for _, _, acc in it}) == len(it) for its in items.values() for it in its)
    # with passes, a group sweeps the vocabulary (reads W) once per two of its row blocks
    if p["two"]:
        for g in range(p["n_groups"]):
            assert sweeps[g] == math.ceil(len(range(g, p["n_mb"], p["n_groups"])) / 2)
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
        assert b8["n_mb"] == 2 * b8["n_groups"]  # one row-pair sweep per group: W is read once
    loop = wino.wino_score_plan_host(1024, 4096, 126464)
    assert (loop["bn"], loop["n_groups"], loop["G"], loop["two"]) == (256, 4, 19, 1)


def test_plan_host_argument_errors():
    for args in ((256, 4096, 126464, 1, 76), (256, 4096, 126464, 152, 0), (0, 4096, 126464, 152, 76),
                 (256, 4096, 1, 152, 76)):
        with pytest.raises(wino.WinoError):
            wino.wino_score_plan_host(*args)
