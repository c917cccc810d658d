"""The LM-head work plan (csrc/common.cuh), compiled for the host and checked
without a GPU: every (m-tile, v-tile) pair of the logits is computed by
exactly one unit, the units of every vocabulary part run in the same round
(so its head slice is fetched once), partial-slot indices stay within what
the merge reads, and the busiest runner carries close to an even share of the
v-tiles. The cases are the five workloads' windows in each kernel's plan plus
ragged and degenerate ones."""

import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_33887_gb300", "csrc")


def _nvcc():
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    return None


@pytest.fixture(scope="module")
def plan_check(tmp_path_factory):
    nvcc = _nvcc()
    if nvcc is None:
        pytest.skip("no CUDA toolkit")
    exe = str(tmp_path_factory.mktemp("plan") / "plan_check")
    r = subprocess.run([nvcc, "-std=c++17", "-O1", "-I" + CSRC, os.path.join(ROOT, "tests", "plan_check.cu"),
                        "-o", exe], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return exe


def run_cases(exe, cases):
    args = [str(x) for c in cases for x in c]
    out = subprocess.run([exe] + args, capture_output=True, text=True, check=True).stdout.split("\n")
    return [l.split() for l in out if l.strip()]


PAIR_G, QUAD_G, SMS = 76, 36, 152
# (n_rows, BM, GM, vt_kb, row_bytes, G, n_vt, cpu, mc, vc, G2, spill_pct); vt_kb =
# KiB of head per v-tile, row_bytes = bytes of a packed token row, as the
# kernels read them; mc = m-tiles a runner holds (2: clusters of two CTA
# pairs sharing head tiles), vc = v-tiles it takes per step (2: clusters of
# two pairs sharing token rows); G2 = spill pairs beside the clusters (0:
# none), spill_pct = a spill pair's time per tile against a cluster pair's
CASES = [
    # pair kernel in clusters of two pairs (BM = 0: token groups from N; GM = 0: bands by rule)
    (294, 0, 0, 1024, 4096, QUAD_G, 594, 2, 2, 1, 0, 100),       # 8 x 2 x 32, d = 2048, bf16
    (2048, 0, 0, 1024, 4096, QUAD_G, 614, 2, 2, 1, 0, 100),      # 32 x 4 x 32
    (8191, 0, 0, 2048, 8192, QUAD_G, 594, 2, 2, 1, 0, 100),      # 64 x 4 x 64, d = 4096
    (8200, 0, 0, 2048, 8192, QUAD_G, 594, 2, 2, 1, 0, 100),      # one row into another group (33 groups: odd)
    (52429, 0, 0, 1280, 10240, QUAD_G, 614, 2, 2, 1, 0, 100),    # 256 x 8 x 64, d = 5120, E4M3 head, two-term rows
    (32, 0, 0, 64, 1024, QUAD_G, 16, 2, 2, 1, 0, 100),           # the tiny window
    (1, 0, 0, 1, 16, QUAD_G, 1, 2, 2, 1, 0, 100),                # one row, one v-tile
    (257, 0, 0, 1024, 4096, 3, 7, 2, 2, 1, 0, 100),              # few runners
    (5000, 0, 7, 1024, 4096, QUAD_G, 100, 2, 2, 1, 0, 100),      # a fixed band size
    # single CTA pairs (quantised heads decoded in the kernel)
    (294, 0, 0, 1024, 4096, PAIR_G, 594, 2, 1, 1, 0, 100),
    (8191, 0, 0, 2048, 8192, PAIR_G, 594, 2, 1, 1, 0, 100),
    (52429, 0, 0, 1280, 10240, PAIR_G, 614, 2, 1, 1, 0, 100),
    # one-CTA kernel (BM = 128) and the SIMT kernel (BM = 32, 64-entry v-tiles)
    (8191, 128, 0, 2048, 8192, SMS, 594, 1, 1, 1, 0, 100),
    (52429, 128, 0, 2560, 10240, SMS, 614, 1, 1, 1, 0, 100),
    (294, 32, 0, 512, 4096, 2 * SMS, 2374, 1, 1, 1, 0, 100),
    (32, 32, 0, 64, 1024, 2 * SMS, 64, 1, 1, 1, 0, 100),
    (5, 32, 0, 1, 100, 2 * SMS, 3, 1, 1, 1, 0, 100),
]


def test_plan_covers_every_tile_once_with_balanced_runners(plan_check):
    res = run_cases(plan_check, CASES)
    assert len(res) == len(CASES)
    for case, r in zip(CASES, res):
        assert r[0] == "ok", (case, r)
        n_mt, gv, slots, max_load, ideal = int(r[1]), int(r[2]), int(r[3]), int(r[4]), float(r[5])
        G, n_vt, cpu, vc = case[5], case[6], case[7], case[9]
        steps = -(-n_vt // vc)
        assert 1 <= gv <= min(G, steps) and slots == gv * cpu * vc
        assert int(r[7]) == n_vt  # no spill launch: the main launch takes every v-tile
        # the busiest runner: within 10% of an even share plus one unit of
        # work (ceil(steps / gv) steps), which no static split can avoid
        assert max_load <= 1.10 * ideal + -(-steps // gv), (case, r)


def test_plan_without_rows(plan_check):
    (r,) = run_cases(plan_check, [(0, 0, 0, 1024, 4096, QUAD_G, 594, 2, 2, 1, 0, 100)])
    assert r[0] == "ok" and int(r[1]) == 0


def test_band_size(plan_check):
    # the chosen band sizes (runner m-tiles): the 64 x 4 x 64 window on 36
    # clusters packs bands of 12 runner m-tiles (12 + 4) into exactly full
    # rounds; the largest window (more than two rounds' worth of m-tiles: rows
    # in flight within 12 MiB) 2 runner m-tiles on clusters, 4 m-tiles on 76
    # single pairs; one row past 32 groups on clusters: 12; the 32 x 4 x 32
    # window is one band (8 m-tiles, within 5% of the best makespan); a fixed GM
    # is kept
    rows = run_cases(plan_check, [(8191, 0, 0, 2048, 8192, QUAD_G, 594, 2, 2, 1, 0, 100),
                                  (52429, 0, 0, 1280, 10240, QUAD_G, 614, 2, 2, 1, 0, 100),
                                  (52429, 0, 0, 1280, 10240, PAIR_G, 614, 2, 1, 1, 0, 100),
                                  (8200, 0, 0, 2048, 8192, QUAD_G, 594, 2, 2, 1, 0, 100),
                                  (2048, 0, 0, 1024, 4096, PAIR_G, 614, 2, 1, 1, 0, 100),
                                  (5000, 0, 7, 1024, 4096, QUAD_G, 100, 2, 2, 1, 0, 100)])
    assert [int(r[6]) for r in rows] == [12, 2, 4, 12, 8, 7]
    # 64 x 4 x 64 on clusters: an even share exactly (16 runner m-tiles x 594 v-tiles / 36)
    assert int(rows[0][4]) == 264


# the clusters-of-two-pairs cases with the 4 spill pairs 152 SMs leave room for
SPILL_CASES = [c[:10] + (4, pct) for c in CASES if c[8] == 2 and c[5] == QUAD_G for pct in (100, 110)]
# the same clusters with their pairs sharing token rows (one m-tile, two v-tiles per step)
SHARE_CASES = [c[:8] + (1, 2) + c[10:] for c in CASES if c[8] == 2 and c[5] == QUAD_G]
SHARE_CASES += [(294, 0, 0, 1024, 4096, QUAD_G, 593, 2, 1, 2, 0, 100),  # odd v-tile count
                (52429, 0, 0, 1280, 10240, QUAD_G, 613, 2, 1, 2, 0, 100)]
SHARE_SPILL_CASES = [c[:10] + (4, pct) for c in SHARE_CASES for pct in (100, 110)]


def test_plan_with_pairs_sharing_token_rows(plan_check):
    res = run_cases(plan_check, SHARE_CASES)
    assert len(res) == len(SHARE_CASES)
    for case, r in zip(SHARE_CASES, res):
        assert r[0] == "ok", (case, r)
        gv, slots, max_load, ideal = int(r[2]), int(r[3]), int(r[4]), float(r[5])
        steps = -(-case[6] // 2)
        assert slots == 4 * gv  # each pair of a unit writes its own partial per CTA
        assert max_load <= 1.10 * ideal + -(-steps // gv), (case, r)


@pytest.mark.parametrize("cases", ["head", "tokens"])
def test_spill_launch_covers_the_rest_of_the_vocabulary(plan_check, cases):
    todo = SPILL_CASES if cases == "head" else SHARE_SPILL_CASES
    res = run_cases(plan_check, todo)
    assert len(res) == len(todo)
    for case, r in zip(todo, res):
        assert r[0] == "ok", (case, r)
        n_mt, gv, slots, load, ideal, gm = int(r[1]), int(r[2]), int(r[3]), int(r[4]), float(r[5]), int(r[6])
        vsplit, load2, gm2, gv2 = int(r[7]), int(r[8]), int(r[9]), int(r[10])
        G, n_vt, cpu, vc, G2, pct = case[5], case[6], case[7], case[9], case[10], case[11]
        assert 1 <= vsplit <= n_vt and slots == gv * cpu * vc + gv2 * 2
        if n_mt == 0 or vsplit == n_vt:
            continue
        assert vsplit % vc == 0
        steps = vsplit // vc
        assert 1 <= gv2 <= min(G2, n_vt - vsplit) and 1 <= gv <= min(G, steps)
        # either launch's busiest runner within 10% of the even share plus one
        # unit of its launch, which no static split avoids
        w = pct / 100
        assert load <= 1.10 * ideal + -(-steps // gv), (case, r)
        assert w * load2 <= 1.10 * ideal + w * -(-(n_vt - vsplit) // gv2), (case, r)


def test_spill_split_of_the_bench_window(plan_check):
    # 8 x 2 x 32 window, 294 rows: two token groups (one runner m-tile of two)
    # on 36 clusters and 4 spill pairs. At equal time per tile the split
    # balances 594 v-tiles as 563 for the clusters (one m-tile pair each) and
    # 31 for the spill pairs (both m-tiles); a spill pair 10% slower gets 29
    (a, b) = run_cases(plan_check, [(294, 0, 0, 1024, 4096, QUAD_G, 594, 2, 2, 1, 4, 100),
                                    (294, 0, 0, 1024, 4096, QUAD_G, 594, 2, 2, 1, 4, 110)])
    assert int(a[7]) == 563 and int(b[7]) == 565


def test_token_sharing_split_is_even(plan_check):
    # 8 x 2 x 32 window on clusters whose pairs share token rows: the split of
    # 594 v-tiles keeps an even count for the clusters' v-tile pairs (562 at
    # equal time per tile against 563 with head sharing)
    (a,) = run_cases(plan_check, [(294, 0, 0, 1024, 4096, QUAD_G, 594, 2, 1, 2, 4, 100)])
    assert a[0] == "ok" and int(a[7]) == 562


def _fuzz_cases(n, seed):
    import random

    rnd = random.Random(seed)
    cases = []
    for _ in range(n):
        kind = rnd.choice(["pair", "pair", "tc", "simt"])
        n_rows = rnd.choice([0, 1, rnd.randint(1, 600), rnd.randint(1, 9000), rnd.randint(1, 60000)])
        n_vt = rnd.choice([1, 2, 3, rnd.randint(1, 40), rnd.randint(1, 700)])
        gm = rnd.choice([0, 0, 0, rnd.randint(1, 40)])
        vt_kb, row_bytes = rnd.choice([(1024, 4096), (2048, 8192), (1280, 10240), (64, 1024)])
        if kind == "pair":
            layout = rnd.choice(["pairs", "head", "tokens"])
            mc, vc = {"pairs": (1, 1), "head": (2, 1), "tokens": (1, 2)}[layout]
            G = rnd.choice([rnd.randint(1, 40), 36, 76]) if layout == "pairs" else rnd.choice([rnd.randint(1, 40), 36])
            G2 = rnd.choice([0, rnd.randint(1, 8)]) if layout != "pairs" else 0
            cases.append((n_rows, 0, gm, vt_kb, row_bytes, G, n_vt, 2, mc, vc, G2, rnd.choice([50, 100, 110, 400])))
        else:
            bm = 128 if kind == "tc" else 32
            G = rnd.choice([rnd.randint(1, 320), 152, 304])
            cases.append((n_rows, bm, gm, vt_kb, row_bytes, G, n_vt, 1, 1, 1, 0, 100))
    return cases


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_random_plans_cover_every_tile_once(plan_check, seed):
    # seeded random shapes over every kernel's plan and both cluster layouts,
    # with and without spill pairs: every (m-tile, v-tile) pair computed once,
    # parts whole within rounds, partial slots within the merge's range
    cases = _fuzz_cases(150, seed)
    res = run_cases(plan_check, cases)
    assert len(res) == len(cases)
    for case, r in zip(cases, res):
        assert r[0] == "ok", (case, r)
