"""The tensor-core kernels' split plans (host logic, no GPU): which tiles of
the last partial wave are split in K, and where.

A small host program includes the kernels' planning header, prints the plan
of each case, and the test checks the rules the launchers rely on: every
tile is either whole or split once (ntiles_full + nsplit = tiles, the split
point strictly inside K), tile counts that fill whole waves are never split,
fewer tiles than SMs are split in halves exactly when all pieces fit in one
wave, and the benchmark's shape keeps the plan its timing was taken with.
A plan only moves work between CTAs; the GPU tests check that split tiles
give the same bits run to run."""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "..", "paper_2608_10010_gb300", "csrc")
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")

PROGRAM = r"""
#include <cstdio>
#include "tcn_common.cuh"
int main(int argc, char** argv) {
  for (int i = 1; i + 2 < argc; i += 3) {
    const long long tiles = atoll(argv[i]);
    const int sms = atoi(argv[i + 1]), nsub = atoi(argv[i + 2]);
    const cfp::TailPlan n = cfp::tcn_plan_search(tiles, sms, nsub);
    const cfp::TailPlan t = cfp::tail_plan_search(tiles, sms, nsub);
    std::printf("%lld %d %d %d %d %d %d %d %d\n", tiles, sms, nsub, n.ntiles_full, n.nsplit, n.split_step,
                t.ntiles_full, t.nsplit, t.split_step);
  }
  return 0;
}
"""

# (tiles, SMs, steps per tile)
CASES = [(2048, 152, 128), (112, 152, 128), (56, 152, 128), (76, 152, 128), (77, 152, 128), (8, 152, 64),
         (152, 152, 128), (304, 152, 128), (224, 152, 128), (448, 152, 128), (4096, 152, 344), (11008, 152, 128),
         (1, 152, 128), (151, 152, 2), (153, 152, 1), (688, 152, 128), (950, 152, 128)]


@pytest.fixture(scope="module")
def plans(tmp_path_factory):
    if not (os.path.exists(NVCC) or shutil.which("nvcc")):
        pytest.skip("nvcc not available")
    d = tmp_path_factory.mktemp("plan")
    src = d / "plan.cu"
    src.write_text(PROGRAM)
    exe = d / "plan"
    cmd = [NVCC, "-gencode", "arch=compute_103a,code=sm_103a", "-std=c++17", "-O1", "-I", CSRC, str(src), "-o",
           str(exe)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    args = [str(v) for c in CASES for v in c]
    out = subprocess.run([str(exe), *args], capture_output=True, text=True, check=True).stdout.split("\n")
    res = {}
    for line in out:
        if line.strip():
            f = [int(v) for v in line.split()]
            res[tuple(f[:3])] = {"narrow": tuple(f[3:6]), "tile": tuple(f[6:9])}
    return res


def test_every_tile_whole_or_split_once(plans):
    for (tiles, sms, nsub), p in plans.items():
        for kind in ("narrow", "tile"):
            full, nsplit, step = p[kind]
            assert full + nsplit == tiles and full >= 0 and nsplit >= 0, (kind, tiles, p)
            if nsplit:
                assert 0 < step < nsub, (kind, tiles, p)


def test_whole_waves_are_not_split(plans):
    for (tiles, sms, nsub), p in plans.items():
        if tiles % sms == 0:
            assert p["narrow"][1] == 0 and p["tile"][1] == 0, (tiles, p)


def test_fewer_tiles_than_sms(plans):
    """Halves when both pieces of every tile fit in one wave; otherwise the
    per-CTA start (about 6 us) makes a second wave of short pieces slower
    than the whole tiles."""
    for (tiles, sms, nsub), p in plans.items():
        if tiles >= sms or nsub < 2:
            continue
        full, nsplit, step = p["narrow"]
        if 2 * tiles <= sms:
            assert (full, nsplit, step) == (0, tiles, nsub // 2), (tiles, p)
        else:
            assert nsplit == 0, (tiles, p)


def test_benchmark_shape_plan(plans):
    """2,048 tiles of 128 steps on 152 SMs: the last 72 tiles split in halves
    (2,120 CTAs), the plan the benchmark's timing and profile were taken
    with."""
    assert plans[(2048, 152, 128)]["narrow"] == (1976, 72, 64)


def test_steps_too_few_to_split(plans):
    assert plans[(153, 152, 1)]["narrow"][1] == 0 and plans[(153, 152, 1)]["tile"][1] == 0
