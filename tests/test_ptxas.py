"""Resource budgets of the hot-path kernels as ptxas reports them for sm_103a
(cross-compiled, no GPU): no register spills anywhere on the path, and the
register counts the launch shapes are designed around -- the pipelined scorer's
18 warps in one SM's register file, the prefix walk's 8 CTAs of 4 warps per SM
(every request of a 4096-request batch in one wave)."""
import concurrent.futures as cf
import os
import re
import subprocess

import pytest

from paper_2606_00946_gb300 import build as B

FILES = ["k_score_tc.cu", "k_prefix_index.cu", "k_train_fast.cu", "k_publish.cu", "k_guards.cu", "k_replay.cu"]


@pytest.fixture(scope="module")
def kernels(tmp_path_factory):
    try:
        cc = B.nvcc()
    except RuntimeError:
        pytest.skip("nvcc not found")
    out = tmp_path_factory.mktemp("ptxas")

    def one(f):
        r = subprocess.run([cc] + B.ARCH + B.FLAGS + ["-Xptxas", "-v", "-c", os.path.join(B.CSRC, f), "-o",
                            str(out / (f + ".o"))], capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
        return r.stdout + r.stderr

    with cf.ThreadPoolExecutor(len(FILES)) as ex:
        text = "\n".join(ex.map(one, FILES))
    res = {}
    entry = None
    for line in text.splitlines():
        m = re.search(r"Compiling entry function '(\w+)'", line)
        if m:
            entry = m.group(1)
            res.setdefault(entry, {})
            continue
        if entry is None:
            continue
        m = re.search(r"(\d+) bytes spill stores, (\d+) bytes spill loads", line)
        if m:
            res[entry]["spill"] = int(m.group(1)) + int(m.group(2))
        m = re.search(r"Used (\d+) registers", line)
        if m:
            res[entry]["regs"] = int(m.group(1))
    return res


def _find(kernels, name):
    hits = {k: v for k, v in kernels.items() if name in k}
    assert hits, f"{name} not compiled"
    return hits


# The guard kernel calls two out-of-line fp64 chains (the exact mean and
# threshold, taken only when an fp32 decision lies within its error bound);
# ptxas saves the caller's live registers around those calls, which it
# reports as spill traffic of the kernel.
CALL_SAVES = {"k_guards": 16}


def test_no_spills_on_the_path(kernels):
    for name in ("k_score_tc_pipe", "k_score_wide", "k_score_pair", "k_feature_image", "k_prefix_index", "k_tr_gemm", "k_tr_step", "k_tr_gather",
                 "k_tr_opt", "k_publish", "k_guards", "k_ring_bounds", "k_dist_rowmin"):
        for k, v in _find(kernels, name).items():
            assert v.get("spill", 0) <= 2 * CALL_SAVES.get(name, 0), (k, v)


def test_register_budgets(kernels):
    (pipe,) = _find(kernels, "k_score_tc_pipe").values()
    assert pipe["regs"] * 576 <= 65536          # 18 warps, one CTA per SM
    pairs = _find(kernels, "k_score_pair").values()  # two and three hidden layers
    assert len(pairs) == 2
    for pair in pairs:
        assert pair["regs"] * 512 <= 65536      # 16 warps, one CTA per SM (budgets then moved by setmaxnreg)
    for words in ("ILi1E", "ILi2E", "ILi4E"):   # 1, 2, 4 instance-mask words (up to 256 instances)
        walk = [v for k, v in _find(kernels, "k_prefix_index").items() if words in k]
        assert walk and walk[0]["regs"] <= 64   # 8 CTAs x 128 threads per SM
    for v in _find(kernels, "k_tr_gemm").values():
        assert v["regs"] * 512 <= 65536
