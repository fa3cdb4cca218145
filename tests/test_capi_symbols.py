"""The C-ABI library builds, loads without a GPU and exports every entry point include/lsgd.h
declares; the binding's argument structs match the header's layout."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "lsgd.h")


@pytest.fixture(scope="module")
def P():
    from paper_1808_07217_gb300 import _build

    _build.build()
    import paper_1808_07217_gb300 as P

    return P


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(lsgd_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_binding_exports(P):
    assert _declared() == sorted(P.EXPORTS)


def test_library_exports_every_declared_symbol(P):
    L = P.lib()
    for name in _declared():
        assert hasattr(L, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", P.LIB_PATH], capture_output=True, text=True)
    if out.returncode == 0:
        syms = set(line.split()[-1] for line in out.stdout.splitlines() if line.strip())
        for name in _declared():
            assert name in syms, name


def test_struct_layout_matches_header(P):
    # compile a tiny C program that prints sizeof/offsetof of the header's structs
    prog = r"""
    #include <stdio.h>
    #include <stddef.h>
    #include "lsgd.h"
    int main(void) {
      printf("%zu %zu %zu %zu %zu %zu %zu %zu %zu %zu %zu\n", sizeof(lsgd_config), sizeof(lsgd_model),
             sizeof(lsgd_lr_schedule), sizeof(lsgd_allocator), offsetof(lsgd_config, model),
             offsetof(lsgd_config, lr), offsetof(lsgd_config, momentum),
             offsetof(lsgd_config, seed), offsetof(lsgd_config, precision),
             offsetof(lsgd_config, fused_update), sizeof(lsgd_profile));
      printf("%zu %zu %zu %zu %zu %zu %zu\n", offsetof(lsgd_config, hier_block),
             offsetof(lsgd_config, hier_rounds), offsetof(lsgd_config, compress),
             offsetof(lsgd_config, global_momentum), offsetof(lsgd_config, h_warmup),
             offsetof(lsgd_config, h_warmup_epochs), offsetof(lsgd_config, sampling));
      return 0;
    }
    """
    import tempfile

    with tempfile.TemporaryDirectory() as d:
        c = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        open(c, "w").write(prog)
        subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), c, "-o", exe], check=True)
        got = [int(v) for v in subprocess.run([exe], capture_output=True, text=True).stdout.split()]
    C = P.Config
    want = [ctypes.sizeof(C), ctypes.sizeof(P.Model), ctypes.sizeof(P.LrSchedule),
            ctypes.sizeof(P.Allocator), C.model.offset, C.lr.offset, C.momentum.offset,
            C.seed.offset, C.precision.offset, C.fused_update.offset, ctypes.sizeof(P.Profile),
            C.hier_block.offset, C.hier_rounds.offset, C.compress.offset, C.global_momentum.offset,
            C.h_warmup.offset, C.h_warmup_epochs.offset, C.sampling.offset]
    assert got == want


def test_creation_without_gpu_fails_cleanly(P):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    cfg = P.make_config(K=2, B_loc=4, N=16, widths=(8, 3))
    with pytest.raises(P.LsgdError):
        P.lsgd_create(cfg, allocator=None, stream=0)
    # invalid configurations are rejected before any device work
    bad = P.make_config(K=0, B_loc=4, N=16, widths=(8, 3))
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_create(bad, allocator=None, stream=0)
    assert e.value.status == P.EINVAL
    bad = P.make_config(K=2, B_loc=4, N=16, widths=(12, 3), precision=P.BF16)
    with pytest.raises(P.LsgdError) as e:
        P.lsgd_create(bad, allocator=None, stream=0)
    assert e.value.status == P.EUNSUPPORTED
