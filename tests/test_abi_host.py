"""Host-side checks of the C ABI that need no GPU.

The library must load, export every function include/cure.h declares, and
reject bad host arguments before launching anything.
"""
import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cure.h")


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    try:
        __graft_entry__.build()
    except RuntimeError as e:  # no toolkit on this machine
        pytest.skip(f"cannot build libcure: {e}")
    from paper_2608_00531_gb300 import _lib
    return _lib.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cure_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_five_stages():
    names = declared_functions()
    for n in ("cure_score_draft", "cure_build_tree", "cure_tree_attn", "cure_accept", "cure_resync_kv"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2608_00531_gb300 import _lib
    out = subprocess.run(["nm", "-D", "--defined-only", _lib.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (cure_[a-z0-9_]+)$", out, flags=re.M))
    for n in declared_functions():
        assert n in exported, n
        assert hasattr(lib, n)
    assert set(_lib.EXPORTS) <= exported


def test_version_and_status_strings(lib):
    assert lib.cure_abi_version() == 105
    assert lib.cure_status_string(0) == b"ok"
    assert lib.cure_status_string(2) == b"workspace too small"


def test_bad_arguments_are_rejected_on_the_host(lib):
    from paper_2608_00531_gb300._lib import KVDesc, TreeParams
    null = C.c_void_p(0)
    # rows < 0, topk outside 2..8, topk > vocab
    assert lib.cure_score_draft(null, -1, 100, 2, null, null, null, null, null) == 1
    assert lib.cure_score_draft(null, 4, 100, 9, null, null, null, null, null) == 1
    assert lib.cure_score_draft(null, 4, 2, 3, null, null, null, null, null) == 1
    # zero rows is a no-op
    assert lib.cure_score_draft(null, 0, 100, 2, null, null, null, null, null) == 0
    # tree parameters
    p = TreeParams(batch=2, block=33, topk=3, tau=1.0, budget=4, branches=2, repair_depth=1, max_ufp=0)
    assert lib.cure_build_tree(C.byref(p), *([null] * 13), null) == 1
    p.block, p.branches = 16, 4          # more branches than stored candidates
    assert lib.cure_build_tree(C.byref(p), *([null] * 13), null) == 1
    p.branches, p.budget = 3, 300       # n_max > 256
    assert lib.cure_build_tree(C.byref(p), *([null] * 13), null) == 5
    p.budget, p.batch = 4, 0            # empty batch: nothing to do
    assert lib.cure_build_tree(C.byref(p), *([null] * 13), null) == 0
    p.batch, p.repair_depth = 1, 2      # depth-2 repairs need the re-drafted successors
    assert lib.cure_build_tree(C.byref(p), *([C.c_void_p(64)] * 5), null, *([C.c_void_p(64)] * 8), null) == 1
    # Eq. (3) dynamic budget: s must be finite and >= 0; b_min within 0..branches-1
    p.batch, p.repair_depth = 0, 1
    for s, bmin, want in ((-1.0, 1, 1), (float("inf"), 1, 1), (float("nan"), 1, 1), (1.0, 3, 1),
                          (1.0, -1, 1), (1.0, 2, 0), (1.0, 0, 0), (0.0, 7, 0)):
        p.margin_scale, p.branch_min = s, bmin
        assert lib.cure_build_tree(C.byref(p), *([null] * 13), null) == want, (s, bmin)
    p.margin_scale, p.branch_min = 0.0, 1
    for md, bw, want in ((-1, 0, 1), (0, -2, 1), (15, 5, 0), (0, 0, 0)):   # caps: >= 0
        p.max_depth, p.beam = md, bw
        assert lib.cure_build_tree(C.byref(p), *([null] * 13), null) == want, (md, bw)
    p.max_depth, p.beam = 0, 0
    # sampling: the temperature must be positive and finite; batch 0 is a no-op
    dev = C.c_void_p(256)
    for T, want in ((0.0, 1), (-1.0, 1), (float("inf"), 1), (float("nan"), 1)):
        assert lib.cure_sample_target(dev, dev, C.c_float(T), 1, 9, 100, dev, dev, null) == want, T
    assert lib.cure_sample_target(dev, null, C.c_float(1.0), 1, 9, 100, dev, dev, null) == 1
    assert lib.cure_sample_target(null, null, C.c_float(1.0), 0, 9, 100, null, null, null) == 0
    # attention: head_dim 64 unsupported, heads_q not a multiple of heads_kv
    kv = KVDesc(layout=0, heads_kv=4, head_dim=64, page_size=16, max_len=100, num_pages=0, block_table=None)
    assert lib.cure_tree_attn(*([null] * 5), C.byref(kv), null, null, null, 1, 9, 8, 1.0, null, null, 0, null) == 5
    kv.head_dim = 128
    assert lib.cure_tree_attn(*([null] * 5), C.byref(kv), null, null, null, 1, 9, 6, 1.0, null, null, 0, null) == 1
    # the in-place layout passes both tree tensors as NULL, never only one of them
    dev = C.c_void_p(256)
    one = (dev, dev, null, dev, dev)
    assert lib.cure_tree_attn(*one, C.byref(kv), dev, dev, dev, 1, 9, 8, 1.0, dev, dev, 1 << 30, null) == 1
    # the softmax scale must be positive and finite
    for bad in (0.0, -1.0, float("inf"), float("nan")):
        assert lib.cure_tree_attn(*([null] * 5), C.byref(kv), null, null, null, 1, 9, 8, bad, null, null, 0,
                                  null) == 1
    # paged without a block table
    kv.layout = 1
    assert lib.cure_tree_attn(*([null] * 5), C.byref(kv), null, null, null, 1, 9, 8, 1.0, null, null, 0, null) == 1
    # resync: more layers than the ABI carries
    kv.layout = 0
    assert lib.cure_resync_kv(129, None, None, C.byref(kv), null, null, 1, 9, 8, *([null] * 9), null) == 1
    # accept: n_max smaller than the chain
    assert lib.cure_accept(null, null, 1, 4, 10, 8, *([null] * 10), null) == 1


def test_workspace_size_is_a_host_computation(lib):
    from paper_2608_00531_gb300._lib import KVDesc
    kv = KVDesc(layout=0, heads_kv=4, head_dim=128, page_size=16, max_len=8192, num_pages=0, block_table=None)
    n = lib.cure_tree_attn_workspace_size(32, 33, 28, C.byref(kv))
    assert n > 0 and n % 256 == 0
    # piece slots: one per (sequence, kv head, row group) plus one per CTA, 256 rows each
    per_slot = 256 * (128 * 4 + 4)
    units = 32 * 4 * 1
    assert n >= (units + 256) * per_slot
    # grows with the batch and the tree, zero on a bad shape
    assert lib.cure_tree_attn_workspace_size(64, 33, 28, C.byref(kv)) > n
    assert lib.cure_tree_attn_workspace_size(32, 97, 28, C.byref(kv)) > n
    kv.head_dim = 96
    assert lib.cure_tree_attn_workspace_size(32, 33, 28, C.byref(kv)) == 0


def test_product_path_has_no_cpu_fallback():
    """The binding fails loudly without the library and never imports the oracle."""
    import importlib
    import paper_2608_00531_gb300 as pkg
    pkg_dir = os.path.dirname(pkg.__file__)
    for fn in os.listdir(pkg_dir):
        if fn.endswith(".py"):
            src = open(os.path.join(pkg_dir, fn)).read()
            assert "import oracle" not in src and "from oracle" not in src, fn
    from paper_2608_00531_gb300 import _lib
    saved, _lib._lib = _lib._lib, None
    real = _lib.LIB_PATH
    try:
        _lib.LIB_PATH = real + ".missing"
        with pytest.raises(ImportError):
            _lib.load()
    finally:
        _lib.LIB_PATH = real
        _lib._lib = saved


def test_noalloc_rejects_shapes_beyond_its_scratch_on_the_host(lib):
    """cure_tree_attn_noalloc returns CURE_ERR_CAPACITY for a shape whose
    split-KV workspace exceeds its 64 MiB static array, before any CUDA call.
    The pointers are stand-ins that are never dereferenced; the test runs only
    where no GPU can be reached, so that a regression in the check can never
    launch a kernel on them."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("runs only without a reachable GPU")
    from paper_2608_00531_gb300._lib import KVDesc
    P, I32 = C.c_void_p, C.c_int32
    lib.cure_tree_attn_noalloc.argtypes = [P, P, P, P, P, C.POINTER(KVDesc), P, P, P, I32, I32, I32,
                                           C.c_float, P, P]
    lib.cure_tree_attn_noalloc.restype = C.c_int
    fake = C.c_void_p(1 << 20)           # aligned, never dereferenced on the host
    kv = KVDesc(layout=1, heads_kv=4, head_dim=128, page_size=16, max_len=600, num_pages=4096,
                block_table=fake)
    scratch = 64 * 1024 * 1024
    assert lib.cure_tree_attn_workspace_size(200, 33, 28, C.byref(kv)) > scratch
    assert lib.cure_tree_attn_noalloc(fake, fake, fake, fake, fake, C.byref(kv), fake, fake, fake, 200, 33, 28,
                                      0.088, fake, None) == 2
    # a shape that fits passes the check and only then needs the device
    assert lib.cure_tree_attn_workspace_size(4, 33, 28, C.byref(kv)) <= scratch
    assert lib.cure_tree_attn_noalloc(fake, fake, fake, fake, fake, C.byref(kv), fake, fake, fake, 4, 33, 28,
                                      0.088, fake, None) == 3


def test_sampling_temperature_must_give_a_finite_scale(lib):
    """log2(e) / T must be a finite float32: subnormal temperatures are
    rejected before anything launches."""
    null = C.c_void_p(0)
    for bad in (0.0, -1.0, float("inf"), float("nan"), 1e-45, 4e-39):
        assert lib.cure_sample_target(null, null, bad, 1, 4, 10, null, null, null) == 1, bad
    # zero sequences with a valid temperature is a no-op
    assert lib.cure_sample_target(null, null, 5e-39, 0, 4, 10, null, null, null) == 0


def test_lm_head_host_checks(lib):
    """Shapes the fused LM head cannot take are refused before any launch."""
    null = C.c_void_p(0)
    fake = C.c_void_p(1 << 20)
    # negative rows, d_model below one K slice, empty vocabulary
    assert lib.cure_lm_head_argmax(null, null, -1, 128, 10, null, null, null, 0, null) == 1
    assert lib.cure_lm_head_argmax(null, null, 4, 32, 10, null, null, null, 0, null) == 1
    assert lib.cure_lm_head_argmax(null, null, 4, 128, 0, null, null, null, 0, null) == 1
    # d_model not a multiple of 64
    assert lib.cure_lm_head_argmax(null, null, 4, 96, 10, null, null, null, 0, null) == 5
    # zero rows is a no-op; missing pointers are rejected
    assert lib.cure_lm_head_argmax(null, null, 0, 128, 10, null, null, null, 0, null) == 0
    assert lib.cure_lm_head_argmax(fake, null, 4, 128, 10, null, fake, fake, 1 << 20, null) == 1
    # misaligned hidden state
    assert lib.cure_lm_head_argmax(C.c_void_p((1 << 20) + 2), fake, 4, 128, 10, null, fake, fake, 1 << 20,
                                   null) == 1
    assert lib.cure_lm_head_workspace_size(-1, 10) == 0
    assert lib.cure_lm_head_workspace_size(4, 0) == 0
    n = lib.cure_lm_head_workspace_size(817, 151936)
    assert n >= 817 * 8 and n % 256 == 0
    # a workspace smaller than the plan's is refused
    assert lib.cure_lm_head_argmax(fake, fake, 817, 4096, 151936, null, fake, fake, n - 256, null) == 2


def test_selftest_limit_is_checked_on_the_host(lib):
    """The failure-detection self-test takes a wait limit of 1 .. 2^30 cycles;
    others are refused before any launch."""
    for bad in (0, -5, (1 << 30) + 1):
        assert lib.cure_selftest_wait_timeout(bad, None) == 1
