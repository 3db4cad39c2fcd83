"""CPU tests of the boundary: the library loads and exports every symbol the
header declares, and host-side argument checks reject bad calls before any
device work (these paths return before touching a GPU)."""
import ctypes
import os
import re

import pytest

from paper_2606_19528_gb300 import lora, build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "lora.h")


def _declared():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:int|int64_t|const char\*)\s+(lora_\w+)\s*\(", src, re.M)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(lora._LIB_PATH):
        build.build_cuda()
    return lora.library()


def test_header_declares_the_binding_names():
    assert _declared() == sorted(lora.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_strerror_and_version(lib):
    assert lora.lora_version() >= 100
    for code in (lora.LORA_OK, lora.LORA_EINVAL, lora.LORA_ENULL, lora.LORA_EALIGN, lora.LORA_ECUDA,
                 lora.LORA_ETIMEOUT, lora.LORA_EWORKSPACE, lora.LORA_EDEVICE):
        assert lora.lora_strerror(code)
    assert lora.lora_strerror(12345) == "unknown error"


def test_null_arguments_are_rejected(lib):
    n = ctypes.c_size_t(0)
    assert lib.lora_workspace_size(None, 1, ctypes.byref(n)) == lora.LORA_ENULL
    assert lib.lora_linear_fwd(None, None, None, None, None, None, None, None, 0, None) == lora.LORA_ENULL
    assert lib.lora_stack_step(None, 1, 1, None, 0, None) == lora.LORA_ENULL
    st = lora.make_shape(128, 256, 256, 8, 2.0)
    assert lib.lora_stack_step(ctypes.byref(lora.make_proj(st)), 0, 1, None, 0, None) == lora.LORA_EINVAL
    assert lib.lora_stack_step(ctypes.byref(lora.make_proj(st)), 1, 7, None, 0, None) == lora.LORA_EINVAL


def test_workspace_sizes_plan_without_a_gpu(lib):
    """Workspace planning is host arithmetic: sizes grow with the problem and
    the split contraction adds partials only where its rule splits (few tiles)."""
    small = lora.lora_workspace_size(lora.make_shape(256, 3072, 3072, 16, 2.0), lora.LORA_FWD_BWD)
    big = lora.lora_workspace_size(lora.make_shape(4096, 3072, 3072, 16, 2.0), lora.LORA_FWD_BWD)
    # T = 256: 1 x 6 output tiles (< 76 pairs), so each contraction splits (at least in two) and
    # needs fp32 partials of 2 x 256 x 3072 x 4 bytes or more; T = 4096: 16 x 6 = 96 tiles, no
    # partials, only the rank-r scratch (T x pad8(r) bf16 per buffer, a few MB)
    assert small >= 2 * 256 * 3072 * 4
    assert 0 < big < 16 * 2 ** 20


def test_stack_ckpt_workspace_covers_the_largest_layer(lib):
    st = lora.make_shape(1024, 3072, 3072, 16, 2.0)
    layer = [lora.make_proj(st) for _ in range(3)]
    one = lora.lora_stack_workspace_size(layer, lora.LORA_FWD_BWD)
    n = lora.lora_stack_ckpt_workspace_size([layer, layer, layer])
    assert n >= one + 3 * 1024 * 16 * 2  # a step's workspace plus one layer's su scratch
    n_bad = ctypes.c_size_t(0)
    arr = (lora.lora_proj * 3)(*layer)
    assert lib.lora_stack_ckpt_workspace_size(arr, 0, 3, ctypes.byref(n_bad)) == lora.LORA_EINVAL
    assert lib.lora_stack_ckpt_workspace_size(arr, 1, 65, ctypes.byref(n_bad)) == lora.LORA_EINVAL


def test_q4_weights_validated_on_the_host(lib):
    st = lora.make_shape(128, 128, 256, 8, 2.0)  # d_in not a multiple of 256
    ws = ctypes.c_void_p(256)
    wq = lora.make_q4(256, 256)
    rc = lib.lora_linear_fwd_q4(ctypes.byref(st), 256, ctypes.byref(wq), 256, 256, 256, None, ws, 1 << 30, None)
    assert rc in (lora.LORA_EINVAL, lora.LORA_EDEVICE, lora.LORA_ECUDA)
    half = lora.make_q4(256, None)
    st = lora.make_shape(128, 256, 256, 8, 2.0)
    rc = lib.lora_linear_fwd_q4(ctypes.byref(st), 256, ctypes.byref(half), 256, 256, 256, None, ws, 1 << 30, None)
    assert rc == lora.LORA_ENULL


def test_ce_and_topk_sizes_and_arguments(lib):
    a = lora.make_ce_args(2048, 3072, 128256, 256, 256, 256, 256, topk=256, ld_topk=500, k=500)
    n = lora.lora_ce_workspace_size(a)
    # worst case |T_set| = T, |J| = V: the fp32 logits alone take T x V x 4 bytes
    assert n >= 2048 * 128256 * 4
    n_bad = ctypes.c_size_t(0)
    bad = lora.make_ce_args(2048, 3070, 128256, 256, 256, 256, 256)  # d not a multiple of 8
    assert lib.lora_ce_workspace_size(ctypes.byref(bad), ctypes.byref(n_bad)) == lora.LORA_EINVAL
    bad = lora.make_ce_args(2048, 3072, 128256, 256, 256, 256, 256, topk=256, ld_topk=10, k=11)  # k > ld_topk
    assert lib.lora_ce_workspace_size(ctypes.byref(bad), ctypes.byref(n_bad)) == lora.LORA_EINVAL
    bad = lora.make_ce_args(2048, 3072, 128256, None, 256, 256, 256)  # h missing
    assert lib.lora_ce_workspace_size(ctypes.byref(bad), ctypes.byref(n_bad)) == lora.LORA_ENULL
    t = lora.lora_topk_workspace_size(128256, 3072, 500)
    assert t >= 128256 * 3072 * 2 + 512 * 128256 * 4  # normalised rows plus one chunk of similarities
    for V, d, k in ((100, 12, 5), (100, 16, 101), (5000, 16, 1025), (0, 16, 1)):
        assert lib.lora_topk_workspace_size(V, d, k, ctypes.byref(n_bad)) == lora.LORA_EINVAL


def test_topk_workspace_switches_to_the_sampled_layout(lib):
    """Rows of at least 32768 tokens take the sampled selection, whose
    candidate lists (4096 slots of 8 bytes per row) live in the workspace;
    shorter rows only need the normalised rows and one 512-row chunk of
    similarities."""
    d, k = 256, 100
    below = lora.lora_topk_workspace_size(32767, d, k)
    at = lora.lora_topk_workspace_size(32768, d, k)
    assert below < 32767 * d * 2 + 512 * 32768 * 4 + 400 * 2 ** 20
    assert at >= 32768 * 4096 * 8 + 32768 * d * 2
    assert at - below > 32768 * 4096 * 8 - 2 ** 20


def test_ce_full_vocabulary_reads_the_embedding_in_place(lib):
    """Without a top-k table J is the whole vocabulary and E is used where it
    lies: the workspace carries no gathered copy of it (V x d bf16)."""
    T, d, V = 256, 1024, 50000
    full = lora.lora_ce_workspace_size(lora.make_ce_args(T, d, V, 256, 256, 256, 256))
    reduced = lora.lora_ce_workspace_size(lora.make_ce_args(T, d, V, 256, 256, 256, 256, topk=256, ld_topk=8, k=8))
    assert reduced - full >= V * d * 2 - 2 ** 16


def test_forward_and_backward_plan_their_splits_for_the_contractions_sms(lib):
    """A forward-and-backward call gives the side stream some SMs, so its
    contractions plan their splits for fewer CTA pairs than a forward-only
    call; both still size their own partials (few output tiles split)."""
    st = lora.make_shape(256, 3072, 8192, 16, 2.0)
    fwd = lora.lora_workspace_size(st, lora.LORA_FWD)
    both = lora.lora_workspace_size(st, lora.LORA_FWD_BWD)
    assert fwd > 0 and both > fwd


def test_forward_and_backward_workspace_covers_every_call_of_the_shape(lib):
    """The size a forward-and-backward query reports from the shape alone
    covers a forward or a backward call of that shape, with bf16 or 4-bit
    weights: the partials of split contractions are sized for the pairs a
    contraction gets beside the side stream (whose width depends on the
    weight kind and, for few output tiles, on the cluster split), and on all
    pairs."""
    # (the first three violated it when the partials were sized for the side stream's pairs alone)
    shapes = [(128, 2048, 8192, 16), (256, 2048, 8192, 16), (128, 4096, 6144, 64), (200, 768, 1024, 24),
              (512, 3072, 3072, 16), (256, 3072, 8192, 16), (256, 8192, 3072, 16), (2048, 3072, 3072, 16),
              (256, 1024, 4096, 128), (1000, 2048, 256, 64), (64, 512, 768, 8)]
    fake_q4 = lora.lora_q4_weight(256, 512)  # sizes only: the pointers are never read
    for T, K, N, r in shapes:
        st = lora.make_shape(T, K, N, r, 2.0)
        both = lora.lora_workspace_size(st, lora.LORA_FWD_BWD)
        for mode in (lora.LORA_FWD, lora.LORA_BWD, lora.LORA_FWD_BWD):
            assert lora.lora_workspace_size(st, mode) <= both, (T, K, N, r, mode)
            if K % 256 == 0:
                q4 = lora.lora_stack_workspace_size([lora.make_proj(st, Wq=fake_q4)], mode)
                if mode != lora.LORA_FWD_BWD:
                    assert q4 <= both, (T, K, N, r, mode, q4, both)


def test_last_error_follows_the_threads_latest_call(lib):
    """lora_last_error repeats the code of the calling thread's latest call,
    successes included, and is per thread."""
    import threading
    n = ctypes.c_size_t(0)
    assert lib.lora_workspace_size(None, 1, ctypes.byref(n)) == lora.LORA_ENULL
    assert lora.lora_last_error() == lora.LORA_ENULL
    st = lora.make_shape(128, 256, 256, 8, 2.0)
    assert lib.lora_workspace_size(ctypes.byref(st), 9, ctypes.byref(n)) == lora.LORA_EINVAL
    assert lora.lora_last_error() == lora.LORA_EINVAL
    seen = []
    t = threading.Thread(target=lambda: seen.append(lora.lora_last_error()))
    t.start()
    t.join()
    assert seen == [lora.LORA_OK], "another thread's calls do not show"
    assert lib.lora_workspace_size(ctypes.byref(st), 1, ctypes.byref(n)) == lora.LORA_OK
    assert lora.lora_last_error() == lora.LORA_OK
    lora.lora_strerror(-1)  # does not record
    assert lora.lora_last_error() == lora.LORA_OK


def test_frozen_projection_plans_no_rank_work(lib):
    """Rank 0 is a frozen projection: no adapter, so its workspace holds no
    rank-r scratch, only the tile counters (and split partials where its
    contraction splits); a negative rank is rejected."""
    big = lora.make_shape(4096, 3072, 3072, 0, 1.0)  # 96 tiles: no split
    assert lora.lora_workspace_size(big, lora.LORA_FWD_BWD) <= 4096
    adapted = lora.lora_workspace_size(lora.make_shape(4096, 3072, 3072, 16, 2.0), lora.LORA_FWD_BWD)
    assert adapted > 4 * 4096 * 16 * 2
    n = ctypes.c_size_t(0)
    bad = lora.make_shape(128, 256, 256, -1, 1.0)
    assert lib.lora_workspace_size(ctypes.byref(bad), 3, ctypes.byref(n)) == lora.LORA_EINVAL
    # a layer adapting q and v only: the frozen projections add nothing beyond their split partials
    layer = [lora.make_proj(lora.make_shape(4096, 3072, 3072, r, 2.0)) for r in (16, 0, 16, 0)]
    two = [lora.make_proj(lora.make_shape(4096, 3072, 3072, 16, 2.0)) for _ in range(2)]
    assert lora.lora_stack_workspace_size(layer, lora.LORA_FWD_BWD) == lora.lora_stack_workspace_size(
        two, lora.LORA_FWD_BWD)
