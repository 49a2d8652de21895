"""GPU parity of Flash Decode over a paged KV cache (through the C ABI) against the fp64
oracle (``oracle.decode_paged``), plus bit equality with the contiguous kernels when the
pages are laid out in order (the two load the same rows into the same places)."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import assert_parity, o_to_f64, to_dev

pytestmark = pytest.mark.gpu

NAN_BF16 = 0x7FC0


@pytest.fixture(scope="module")
def loom():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    yield m
    m.loom_debug_inject(0)
    m.loom_debug_set_timeout_ns(0)


@pytest.fixture(autouse=True, params=[(1, 1), (1, 0), (2, 1), (3, 1)],
                ids=["split_merge", "split_merge_cuda_core", "persistent", "cluster"])
def form(request, loom):
    """Every test runs with each Flash Decode form forced: split kernel + merge (the split
    kernel on the tensor cores -- persistent CTAs copying each stage page by page -- and
    on the CUDA cores), persistent split kernel + merge, and the single-kernel cluster
    form (the model's cluster size)."""
    f, tc = request.param
    loom.loom_debug_decode_form(f)
    loom.loom_debug_decode_tensor_cores(tc)
    yield f
    loom.loom_debug_decode_form(0)
    loom.loom_debug_decode_tensor_cores(1)


def paged_case(seed, B, Hq, Hkv, P, lens, D, spare=5, poison=True, shuffle=True):
    """Pages dealt to the sequences in a (shuffled) order; rows past each sequence's end
    and the spare pages hold NaN, table entries past a sequence's last page hold -1."""
    lens = np.asarray(lens, dtype=np.int32)
    need = [(int(n) + P - 1) // P for n in lens]
    max_pages = max(1, max(need)) + 1
    npages = sum(need) + spare
    kc = synth.bf16_normal(seed, synth.STREAM_K, (npages, P, Hkv, D))
    vc = synth.bf16_normal(seed, synth.STREAM_V, (npages, P, Hkv, D))
    q = synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, 1, D))
    order = np.random.default_rng(seed).permutation(npages) if shuffle else np.arange(npages)
    table = np.full((B, max_pages), -1, dtype=np.int32)
    i = 0
    for b in range(B):
        table[b, :need[b]] = order[i:i + need[b]]
        i += need[b]
        if poison and need[b]:
            tail = int(lens[b]) - (need[b] - 1) * P
            kc[table[b, need[b] - 1], tail:] = NAN_BF16
            vc[table[b, need[b] - 1], tail:] = NAN_BF16
    if poison:
        for p in order[i:]:
            kc[p] = NAN_BF16
            vc[p] = NAN_BF16
    return q, kc, vc, table, lens


def run_paged(loom, q, kc, vc, table, lens, splits=0, layout="nhd"):
    """kc / vc are token-major [pages, page_size, Hkv, D]; layout "hnd" hands the kernel
    the same pages head-major [pages, Hkv, page_size, D]."""
    import torch
    if layout == "hnd":
        kc = np.ascontiguousarray(kc.transpose(0, 2, 1, 3))
        vc = np.ascontiguousarray(vc.transpose(0, 2, 1, 3))
    o, lse = loom.loom_attn_decode_paged(to_dev(q), to_dev(kc), to_dev(vc),
                                         torch.from_numpy(table).cuda(), torch.from_numpy(lens).cuda(),
                                         num_splits=splits, return_lse=True, layout=layout)
    loom.loom_attn_check_error()
    return o, lse


LAYOUTS = pytest.mark.parametrize("layout", ["nhd", "hnd"])


@LAYOUTS
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("P", [8, 16, 32, 64, 128, 256])
def test_page_sizes(loom, P, D, layout):
    B, Hq, Hkv = 4, 8, 2
    lens = [1, P - 1, 3 * P + 1, 700]
    q, kc, vc, table, sl = paged_case(P + D, B, Hq, Hkv, P, lens, D)
    for splits in (1, 0, 7):
        o, lse = run_paged(loom, q, kc, vc, table, sl, splits, layout)
        o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
        assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, f"P={P} D={D} splits={splits}")


@LAYOUTS
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("P", [64, 128, 256])
def test_splits_starting_mid_page(loom, P, D, layout):
    """Chunks of 192 keys (900 keys in 5 splits): splits start on odd multiples of 64, so
    a stage (128 keys at D = 64) runs across a page boundary; every copy must stay within
    its page."""
    B, Hq, Hkv = 3, 8, 2
    lens = [900, 2 * P + 192, 191]
    q, kc, vc, table, sl = paged_case(P + 3 * D, B, Hq, Hkv, P, lens, D)
    for splits in (5, 3):
        o, lse = run_paged(loom, q, kc, vc, table, sl, splits, layout)
        o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
        assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, f"P={P} D={D} splits={splits}")


@pytest.mark.parametrize("G", [1, 2, 4, 8, 16])
def test_gqa_groups(loom, G):
    B, Hkv, P, D = 2, 2, 16, 128
    q, kc, vc, table, sl = paged_case(G, B, G * Hkv, Hkv, P, [515, 64], D)
    o, lse = run_paged(loom, q, kc, vc, table, sl)
    o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
    assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, f"G={G}")


@LAYOUTS
def test_edge_lengths_and_empty(loom, layout):
    B, Hq, Hkv, P, D = 8, 4, 1, 16, 64
    lens = [0, 1, 15, 16, 17, 63, 64, 65]
    q, kc, vc, table, sl = paged_case(4, B, Hq, Hkv, P, lens, D)
    for splits in (1, 3, 64):
        o, lse = run_paged(loom, q, kc, vc, table, sl, splits, layout)
        o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
        assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, f"edges splits={splits}")
        assert np.all(o_to_f64(o)[0] == 0.0) and np.all(np.isneginf(lse.cpu().numpy()[0]))


@LAYOUTS
@pytest.mark.parametrize("P", [16, 64])
def test_in_order_pages_match_contiguous_kernel_bitwise(loom, P, layout):
    """With page j of sequence b at physical index b * pages + j, the paged and the
    contiguous kernels of each form (and of either split kernel) copy identical rows to
    identical places: outputs are equal bit for bit."""
    import torch
    B, Hq, Hkv, S, D = 3, 16, 4, 1024, 128
    k = synth.bf16_normal(8, synth.STREAM_K, (B, Hkv, S, D))
    v = synth.bf16_normal(8, synth.STREAM_V, (B, Hkv, S, D))
    q = synth.bf16_normal(8, synth.STREAM_Q, (B, Hq, 1, D))
    npg = S // P
    kc = k.reshape(B, Hkv, npg, P, D).transpose(0, 2, 3, 1, 4).reshape(B * npg, P, Hkv, D).copy()
    vc = v.reshape(B, Hkv, npg, P, D).transpose(0, 2, 3, 1, 4).reshape(B * npg, P, Hkv, D).copy()
    table = np.arange(B * npg, dtype=np.int32).reshape(B, npg)
    lens = np.array([S, 777, 64], dtype=np.int32)
    for splits in (1, 5):
        o1, l1 = run_paged(loom, q, kc, vc, table, lens, splits, layout)
        o2, l2 = loom.loom_attn_decode(to_dev(q), to_dev(k), to_dev(v), torch.from_numpy(lens).cuda(),
                                       num_splits=splits, return_lse=True)
        loom.loom_attn_check_error()
        assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
        assert torch.equal(l1, l2)


@LAYOUTS
@pytest.mark.parametrize("P", [16, 64])
def test_batched_serving_shape(loom, form, P, layout):
    """The batched decode shape (B=16, Hq=32, Hkv=8, D=128, lengths U[4096, 8192]) paged,
    pages shuffled, model-chosen splits."""
    B, Hq, Hkv, D = 16, 32, 8, 128
    lens = synth.decode_lengths(0, B, 4096, 8192)
    q, kc, vc, table, sl = paged_case(0, B, Hq, Hkv, P, lens, D, spare=0, poison=False)
    o, lse = run_paged(loom, q, kc, vc, table, sl, 16, layout)
    assert loom.loom_attn_decode_form(B, Hq, Hkv, table.shape[1] * P, D, 16, paged=True)[0] == form
    o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
    assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, f"batched paged P={P} {layout}")


@LAYOUTS
def test_out_of_range_page_reads_zeros_without_fault(loom, layout):
    """A table entry outside the cache (a caller error) is bounded by the copy engine: the
    keys it names read as zeros, so the call completes and reports no error."""
    import torch
    B, Hq, Hkv, P, D = 1, 4, 1, 16, 64
    q, kc, vc, table, sl = paged_case(12, B, Hq, Hkv, P, [48], D, poison=False)
    bad = table.copy()
    bad[0, 1] = kc.shape[0] + 1000
    o, lse = run_paged(loom, q, kc, vc, bad, sl, 1, layout)
    kz, vz = kc.copy(), vc.copy()
    zero_page = np.zeros((1, P, Hkv, D), np.uint16)
    kz = np.concatenate([kz, zero_page])
    vz = np.concatenate([vz, zero_page])
    t2 = table.copy()
    t2[0, 1] = kz.shape[0] - 1
    o_ref, lse_ref = oracle.decode_paged(q, kz, vz, t2, sl, page_size=P)
    assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, "out-of-range page")


def test_timeout_is_reported_and_context_survives(loom):
    import torch
    B, Hq, Hkv, P, D = 1, 4, 1, 16, 128
    q, kc, vc, table, sl = paged_case(31, B, Hq, Hkv, P, [2048], D)
    args = (to_dev(q), to_dev(kc), to_dev(vc), torch.from_numpy(table).cuda(), torch.from_numpy(sl).cuda())
    loom.loom_attn_check_error()
    loom.loom_debug_set_timeout_ns(50_000_000)
    try:
        loom.loom_debug_inject(1)
        loom.loom_attn_decode_paged(*args, num_splits=1)
        with pytest.raises(loom.LoomError) as e:
            loom.loom_attn_check_error()
        assert e.value.status == 6
    finally:
        loom.loom_debug_inject(0)
        loom.loom_debug_set_timeout_ns(0)
    o, lse = loom.loom_attn_decode_paged(*args, num_splits=1, return_lse=True)
    loom.loom_attn_check_error()
    o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
    assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, "after timeout")


def test_large_pages_and_long_table(loom):
    """512-key pages (eight 64-key copies per page) and a 40-entry block table."""
    B, Hq, Hkv, P, D = 3, 8, 2, 512, 128
    lens = [20000, 513, 9000]
    q, kc, vc, table, sl = paged_case(41, B, Hq, Hkv, P, lens, D, spare=2)
    for splits in (0, 3):
        o, lse = run_paged(loom, q, kc, vc, table, sl, splits)
        o_ref, lse_ref = oracle.decode_paged(q, kc, vc, table, sl, page_size=P)
        assert_parity(o_to_f64(o)[:, :, 0], o_ref, lse.cpu().numpy(), lse_ref, f"P=512 splits={splits}")
