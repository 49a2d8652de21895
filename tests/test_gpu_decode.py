"""GPU parity of the Flash Decode kernels through the C ABI, in both forms: split kernel +
merge kernel, and the single persistent kernel whose clusters of CTAs walk the (batch, kv
head) pairs and merge their partials over distributed shared memory."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import assert_parity, o_to_f64, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def loom():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    return m


@pytest.fixture(autouse=True, params=[(0, 1), (1, 1), (1, 2), (1, 0), (2, 1), (3, 1)],
                ids=["model_form", "split_merge", "split_merge_tc_per_split", "split_merge_cuda_core",
                     "persistent", "cluster"])
def form(request, loom):
    """Every test runs with the model's choice of form and with each form forced: split
    kernel + merge (its split kernel on the tensor cores where it takes the shape --
    persistent CTAs, or one CTA per split -- and on the CUDA cores), persistent split
    kernel + merge, and the single-kernel cluster form (at the model's cluster size)."""
    f, tc = request.param
    loom.loom_debug_decode_form(f)
    loom.loom_debug_decode_tensor_cores(tc)
    yield f
    loom.loom_debug_decode_form(0)
    loom.loom_debug_decode_tensor_cores(1)


def _expect_form(loom, form, B, Hq, Hkv, Skv, D, splits):
    used, cs = loom.loom_attn_decode_form(B, Hq, Hkv, Skv, D, splits)
    if form:
        assert used == form
    elif splits:  # a split count the caller fixes runs the split + merge form
        assert used == loom.DECODE_SPLIT_MERGE
    if used == loom.DECODE_CLUSTER:
        s = splits or loom.loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D)
        assert cs >= 1 and s % cs == 0


def _inputs(seed, B, Hq, Hkv, Skv, D):
    return (synth.bf16_normal(seed, synth.STREAM_Q, (B, Hq, 1, D)),
            synth.bf16_normal(seed, synth.STREAM_K, (B, Hkv, Skv, D)),
            synth.bf16_normal(seed, synth.STREAM_V, (B, Hkv, Skv, D)))


def _run(loom, q, k, v, lens, num_splits, workspace=None):
    import torch
    sl = None if lens is None else torch.from_numpy(np.asarray(lens, np.int32)).cuda()
    o, lse = loom.loom_attn_decode(to_dev(q), to_dev(k), to_dev(v), sl, num_splits=num_splits,
                                   workspace=workspace, return_lse=True)
    loom.loom_attn_check_error()
    return o, lse


def test_batched_decode_config(loom, form):
    # B=16, Hq=32, Hkv=8, Skv=8192, lengths U[4096, 8192] (stream 3), D=128, 16 splits
    B, Hq, Hkv, Skv, D = 16, 32, 8, 8192, 128
    _expect_form(loom, form, B, Hq, Hkv, Skv, D, 16)
    q, k, v = _inputs(0, B, Hq, Hkv, Skv, D)
    lens = synth.decode_lengths(0, B, 4096, 8192)
    o, lse = _run(loom, q, k, v, lens, 16)
    o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=lens)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, "batched decode")


@pytest.mark.slow
def test_long_context_decode_config(loom, form):
    # B=1, Hq=32, Hkv=8, Skv=131072, D=128, model-chosen splits (>= one wave of CTAs)
    B, Hq, Hkv, Skv, D = 1, 32, 8, 131072, 128
    _expect_form(loom, form, B, Hq, Hkv, Skv, D, 0)
    q, k, v = _inputs(0, B, Hq, Hkv, Skv, D)
    splits = loom.loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D)
    assert splits * Hkv >= 148
    o, lse = _run(loom, q, k, v, None, 0)
    o_ref, lse_ref = oracle.attention(q, k, v)
    assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, "long decode")


@pytest.mark.parametrize("splits,clusters", [(16, (1, 2, 4, 8, 16)), (12, (3, 6, 12)), (5, (5,)), (38, (2, 19))])
def test_every_cluster_size(loom, form, splits, clusters):
    """The cluster form with each cluster size pinned (CTA r takes splits r, r + cs, ...):
    sequences of 0 .. Skv keys over a batch that leaves clusters several units each."""
    import torch
    if form != 3:
        pytest.skip("cluster sizes are pinned under the forced cluster form")
    B, Hq, Hkv, Skv, D = 9, 16, 4, 4000, 128
    q, k, v = _inputs(splits, B, Hq, Hkv, Skv, D)
    lens = np.array([4000, 0, 1, 63, 65, 1000, 3999, 2048, 777], np.int32)
    o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=lens)
    for cs in clusters:
        loom.loom_debug_decode_form(3, cs)
        used, got = loom.loom_attn_decode_form(B, Hq, Hkv, Skv, D, splits)
        assert used == loom.DECODE_CLUSTER
        if splits % cs == 0 and cs <= 16:
            assert got == cs
        else:
            assert got != cs
        o, lse = _run(loom, q, k, v, lens, splits)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"splits={splits} cluster={cs}")
    loom.loom_debug_decode_form(3, 0)


@pytest.mark.parametrize("D", [64, 128])
def test_edge_lengths(loom, form, D):
    # empty sequence, single key, chunk-1, chunk+1, full; splits that leave whole empty
    # CTAs in a cluster (16 splits of 300 keys: chunks of 64, splits 5..15 empty)
    B, Hq, Hkv, Skv = 6, 4, 2, 300
    q, k, v = _inputs(3, B, Hq, Hkv, Skv, D)
    lens = np.array([0, 1, 63, 65, 129, 300], np.int32)
    for splits in (1, 2, 3, 7, 16, 64):
        _expect_form(loom, form, B, Hq, Hkv, Skv, D, splits)
        o, lse = _run(loom, q, k, v, lens, splits)
        o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=lens)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"D={D} splits={splits}")


@pytest.mark.parametrize("D", [64, 128])
def test_cache_past_length_is_never_used(loom, form, D):
    """Keys and values past a sequence's length may hold anything (NaN here): the output
    equals the oracle's on a finite cache, in every form (the tensor-core split kernel
    zeroes the V rows of a ragged last stage before P.V)."""
    B, Hq, Hkv, Skv = 3, 16, 4, 400
    q, k, v = _inputs(21, B, Hq, Hkv, Skv, D)
    lens = np.array([1, 257, 390], np.int32)
    kp, vp = k.copy(), v.copy()
    for b, n in enumerate(lens):
        kp[b, :, n:] = 0x7FC0  # bf16 quiet NaN
        vp[b, :, n:] = 0x7FC0
    o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=lens)
    for splits in (1, 3, 7):
        o, lse = _run(loom, q, kp, vp, lens, splits)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"D={D} splits={splits}")


@pytest.mark.parametrize("Hq,Hkv", [(1, 1), (3, 1), (8, 8), (16, 2), (32, 1), (12, 4), (64, 2)])
def test_group_sizes(loom, form, Hq, Hkv):
    B, Skv, D = 2, 777, 128
    q, k, v = _inputs(Hq + Hkv, B, Hq, Hkv, Skv, D)
    for splits in (1, 5, 13):
        _expect_form(loom, form, B, Hq, Hkv, Skv, D, splits)
        o, lse = _run(loom, q, k, v, None, splits)
        o_ref, lse_ref = oracle.attention(q, k, v)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"Hq={Hq} Hkv={Hkv} splits={splits}")


def test_partials_match_oracle_split_form(loom, form):
    """The workspace holds the per-split partial (O_i, lse_i) of the Flash Decode form
    (split + merge kernels; the cluster form keeps its partials in shared memory)."""
    import torch
    loom.loom_debug_decode_form(1)
    B, Hq, Hkv, Skv, D, S = 2, 8, 2, 1000, 128, 5
    q, k, v = _inputs(9, B, Hq, Hkv, Skv, D)
    lens = np.array([1000, 333], np.int32)
    nbytes = loom.loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, S)
    ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    o, lse = _run(loom, q, k, v, lens, S, workspace=ws)
    _, _, o_part_ref, lse_part_ref = oracle.decode_split_merge(q, k, v, num_splits=S, seqlens_k=lens)
    n = B * Hq * S
    opart = ws[: n * D * 4].view(torch.float32).cpu().numpy().astype(np.float64).reshape(B, Hq, S, D)
    off = (n * D * 4 + 255) // 256 * 256
    lpart = ws[off: off + n * 4].view(torch.float32).cpu().numpy().astype(np.float64).reshape(B, Hq, S)
    assert_parity(opart, o_part_ref, lpart, lse_part_ref, "partials")


def test_item_counter_first_call_static_then_armed(loom, form):
    """The persistent tensor-core split kernel takes items from a counter in the
    workspace's last 256 bytes.  A workspace never used (all bytes 0xFF) is dealt
    statically; the merge kernel then arms the counter, and the next call, dealt on
    demand, gives the same bits (each item's arithmetic does not depend on its CTA)."""
    import torch
    B, Hq, Hkv, Skv, D, S = 4, 32, 8, 3000, 128, 7
    q, k, v = (to_dev(x) for x in _inputs(17, B, Hq, Hkv, Skv, D))
    sl = torch.tensor([3000, 1, 2047, 700], dtype=torch.int32, device="cuda")
    nbytes = loom.loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, S)
    ws = torch.full((nbytes,), 0xFF, dtype=torch.uint8, device="cuda")
    o1, l1 = loom.loom_attn_decode(q, k, v, sl, num_splits=S, workspace=ws, return_lse=True)
    loom.loom_attn_check_error()
    word = int(ws[nbytes - 256: nbytes - 248].cpu().view(torch.int64)[0]) & 0xFFFFFFFFFFFFFFFF
    if form in (0, 1):  # the split + merge form's merge kernel arms the counter
        assert word == 0x7FBADC0D << 32
    o2, l2 = loom.loom_attn_decode(q, k, v, sl, num_splits=S, workspace=ws, return_lse=True)
    loom.loom_attn_check_error()
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(l1, l2)
    o_ref, lse_ref = oracle.attention(*(_inputs(17, B, Hq, Hkv, Skv, D)), seqlens_k=sl.cpu().numpy())
    assert_parity(o_to_f64(o2), o_ref, l2.cpu().numpy(), lse_ref, "armed counter")


def test_more_sequences_than_the_length_sort_takes(loom, form):
    """Above 256 sequences the persistent kernels take the sequences in index order instead
    of sorting them by length; lengths 0..200 with empty sequences and empty splits."""
    B, Hq, Hkv, Skv, D = 300, 4, 1, 200, 64
    q, k, v = _inputs(23, B, Hq, Hkv, Skv, D)
    lens = np.random.default_rng(23).integers(0, Skv + 1, size=B).astype(np.int32)
    lens[:3] = [0, 200, 1]
    o_ref, lse_ref = oracle.attention(q, k, v, seqlens_k=lens)
    for splits in (1, 3):
        o, lse = _run(loom, q, k, v, lens, splits)
        assert_parity(o_to_f64(o), o_ref, lse.cpu().numpy(), lse_ref, f"B=300 splits={splits}")


def test_workspace_and_argument_errors(loom):
    import torch
    B, Hq, Hkv, Skv, D = 1, 4, 2, 256, 128
    q, k, v = _inputs(1, B, Hq, Hkv, Skv, D)
    small = torch.empty(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(loom.LoomError) as e:
        loom.loom_attn_decode(to_dev(q), to_dev(k), to_dev(v), None, workspace=small, num_splits=4)
    assert e.value.status == 4
    with pytest.raises(loom.LoomError) as e:
        loom.loom_attn_decode(to_dev(q), to_dev(k), to_dev(v), None, num_splits=2000)
    assert e.value.status == 2


def test_cluster_form_is_deterministic(loom, form):
    """The cluster form reads the splits in a fixed order: repeated calls agree bit for bit."""
    import torch
    B, Hq, Hkv, Skv, D = 3, 16, 4, 5000, 128
    q, k, v = (to_dev(x) for x in _inputs(13, B, Hq, Hkv, Skv, D))
    sl = torch.tensor([5000, 4097, 100], dtype=torch.int32, device="cuda")
    outs = [loom.loom_attn_decode(q, k, v, sl, num_splits=11, return_lse=True) for _ in range(3)]
    loom.loom_attn_check_error()
    for o, lse in outs[1:]:
        assert torch.equal(o.view(torch.int16), outs[0][0].view(torch.int16))
        assert torch.equal(lse, outs[0][1])
