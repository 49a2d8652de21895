"""The analytic schedule model (Sec. 2.6, Eq. 5-9; architecture description of Sec. 2.7),
checked through the C ABI on the CPU against properties that hold whatever the numbers in
the architecture description are: Eq. 6's limiting cases, the capacity constraints of
Eq. 8, the argmin of Eq. 9 recomputed by brute force over every candidate, the one-wave
rule of the split decode, and the rooflines no modeled time may beat."""
import itertools
import math

import pytest

PEAK_TFLOPS = 1910.3   # measured dense bf16 (cuBLAS) on GB300
PEAK_GBS = 6783.5      # measured HBM copy bandwidth on GB300
NUM_SMS = 152


@pytest.fixture(scope="module")
def loom():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_29219_gb300 as m
    return m


# ------------------------------------------------------------------ Eq. 6
@pytest.mark.parametrize("l,m,s", [(1.0, 2.0, 3.0), (5.0, 1.0, 1.0), (0.5, 4.0, 0.25), (2.0, 2.0, 2.0)])
def test_heg_pipe_limits(loom, l, m, s):
    seq = loom.loom_model_heg_pipe(l, m, s, 0, 0)
    full = loom.loom_model_heg_pipe(l, m, s, 1, 1)
    assert seq == pytest.approx(l + m + s)        # no boundary open: the stages run in turn
    assert full == pytest.approx(max(l, m, s))    # both open: the slowest stage sets the pace
    for b in itertools.product((0, 1), repeat=2):
        t = loom.loom_model_heg_pipe(l, m, s, *b)
        assert full - 1e-12 <= t <= seq + 1e-12   # opening a boundary never slows the pipe
    # opening one boundary hides exactly the stage on its other side behind its neighbour
    assert loom.loom_model_heg_pipe(l, m, s, 1, 0) == pytest.approx(max(l, m + s))
    assert loom.loom_model_heg_pipe(l, m, s, 0, 1) == pytest.approx(max(l + m, s))


# ------------------------------------------------------------------ Eq. 8 / 9, prefill
@pytest.mark.parametrize("D", [64, 128])
def test_fwd_plan_within_capacities(loom, D):
    p = loom.loom_model_fwd_plan(D)
    assert p["smem_bytes"] <= 227 * 1024          # dynamic shared memory per CTA
    assert p["tmem_cols"] <= 512                  # TMEM columns per SM
    assert p["bm"] in (64, 128)
    assert p["bn"] % 16 == 0 and 16 <= p["bn"] <= 256
    assert p["kv_slots"] >= 2
    assert p["design"] in (1, 2, 3, 4)
    assert p["t_iter_ns"] > 0


@pytest.mark.parametrize("D", [64, 128])
def test_fwd_plan_is_argmin_over_designs(loom, D):
    chosen = loom.loom_model_fwd_plan(D)
    variants = {d: loom.loom_model_fwd_plan_variant(D, d) for d in (1, 2, 3, 4)}
    feasible = {d: v for d, v in variants.items() if v is not None}
    assert chosen["design"] in feasible
    best = min(v["t_iter_ns"] / v["bn"] for v in feasible.values())
    assert chosen["t_iter_ns"] / chosen["bn"] == pytest.approx(best)
    for v in feasible.values():                   # every candidate obeys Eq. 8
        assert v["smem_bytes"] <= 227 * 1024 and v["tmem_cols"] <= 512


@pytest.mark.parametrize("D", [64, 128])
def test_fwd_plan_ranks_the_measured_best_design_first(loom, D):
    # GB300 same-box measurements (warp-wide MMA issue): design 2 leads at both head
    # dimensions (D=128: 1481 vs 1370 TFLOP/s for design 1; D=64 (B1 H64 S8192 causal): 1004
    # vs 876 for design 4, 874 for design 3 and 813 for design 1), and at D=64 designs 3
    # and 4 measure ahead of design 1 (cost per key: t_iter / bn)
    t = {d: loom.loom_model_fwd_plan_variant(D, d) for d in (1, 2, 3, 4)}
    assert loom.loom_model_fwd_plan(D)["design"] == 2
    if D == 64:
        cost = {d: t[d]["t_iter_ns"] / t[d]["bn"] for d in (1, 2, 3, 4)}
        assert cost[2] < cost[3] < cost[1]
        assert cost[2] < cost[4] < cost[1]


def test_three_s_buffers_do_not_fit_at_d128(loom):
    # 3 S buffers of 128 columns + 2 O tiles of 128 columns = 640 > 512 TMEM columns;
    # three tiles of 96-key S and 128-column O: 3 x 224 = 672 > 512
    assert loom.loom_model_fwd_plan_variant(128, 3) is None
    assert loom.loom_model_fwd_plan_variant(64, 3) is not None
    assert loom.loom_model_fwd_plan_variant(128, 4) is None
    p4 = loom.loom_model_fwd_plan_variant(64, 4)
    assert p4 is not None and p4["q_tiles"] == 3 and p4["bn"] == 96 and p4["tmem_cols"] == 480


@pytest.mark.parametrize("B,Hq,S,D,causal", [(4, 32, 2048, 128, 0), (4, 32, 2048, 128, 1),
                                            (1, 32, 8192, 128, 1), (1, 64, 8192, 64, 1),
                                            (1, 2, 128, 64, 0)])
def test_fwd_time_not_below_tensor_roofline(loom, B, Hq, S, D, causal):
    t = loom.loom_model_fwd_time_us(B, Hq, S, S, D, causal)
    pairs = S * (S + 1) / 2 if causal else S * S
    flops = 4.0 * B * Hq * D * pairs
    assert t > 0
    assert t * 1e-6 >= flops / (PEAK_TFLOPS * 1e12) * 0.999


def test_fwd_time_scales_with_work(loom):
    t1 = loom.loom_model_fwd_time_us(8, 32, 4096, 4096, 128, 0)
    t2 = loom.loom_model_fwd_time_us(16, 32, 4096, 4096, 128, 0)
    assert 1.8 <= t2 / t1 <= 2.2                  # many waves: time ~ work
    tc = loom.loom_model_fwd_time_us(8, 32, 4096, 4096, 128, 1)
    assert tc < t1                                # the causal triangle is cheaper


# ------------------------------------------------------------------ decode
DECODE_SHAPES = [(16, 32, 8, 8192, 128), (1, 32, 8, 131072, 128), (1, 8, 8, 4096, 64),
                 (4, 16, 2, 30000, 128), (2, 4, 4, 64, 128)]


def _decode_candidates(loom, B, Hq, Hkv, Skv, D):
    """Modeled time of every (form, split count) candidate: the split + merge form (its
    split kernel on the tensor cores where that kernel takes the shape, at most 32 query
    heads per kv head; elsewhere also the CUDA-core persistent split + merge form) for
    every split count, the
    cluster form for every split count and cluster size dividing it, with the CTAs and
    clusters they are priced at.  Form order for ties: split + merge (0), persistent (1),
    cluster (2)."""
    cands = []
    G = Hq // Hkv
    slots = loom.loom_decode_persistent_slots(D, G)
    tc = G <= 32
    split_merge = loom.loom_model_decode_tc_time_us if tc else loom.loom_model_decode_time_us
    for s in range(1, min(1024, math.ceil(Skv / 64)) + 1):
        cands.append((split_merge(s, B, Hq, Hkv, Skv, D, NUM_SMS), 0, s))
        if not tc:  # the CUDA-core persistent split kernel, where the tensor-core one does not run
            cands.append((loom.loom_model_decode_persistent_time_us(s, B, Hq, Hkv, Skv, D, slots), 1, s))
        for cs in range(1, min(16, s) + 1):
            if s % cs:
                continue
            t = loom.loom_model_decode_cluster_time_us(s, cs, B, Hq, Hkv, Skv, D, loom.loom_decode_max_clusters(D, G, cs))
            if t > 0:
                cands.append((t, 2, s))
    return cands


@pytest.mark.parametrize("B,Hq,Hkv,Skv,D", DECODE_SHAPES)
def test_decode_split_is_brute_force_argmin(loom, B, Hq, Hkv, Skv, D):
    # Eq. 9 over both Flash Decode forms: the chosen (form, splits) is the fastest candidate
    chosen = loom.loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D)
    cands = _decode_candidates(loom, B, Hq, Hkv, Skv, D)
    best = min(t for t, _, _ in cands)
    winners = sorted((f, s) for t, f, s in cands if t <= best * (1 + 1e-9))
    assert winners[0][1] == chosen                # ties: the earlier form, then the fewest splits


def test_cluster_form_limits(loom):
    B, Hq, Hkv, Skv, D = 16, 32, 8, 8192, 128
    assert loom.loom_decode_max_clusters(D, 4, 16) > 0
    t = lambda s, cs, n: loom.loom_model_decode_cluster_time_us(s, cs, B, Hq, Hkv, Skv, D, n)
    assert t(32, 17, 100) < 0      # more than 16 CTAs per cluster
    assert t(16, 3, 100) < 0       # the cluster size must divide the split count
    assert t(16, 16, 0) < 0        # no cluster fits
    # more resident clusters never make it slower; the HBM roof bounds it
    ts = [t(16, 16, n) for n in (1, 2, 4, 8, 14, 32)]
    assert all(a >= b * (1 - 1e-9) for a, b in zip(ts, ts[1:]))
    assert ts[-1] * 1e-6 >= 2.0 * B * Hkv * Skv * D * 2 / (PEAK_GBS * 1e9) * 0.999


def test_long_decode_fills_one_wave(loom):
    # split-KV across >= one wave of CTAs over all SMs (B * Hkv * splits >= #SM)
    s = loom.loom_attn_decode_num_splits(1, 32, 8, 131072, 128)
    assert 8 * s >= NUM_SMS


@pytest.mark.parametrize("B,Hq,Hkv,Skv,D", DECODE_SHAPES)
def test_decode_time_not_below_hbm_roofline(loom, B, Hq, Hkv, Skv, D):
    s = loom.loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D)
    t = min(t for t, _, n in _decode_candidates(loom, B, Hq, Hkv, Skv, D) if n == s)
    kv_bytes = 2.0 * B * Hkv * Skv * D * 2
    assert t * 1e-6 >= kv_bytes / (PEAK_GBS * 1e9) * 0.999


def test_decode_more_splits_than_needed_cost_more(loom):
    # beyond the argmin, extra splits only add merge work and item boundaries
    B, Hq, Hkv, Skv, D = 16, 32, 8, 8192, 128
    s = loom.loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D)
    t = lambda n: loom.loom_model_decode_tc_time_us(n, B, Hq, Hkv, Skv, D, NUM_SMS)
    assert t(min(128, 8 * s)) > t(s)


@pytest.mark.parametrize("B,Hq,Hkv,Skv,D", DECODE_SHAPES)
def test_tc_decode_pays_the_start_up_once(loom, B, Hq, Hkv, Skv, D):
    # the persistent tensor-core split kernel starts once and streams its items back to
    # back, where the one-CTA-per-split kernel pays the start-up in every round of CTAs:
    # with more than one round it is faster; no count beats the HBM roofline
    for s in range(1, min(64, math.ceil(Skv / 64)) + 1):
        t_tc = loom.loom_model_decode_tc_time_us(s, B, Hq, Hkv, Skv, D, NUM_SMS)
        t_cc = loom.loom_model_decode_time_us(s, B, Hq, Hkv, Skv, D, NUM_SMS)
        if B * Hkv * s > 2 * NUM_SMS:
            assert 0 < t_tc < t_cc, (s, t_tc, t_cc)
        assert t_tc * 1e-6 >= 2.0 * B * Hkv * Skv * D * 2 / (PEAK_GBS * 1e9) * 0.999


def test_tc_decode_rounds_and_limits(loom):
    t = lambda s, Hq=32, Hkv=8: loom.loom_model_decode_tc_time_us(s, 1, Hq, Hkv, 131072, 128, NUM_SMS)
    assert t(8, Hq=512, Hkv=8) < 0          # 64 query heads per kv head: not this kernel
    assert t(0) < 0
    # 38 splits x 8 kv heads = 304 items: one round on two CTAs per SM; one more split
    # leaves 8 items to a second round, streamed by 8 CTAs at the rate one CTA sustains
    assert 8 * 38 == 2 * NUM_SMS
    assert t(39) > t(38) * 1.3
    # the long decode's count fills the SMs once, two CTAs on some of them (32 splits x 8
    # kv heads = 256 CTAs: the sweep's measured best)
    s = loom.loom_attn_decode_num_splits(1, 32, 8, 131072, 128)
    assert NUM_SMS < 8 * s <= 2 * NUM_SMS


def test_tc_decode_stage_chain_floor(loom):
    # at D = 64 a 64-key stage carries half the bytes for the same S -> softmax -> P.V
    # chain: with every SM busy the chain, not HBM, bounds the stage, so the modeled time
    # exceeds the byte time by the chain's share
    t64 = loom.loom_model_decode_tc_time_us(19, 1, 64, 16, 65536, 64, NUM_SMS)
    bytes_time = 2.0 * 16 * 65536 * 64 * 2 / (PEAK_GBS * 1e3)  # us
    assert t64 > bytes_time * 1.2


@pytest.mark.parametrize("D", [64, 128])
def test_per_design_time_matches_the_choice(loom, D):
    # the per-design modeled time of the chosen design is the model's launch time; an
    # infeasible design reports a negative time
    chosen = loom.loom_model_fwd_plan(D)["design"]
    args = (4, 32, 2048, 2048, D, 0)
    assert loom.loom_model_fwd_time_us_design(chosen, *args) == pytest.approx(loom.loom_model_fwd_time_us(*args))
    for d in (1, 2, 3, 4):
        t = loom.loom_model_fwd_time_us_design(d, *args)
        assert (t < 0) == (loom.loom_model_fwd_plan_variant(D, d) is None)
        if t > 0:
            assert t >= loom.loom_model_fwd_time_us(*args) * (1 - 1e-9)  # the choice is the fastest
