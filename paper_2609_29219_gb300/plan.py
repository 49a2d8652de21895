"""Print the analytic model's choices (Sec. 2.6, Eq. 5-9): the prefill plan per head
dimension with every design it ranked, and the decode split count with the modeled time of
each workload.  Runs on the host; no GPU is needed (the decode choice then assumes the
GB300's 152 SMs).

    python -m paper_2609_29219_gb300.plan
"""
import paper_2609_29219_gb300 as loom

PREFILL = [("tiny attention", 1, 2, 128, 64, False), ("tiny attention causal", 1, 2, 128, 64, True),
           ("prefill B4 H32 S2048 D128", 4, 32, 2048, 128, False),
           ("prefill B4 H32 S2048 D128 causal", 4, 32, 2048, 128, True),
           ("long prefill B1 H32/8 S8192 D128 causal", 1, 32, 8192, 128, True),
           ("long prefill B1 H64/16 S8192 D64 causal", 1, 64, 8192, 64, True)]
DECODE = [("batched decode B16 H32/8 Skv8192 D128", 16, 32, 8, 8192, 128),
          ("long decode B1 H32/8 Skv131072 D128", 1, 32, 8, 131072, 128)]
DESIGNS = {1: "one query tile, S double-buffered", 2: "two query tiles, alternating",
           3: "two query tiles, ring of three S buffers"}


def main():
    for D in (64, 128):
        p = loom.loom_model_fwd_plan(D)
        print(f"prefill D={D}: design {p['design']} ({DESIGNS[p['design']]}), BM={p['bm']} BN={p['bn']} "
              f"query tiles/CTA={p['q_tiles']} S buffers={p['s_buffers']} K/V slots={p['kv_slots']} "
              f"knob b=({p['b_lm']},{p['b_ms']}) smem={p['smem_bytes']} B tmem={p['tmem_cols']} cols")
        for d in (1, 2, 3):
            v = loom.loom_model_fwd_plan_variant(D, d)
            if v is None:
                print(f"    design {d}: infeasible (Eq. 8)")
            else:
                print(f"    design {d}: T_iter={v['t_iter_ns']:.0f} ns per KV tile and query tile "
                      f"(load {v['t_load_ns']:.0f}, MMA {v['t_mma_ns']:.0f}, softmax {v['t_softmax_ns']:.0f})")
    for name, B, H, S, D, causal in PREFILL:
        t = loom.loom_model_fwd_time_us(B, H, S, S, D, causal)
        pairs = S * (S + 1) / 2 if causal else S * S
        print(f"{name}: modeled {t:.1f} us = {4.0 * B * H * D * pairs / (t * 1e-6) / 1e12:.0f} TFLOP/s")
    for name, B, Hq, Hkv, S, D in DECODE:
        s = loom.loom_attn_decode_num_splits(B, Hq, Hkv, S, D)
        t = loom.loom_model_decode_time_us(s, B, Hq, Hkv, S, D, 152)
        print(f"{name}: {s} splits ({B * Hkv * s} split CTAs), modeled {t:.1f} us = "
              f"{2.0 * B * Hkv * S * D * 2 / (t * 1e-6) / 1e9:.0f} GB/s (all sequences at Skv)")


if __name__ == "__main__":
    main()
