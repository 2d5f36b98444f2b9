"""The algorithmic bytes and flops bench.py divides by, checked against the
cost model written out by hand for the Llama-3-8B-shaped step (32 layers,
32 query / 8 KV heads, head_dim 128, k = 128 selected rows, W = 512 window)
and the paper's MACs per generated token (appendix, Attention MACs
Analysis: MACs_t = 2 n_h d_h n_l L_t, two flops per MAC)."""

import bench


def test_decode_step_bytes_llama_shape():
    B, L, Hq, Hkv, d, k, W = 1, 32, 32, 8, 128, 128, 512
    row = d * 2  # one bf16 K or V row
    units = B * L * Hkv
    kv_read = units * 2 * row * (k + W - 1)   # k Tier-1 rows and W - 1 old ring rows, K and V
    new_tok = units * 2 * row * 2             # the new token's K,V read once and written once
    q_out = B * L * Hq * d * 2 * 2            # q read, out written
    assert bench.decode_step_bytes(B, L, Hq, Hkv, d, k, W) == kv_read + new_tok + q_out
    assert bench.decode_step_bytes(B, L, Hq, Hkv, d, k, W) == 84_541_440
    # idx read as well when the step gathers the Tier-1 rows itself
    assert bench.decode_step_bytes(B, L, Hq, Hkv, d, k, W, gather=True) == 84_541_440 + 4 * k


def test_decode_step_flops_are_twice_the_papers_macs():
    B, L, Hq, d, k, W = 1, 32, 32, 128, 128, 512
    macs_per_token = 2 * Hq * d * L * (k + W)  # MACs_t with L_t = k + W cached keys
    assert bench.decode_step_flops(B, L, Hq, d, k, W) == 2 * macs_per_token == 335_544_320


def test_select_and_gather_bytes():
    # one bank of 1,024 CMEs of dimension 4,096 (fp32) read once, q_vec read,
    # k indices written
    assert bench.select_bytes(1, 1024, 4096, 128) == 4 * 1024 * 4096 + 4 * 4096 + 4 * 128
    # the selected K and V rows of every (layer, KV head) read and written,
    # idx read
    assert bench.tier1_gather_bytes(1, 32, 8, 128, 128) == 2 * 2 * 32 * 8 * 128 * 128 * 2 + 4 * 128


def test_job_value_counts_every_rank():
    # tokens/s of the whole job: N ranks x steps x requests x batch x decode steps / time
    assert bench.job_tokens_per_s(2, 10, 4, 1, 3000, 1000.0) == 2 * 10 * 4 * 1 * 3000 / 1.0


def test_select_launches_follow_the_one_launch_rule():
    """One launch when CTAs of at most 8 rows (a divisor of N) cover the bank
    in one wave of one CTA per SM and N <= 2,048, D <= 4,096; else two."""
    assert bench.select_launches(1, 1024, 4096, 152) == 1      # Llama shape: 128 CTAs of 8
    assert bench.select_launches(1, 1216, 64, 152) == 1        # 152 CTAs of 8
    assert bench.select_launches(1, 1217, 64, 152) == 2        # prime: 1 row a CTA, 1,217 CTAs
    assert bench.select_launches(32, 2048, 4096, 152) == 2     # Mistral batch: too many rows
    assert bench.select_launches(1, 1024, 4100, 152) == 2      # D above 4,096
    assert bench.select_launches(1, 4096, 64, 152) == 2        # N above 2,048
    assert bench.select_launches(4, 256, 512, 152) == 1        # tiny batch of 4: 128 CTAs of 8


def test_profiled_traffic_reads_both_figures(tmp_path, monkeypatch):
    """The traffic record: (request-loop bytes, flushed-cache bytes) while its
    kernel hash and workload match the current source and run; (None, None)
    otherwise; the loop figure None when the record has none."""
    import json
    rec = {"workload": "llama3_8b", "tier1": "dense", "dram_bytes_per_launch": 86,
           "kernel_source_sha256": bench.kernel_source_hash(),
           "in_loop": {"dram_bytes_per_launch": 77}}
    f = tmp_path / "rec.json"
    f.write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "PROFILE_FILE", str(f))
    assert bench.profiled_traffic("llama3_8b", "dense") == (77, 86)
    assert bench.profiled_traffic("llama3_8b", "gather") == (None, None)
    assert bench.profiled_traffic("tiny", "dense") == (None, None)
    del rec["in_loop"]
    f.write_text(json.dumps(rec))
    assert bench.profiled_traffic("llama3_8b", "dense") == (None, 86)
    rec["kernel_source_sha256"] = "0" * 64
    f.write_text(json.dumps(rec))
    assert bench.profiled_traffic("llama3_8b", "dense") == (None, None)
