"""Host logic of the benchmark (no GPU): the algorithmic byte count of a step is the
sum of the weights it streams (from the weight shapes themselves) plus the KV rows it
reads, and the job rate / max-over-ranks helpers."""
import bench
import synth


def _weights(cfg, prefix):
    n = 0
    for name, shape in synth.weight_shapes(cfg):
        if name.startswith(prefix) and not name.endswith("norm"):
            m = 1
            for v in shape:
                m *= v
            n += m
    return n * 2  # bf16


def test_step_bytes_from_weight_shapes():
    cfg = synth.get_config("7b")
    d, L, N, V = cfg["d_model"], cfg["n_layers"], cfg["tree_nodes"], cfg["vocab"]
    n_ctx = 527
    b = bench.step_bytes(cfg, n_ctx)
    layers = _weights(cfg, "layers.")
    verify_w = layers + _weights(cfg, "lm_head") + N * d * 2  # gathered embedding rows
    assert b["verify_weights"] == verify_w
    assert b["verify_kv"] == L * (n_ctx + N) * 2 * d * 2
    draft_block = _weights(cfg, "draft.")
    tri = _weights(cfg, "tri_w")
    heads = _weights(cfg, "heads.")
    K = cfg["n_draft_heads"]
    draft_w = K * (tri + draft_block) + heads + K * 3 * d * 2
    draft_kv = sum((n_ctx + k + 1) * 2 * d * 2 for k in range(K))
    assert b["draft"] == draft_w + draft_kv
    assert abs(b["total"] - (b["verify"] + b["draft"] + b["commit"])) < 1
    # the 7B step streams ~17.9 GB of weights and KV at this committed length
    assert 17.5e9 < b["total"] < 18.2e9


def test_job_rate_and_single_rank_max():
    assert bench.max_over_ranks(3.25, 1) == 3.25
    assert abs(bench.job_rate(64, 4, 2.0) - 4 * 64 / 2e-3) < 1e-6


def test_step_bytes_batch_shares_weights_and_sums_kv():
    # a batch reads every weight once and each sequence's own KV rows; a batch of one
    # given as a list is the int case
    cfg = synth.get_config("7b_b8")
    d, L, N, K = cfg["d_model"], cfg["n_layers"], cfg["tree_nodes"], cfg["n_draft_heads"]
    ns = [2943, 3503, 2192, 1807, 3696, 649, 3521, 1451]
    b = bench.step_bytes(cfg, ns)
    one = bench.step_bytes(cfg, ns[0])
    assert bench.step_bytes(cfg, [ns[0]]) == one
    kv_row = 2 * d * 2
    assert b["verify_kv"] == L * sum(n + N for n in ns) * kv_row
    # weights: the single-sequence count minus its gathered rows, plus the batch's rows
    assert b["verify_weights"] == one["verify_weights"] + (len(ns) - 1) * N * d * 2
    assert b["draft"] - sum((n + k + 1) * kv_row for n in ns for k in range(K)) == \
        one["draft"] - sum((ns[0] + k + 1) * kv_row for k in range(K)) + (len(ns) - 1) * K * 3 * d * 2
