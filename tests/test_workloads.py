"""The seeded synthetic inputs against the recipe they stand for: shapes of
the paper's GQA workloads, the budget split (B_t = round(beta N), k_head =
round(0.2 B_t), capacity with a Poisson margin), score distributions and the
dialogue's 30 decaying segments, the outlier channels of the Qwen-7B-shaped
cache, and determinism of the seeds."""
import math

import numpy as np
import torch

from paper_2607_21475_gb300.workloads import WORKLOADS, make_layer_inputs, sweep_workloads


def test_configurations_have_the_stated_shapes():
    w = WORKLOADS["dialogue_32k"]
    assert (w.batch, w.n_q_heads, w.n_kv_heads, w.group, w.head_dim, w.n_ctx) == \
        (32, 32, 8, 4, 128, 32768)
    assert (w.budget_tokens, w.k_head) == (3277, 655)
    q = WORKLOADS["qwen7b_6k"]
    assert (q.n_layers, q.batch, q.n_q_heads, q.n_kv_heads, q.group, q.n_ctx) == \
        (28, 8, 28, 4, 7, 6144)
    assert (q.budget_tokens, q.k_head, q.n_obs * q.group) == (1536, 307, 448)
    t = WORKLOADS["tiny"]
    assert (t.dtype, t.n_ctx, t.budget_tokens, t.k_head) == ("f32", 512, 51, 10)
    for b, name in ((0.10, "qwen7b_16k_b10"), (0.25, "qwen7b_16k_b25"), (0.50, "qwen7b_16k_b50")):
        w16 = WORKLOADS[name]
        assert (w16.batch, w16.n_ctx, w16.budget) == (16, 16384, b)
    sw = sweep_workloads()
    assert len(sw) == 64
    assert {(w.batch, w.n_ctx, w.budget) for w in sw} == {
        (b, n, p) for b in (1, 8, 32, 64) for n in (4096, 16384, 65536, 131072)
        for p in (0.05, 0.10, 0.25, 0.50)}


def test_capacity_holds_the_expected_kept_rows_with_margin():
    for w in list(WORKLOADS.values()) + sweep_workloads()[:8]:
        bt = w.budget_tokens
        assert w.capacity % 64 == 0
        # B_t plus eight standard deviations of a Poisson tail, capped at the context
        assert w.capacity >= min(bt + 8 * math.sqrt(bt), ((w.n_ctx + 63) // 64) * 64)
        assert w.capacity <= ((w.n_ctx + 63) // 64) * 64


def test_dialogue_scores_decay_over_thirty_segments():
    w = WORKLOADS["dialogue_32k"].with_(batch=2)
    s = make_layer_inputs(w, 0, "cpu")["scores"].double().numpy()
    seg = np.minimum(np.arange(w.n_ctx) // 1092, 29)
    assert seg.max() == 29 and np.sum(seg == 29) == 32768 - 29 * 1092 == 1100
    # log-normal(0, 1.5) times 0.5^((29 - seg)/10): the mean of log s per segment
    for k in (0, 10, 29):
        logs = np.log(s[..., seg == k])
        assert abs(logs.mean() - (29 - k) / 10 * math.log(0.5)) < 0.05
        assert abs(logs.std() - 1.5) < 0.05


def test_score_distributions():
    w = WORKLOADS["qwen7b_16k_b25"].with_(batch=2)
    s = make_layer_inputs(w, 0, "cpu")["scores"].double().numpy().ravel()
    assert s.min() >= 1.0                       # Pareto with x_m = 1
    # tail of Pareto(1.2): P(s > x) = x^-1.2
    for x in (2.0, 10.0):
        assert abs(np.mean(s > x) - x ** -1.2) < 0.01
    t = WORKLOADS["tiny"]
    z = np.log(make_layer_inputs(t, 0, "cpu")["scores"].double().numpy().ravel())
    assert abs(z.mean()) < 0.1 and abs(z.std() - 1.5) < 0.1


def test_outlier_channels_scale_keys_and_values():
    w = WORKLOADS["qwen7b_6k"].with_(batch=2, n_ctx=512)
    inp = make_layer_inputs(w, 0, "cpu")
    assert "q_obs" in inp and inp["q_obs"].shape == (2, 4, 448, 128)
    for t in ("K", "V"):
        rms = inp[t].float().pow(2).mean(dim=(0, 2)).sqrt()   # [Hkv, d]
        for h in range(4):
            big = (rms[h] > 4).nonzero().flatten()
            assert big.numel() == 4                       # four channels per KV head
            assert bool(((rms[h, big] > 6) & (rms[h, big] < 10)).all())   # x 8
    k_big = {tuple((inp["K"].float().pow(2).mean(dim=(0, 2)).sqrt()[h] > 4).nonzero().flatten().tolist())
             for h in range(4)}
    assert len(k_big) > 1                                 # chosen per head


def test_inputs_are_deterministic_per_seed_and_layer():
    w = WORKLOADS["tiny"]
    a, b = make_layer_inputs(w, 0, "cpu"), make_layer_inputs(w, 0, "cpu")
    c = make_layer_inputs(w, 1, "cpu")
    for k in ("K", "V", "Q", "scores"):
        assert torch.equal(a[k], b[k])
        assert not torch.equal(a[k], c[k])


def test_peaked_attention_inputs_follow_their_recipe():
    """Sharpened queries: Q = 3 Q0; observation row r of KV head h is
    3 (Q0[h G + r // 64] + 0.5 z): its mean over the 64 rows of a query head
    sits within a few standard errors of that head's query."""
    from paper_2607_21475_gb300.workloads import peaked_attention_inputs
    w = WORKLOADS["qwen7b_6k"].with_(batch=1)
    base = make_layer_inputs(w, 2, "cpu")
    inp = peaked_attention_inputs(w, 2, "cpu", q_scale=3.0, obs_noise=0.5)
    assert "scores" not in inp and inp["q_obs"].shape == (1, 4, 64 * 7, 128)
    assert torch.equal(inp["K"], base["K"]) and torch.equal(inp["V"], base["V"])
    torch.testing.assert_close(inp["Q"].float(), (3 * base["Q"].float()).to(torch.bfloat16).float())
    qo = inp["q_obs"].float().view(1, 4, 7, 64, 128)
    dev = (qo.mean(dim=3) - 3 * base["Q"].float().view(1, 4, 7, 128)).abs()
    assert float(dev.max()) < 6 * 3 * 0.5 / 8 + 0.1  # 6 standard errors of a 64-row mean
    again = peaked_attention_inputs(w, 2, "cpu", q_scale=3.0, obs_noise=0.5)
    assert torch.equal(again["q_obs"], inp["q_obs"])
