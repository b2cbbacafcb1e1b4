"""The benchmark's algorithmic byte and flop counts, which every reported
rate and roofline fraction divides by, against the definitions written out
by hand: one pass over the compact cache (K and V rows plus one float32
log(1/pi) per row, the queries, the five outputs) for the certified decode;
kept rows read and written plus their indices for the gather; two passes of
Q_obs K^T for the accumulated-attention scores."""
import numpy as np

import bench
from paper_2607_21475_gb300.workloads import WORKLOADS


def test_decode_bytes_of_the_dialogue_workload():
    w = WORKLOADS["dialogue_32k"]          # B=32, 32/8 heads, d=128, bf16
    n = [np.full((32, 8), 3277)]
    rows = 32 * 8 * 3277 * (128 * 2 * 2 + 4)   # K and V rows of 256 bytes, log(1/pi)
    q = 32 * 32 * 128 * 2                      # one bf16 query per query head
    outs = 32 * 32 * (128 + 4) * 4             # y [d] and lse, V_hat, b_t, r_t, float32
    assert bench.decode_bytes(w, n) == rows + q + outs == 433_681_408


def test_decode_bytes_sum_over_layers_and_ragged_units():
    w = WORKLOADS["qwen7b_6k"].with_(n_layers=2)   # B=8, 28/4 heads, d=128, bf16
    n = [np.arange(32).reshape(8, 4), np.zeros((8, 4), dtype=np.int64)]
    per_layer_fixed = 8 * 28 * 128 * 2 + 8 * 28 * 132 * 4
    assert bench.decode_bytes(w, n) == sum(range(32)) * 516 + 2 * per_layer_fixed


def test_gather_bytes_count_each_kept_row_read_and_written():
    w = WORKLOADS["tiny"]                  # float32, d=64
    n = [np.array([[51, 50, 52, 49]])]
    assert bench.gather_bytes(w, n) == 202 * (4 * 64 * 4 + 4)


def test_score_flops_are_two_passes_of_the_observation_product():
    w = WORKLOADS["qwen7b_6k"]             # 64 observation rows x G=7 per KV head
    units = 8 * 4
    per_pass = 2 * (64 * 7) * 6144 * 128   # multiply-adds of Q_obs K^T per unit
    assert bench.score_flops(w) == 28 * units * 2 * per_pass == 45_097_156_608 * 28


def test_whole_job_rate_is_weak_scaling():
    assert bench.whole_job_rate(10.0, 4, 2.0) == 20.0
