"""The benchmark's all-core oracle timing on the host: a spawn-started pool
runs the eviction, then the decode, of a sample of units and reports rates
from the per-process compute times."""
import numpy as np

import bench
from oracle import ebd_oracle as O
from paper_2607_21475_gb300.workloads import WORKLOADS, make_layer_inputs


def test_all_core_oracle_pool_runs_the_oracle_per_unit():
    w = WORKLOADS["tiny"]
    inp = make_layer_inputs(w, 0, "cpu")
    r = bench.oracle_all_cores(w, inp, max_units=4, processes=2)
    assert r["kind"] == "oracle" and r["cores"] == 2 and r["unit"] == "GB/s"
    assert r["value"] > 0 and r["evict_mtok_s"] > 0
    assert "4 of 4" in r["sample"]


def test_pool_tasks_match_the_oracle_called_directly():
    w = WORKLOADS["tiny"]
    inp = make_layer_inputs(w, 0, "cpu")
    p = {"H": w.n_kv_heads, "n_sink": w.n_sink, "n_recent": w.n_recent, "k_head": w.k_head,
         "budget": w.budget_tokens, "eps": w.eps, "seed": w.philox_seed, "cap": w.capacity}
    u = 3
    K, V = bench._host_array(inp["K"][0, u]), bench._host_array(inp["V"][0, u])
    s = inp["scores"][0, u].numpy()
    _, _, idx, logw = bench._oracle_evict_task((p, u, K, V, s, None))
    ref = O.evict_unit(K.astype(np.float64), V.astype(np.float64), s, n_sink=w.n_sink,
                       n_recent=w.n_recent, k_head=w.k_head, budget_tokens=w.budget_tokens,
                       eps=w.eps, seed=w.philox_seed, layer=0, b=0, kvh=u, capacity=w.capacity)
    assert np.array_equal(idx, ref.idx) and np.array_equal(logw, ref.logw)
