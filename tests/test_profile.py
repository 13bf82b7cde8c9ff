"""profile.json (App. A.4 schema): the native writer, fed with the oracle's
join on CPU, read back and checked field by field.  CPU only."""
import json

import numpy as np
import pytest

import oracle
import tracegen

COUNTER_FIELDS = ["gpu_time_duration_ns", "dram_bytes_read", "dram_bytes_written", "memory_throughput_pct",
                  "dram_throughput_pct", "mem_busy_pct", "l1_hit_rate", "l2_hit_rate", "sm_throughput_pct",
                  "tensor_core_active_pct", "sm_active_cycles", "achieved_occupancy", "warp_cycles_per_instr",
                  "eligible_cycles_pct", "executed_instructions", "ipc_active", "avg_threads_per_warp",
                  "registers_per_thread", "local_memory_spills", "dynamic_smem_per_block"]
METHOD = {0: "unattributed", 1: "torch_profiler_correlation", 2: "nvtx", 3: "inductor_fusion"}
CONF = {1: "high", 2: "medium", 3: "medium"}


def _val(x):
    return None if np.isnan(x) else float(x)


def write_and_read(tmp_path, t, r, **kw):
    import paper_2609_11938_gb300 as opa
    path = tmp_path / "profile.json"
    n = opa.write_profile(path, t.k_stream, t.k_dur, t.k_name, r["op_of_kernel"], r["ncu_idx"], t.counters, r["ops"],
                          tier=r["tier"], is_fused=r["is_fused"], fused_with=r["fused_with"], **kw)
    text = path.read_text()
    assert n == len(text.encode())
    return json.loads(text)


@pytest.mark.parametrize("name", ["tiny", "gpt2_dedup"])
def test_profile_document(tmp_path, name):
    t = tracegen.with_tiers(tracegen.generate(name))
    r = oracle.run_tiers(t)
    names = [f"kern{i}" for i in range(int(t.k_name.max()) + 1)]
    opn = [f"aten::op{i % 7}" for i in range(t.n_ops)]
    d = write_and_read(tmp_path, t, r, kernel_names=names, op_names=opn,
                       meta={"model_name": "synthetic", "device_name": "GB300"})
    assert d["schema_version"] == "1.0"
    assert d["capture_metadata"] == {"model_name": "synthetic", "device_name": "GB300"}
    op = r["op_of_kernel"]
    ops = r["ops"]
    present = np.nonzero(ops["kernel_count"] > 0)[0]
    assert [o["call_index"] for o in d["operators"]] == present.tolist()
    seen = np.zeros(t.K, int)
    for rec, o in zip(d["operators"], present):
        assert rec["operator_name"] == opn[o] and rec["operator_id"] == f"{opn[o]}_{o}"
        ks = [int(k["kernel_id"][2:]) for k in rec["kernels"]]
        assert ks == sorted(ks) and all(op[k] == o for k in ks)
        seen[ks] += 1
        assert rec["is_fused"] == bool(r["is_fused"][ks].any())
        fw = {opn[f] for f in r["fused_with"][ks] if f != oracle.OP_NONE and f != o}
        assert set(rec["fused_with"]) == fw and len(rec["fused_with"]) == len(fw)
        a = rec["aggregated"]
        assert a["kernel_count"] == ops["kernel_count"][o] == len(ks)
        assert a["total_duration_ns"] == ops["total_duration_ns"][o]
        assert a["matched_count"] == ops["matched_count"][o]
        for c, f in enumerate(COUNTER_FIELDS):
            assert a[f] == _val(ops["agg"][c][o]), (o, f)        # 17 digits read back exactly
        for k, kr in zip(ks, rec["kernels"]):
            assert kr["kernel_name"] == names[t.k_name[k]]
            assert kr["attribution_method"] == METHOD[int(r["tier"][k])]
            assert kr["confidence"] == CONF[int(r["tier"][k])]
            assert kr["duration_ns"] == t.k_dur[k] and kr["stream_id"] == t.k_stream[k]
            j = r["ncu_idx"][k]
            want = [_val(np.float64(v)) for v in t.counters[j]] if j >= 0 else [None] * 20
            assert [kr["metrics"][f] for f in COUNTER_FIELDS] == want
    un = [int(k["kernel_id"][2:]) for k in d["unattributed_kernels"]]
    assert un == np.nonzero(op == oracle.OP_NONE)[0].tolist()
    assert all(k["attribution_method"] == "unattributed" and "confidence" not in k for k in d["unattributed_kernels"])
    seen[un] += 1
    assert (seen == 1).all()                     # every kernel exactly once


def test_profile_without_kernels_and_defaults(tmp_path):
    t = tracegen.generate("tiny")
    r = oracle.run_tiers(t, use_corr=False, use_fusion=False)
    d = write_and_read(tmp_path, t, r, include_kernels=False)
    assert d["capture_metadata"] == {}
    assert all("kernels" not in o for o in d["operators"])
    o0 = d["operators"][0]
    assert o0["operator_name"] == f"op_{o0['call_index']}" and o0["fused_with"] == []
    assert d["unattributed_kernels"][0]["kernel_name"].startswith("kernel_")


def test_profile_rejects(tmp_path):
    import paper_2609_11938_gb300 as opa
    t = tracegen.generate("tiny")
    r = oracle.run_tiers(t)
    bad = r["op_of_kernel"].copy()
    bad[0] = t.n_ops
    with pytest.raises(opa.OpattrError):
        opa.write_profile(tmp_path / "p.json", t.k_stream, t.k_dur, t.k_name, bad, r["ncu_idx"], t.counters, r["ops"])
    with pytest.raises(opa.OpattrError):
        opa.write_profile(tmp_path / "no_dir" / "p.json", t.k_stream, t.k_dur, t.k_name, r["op_of_kernel"],
                          r["ncu_idx"], t.counters, r["ops"])
