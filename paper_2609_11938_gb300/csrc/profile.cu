// profile.cu -- profile.json writer (the schema of App. A.4): host code over
// the join's outputs, copied back by the caller.
//
// Layout: schema_version, capture_metadata, operators[] (one per operator
// with attributed kernels, in op-id order: operator_id "<name>_<call_index>",
// operator_name, call_index, is_fused, fused_with[], kernels[] in kernel
// order, aggregated{}), unattributed_kernels[].  The attribution tier gives
// attribution_method and confidence (Fig. 2: correlation = high, NVTX and
// Inductor fusion = medium).  Counter fields use the profile names of Table 8
// in its order; NaN (null counter, or no row) is written as null.  Doubles
// are printed with 17 significant digits, so they read back exactly.
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <string>
#include <vector>

#include "opattr.h"

namespace {

const char *const COUNTER_FIELD[OPATTR_N_COUNTERS] = {
    "gpu_time_duration_ns", "dram_bytes_read",      "dram_bytes_written",    "memory_throughput_pct",
    "dram_throughput_pct",  "mem_busy_pct",         "l1_hit_rate",           "l2_hit_rate",
    "sm_throughput_pct",    "tensor_core_active_pct", "sm_active_cycles",    "achieved_occupancy",
    "warp_cycles_per_instr", "eligible_cycles_pct", "executed_instructions", "ipc_active",
    "avg_threads_per_warp", "registers_per_thread", "local_memory_spills",   "dynamic_smem_per_block",
};

// Buffered output with a running byte count.
struct Out {
    FILE *f = nullptr;
    std::string buf;
    int64_t total = 0;
    bool ok = true;
    void flush() {
        if (!buf.empty() && f) {
            if (fwrite(buf.data(), 1, buf.size(), f) != buf.size()) ok = false;
            total += (int64_t)buf.size();
        }
        buf.clear();
    }
    void put(const char *s) {
        buf += s;
        if (buf.size() > (1u << 22)) flush();
    }
    void put(const std::string &s) { put(s.c_str()); }
    void i64(long long v) {
        char t[32];
        snprintf(t, sizeof t, "%lld", v);
        put(t);
    }
    void f64(double v) {
        if (isnan(v) || isinf(v)) {
            put("null");
            return;
        }
        char t[40];
        snprintf(t, sizeof t, "%.17g", v);
        put(t);
    }
    void str(const char *s) {              // JSON string with escapes
        std::string o = "\"";
        for (const unsigned char *p = (const unsigned char *)s; *p; ++p) {
            if (*p == '"' || *p == '\\') { o += '\\'; o += (char)*p; }
            else if (*p < 0x20) { char t[8]; snprintf(t, sizeof t, "\\u%04x", *p); o += t; }
            else o += (char)*p;
        }
        o += '"';
        put(o);
    }
};

std::string kernel_name(const opattr_profile_names *nm, uint32_t id) {
    if (nm && nm->kernel_name && (int64_t)id < nm->n_kernel_names && nm->kernel_name[id]) return nm->kernel_name[id];
    return "kernel_" + std::to_string(id);
}
std::string op_name(const opattr_profile_names *nm, uint32_t op) {
    if (nm && nm->op_name && nm->op_name[op]) return nm->op_name[op];
    return "op_" + std::to_string(op);
}
long long call_index(const opattr_profile_names *nm, uint32_t op) {
    return nm && nm->op_call_index ? (long long)nm->op_call_index[op] : (long long)op;
}

void kernel_record(Out &o, const opattr_profile_names *nm, const opattr_kernels *k, int64_t i, uint8_t t,
                   const int32_t *nidx, const float *counters) {
    static const char *method[4] = {"unattributed", "torch_profiler_correlation", "nvtx", "inductor_fusion"};
    static const char *conf[4] = {nullptr, "high", "medium", "medium"};
    char id[32];
    snprintf(id, sizeof id, "k_%05lld", (long long)i);
    o.put("{\"kernel_id\": ");
    o.str(id);
    o.put(", \"kernel_name\": ");
    o.str(kernel_name(nm, k->name_id[i]).c_str());
    o.put(", \"attribution_method\": ");
    o.str(method[t & 3]);
    if (conf[t & 3]) {
        o.put(", \"confidence\": ");
        o.str(conf[t & 3]);
    }
    o.put(", \"duration_ns\": ");
    o.i64(k->dur_ns[i]);
    o.put(", \"stream_id\": ");
    o.i64(k->stream[i]);
    o.put(", \"metrics\": {");
    const int32_t j = nidx[i];
    for (int c = 0; c < OPATTR_N_COUNTERS; ++c) {
        if (c) o.put(", ");
        o.str(COUNTER_FIELD[c]);
        o.put(": ");
        o.f64(j >= 0 ? (double)counters[(int64_t)j * OPATTR_N_COUNTERS + c] : NAN);
    }
    o.put("}}");
}

}  // namespace

extern "C" opattr_status opattr_write_profile(const char *path, const opattr_profile_meta *meta,
                                              const opattr_profile_names *names, const opattr_kernels *kernels,
                                              const uint32_t *op_of_kernel, const uint8_t *tier,
                                              const uint8_t *is_fused, const uint32_t *fused_with,
                                              const int32_t *ncu_idx_of_kernel, const float *counters,
                                              int64_t n_rows, uint32_t n_ops, const opattr_op_aggregates *ops,
                                              int64_t *bytes_written) {
    if (!path || !kernels || !ops) return OPATTR_E_INVALID_ARG;
    const int64_t K = kernels->n, O = n_ops;
    if (K < 0 || n_rows < 0) return OPATTR_E_INVALID_ARG;
    if (K > 0 && (!kernels->stream || !kernels->dur_ns || !kernels->name_id || !op_of_kernel || !ncu_idx_of_kernel))
        return OPATTR_E_INVALID_ARG;
    if (n_rows > 0 && !counters) return OPATTR_E_INVALID_ARG;
    if (O > 0 && (!ops->kernel_count || !ops->total_duration_ns || !ops->matched_count || !ops->agg))
        return OPATTR_E_INVALID_ARG;
    // kernels per operator, in kernel order (counting sort)
    std::vector<int64_t> start((size_t)O + 1, 0);
    for (int64_t i = 0; i < K; ++i) {
        const uint32_t op = op_of_kernel[i];
        if (op != OPATTR_OP_NONE && (int64_t)op >= O) return OPATTR_E_INVALID_ARG;
        if (ncu_idx_of_kernel[i] < -1 || ncu_idx_of_kernel[i] >= n_rows) return OPATTR_E_INVALID_ARG;
        if (op != OPATTR_OP_NONE) start[(size_t)op + 1]++;
    }
    for (int64_t o = 0; o < O; ++o) start[(size_t)o + 1] += start[(size_t)o];
    std::vector<int64_t> member((size_t)start[(size_t)O]);
    {
        std::vector<int64_t> fill(start.begin(), start.end() - 1);
        for (int64_t i = 0; i < K; ++i)
            if (op_of_kernel[i] != OPATTR_OP_NONE) member[(size_t)fill[op_of_kernel[i]]++] = i;
    }
    Out o;
    o.f = fopen(path, "wb");
    if (!o.f) return OPATTR_E_INVALID_ARG;
    const bool with_kernels = !meta || meta->include_kernels;
    o.put("{\n  \"schema_version\": \"1.0\",\n  \"capture_metadata\": {");
    {
        const char *keys[4] = {"model_name", "device_name", "compile_mode", "capture_timestamp_utc"};
        const char *vals[4] = {meta ? meta->model_name : nullptr, meta ? meta->device_name : nullptr,
                               meta ? meta->compile_mode : nullptr, meta ? meta->capture_timestamp_utc : nullptr};
        bool first = true;
        for (int q = 0; q < 4; ++q) {
            if (!vals[q]) continue;
            o.put(first ? "" : ", ");
            first = false;
            o.str(keys[q]);
            o.put(": ");
            o.str(vals[q]);
        }
    }
    o.put("},\n  \"operators\": [");
    bool first_op = true;
    for (int64_t op = 0; op < O; ++op) {
        const int64_t b = start[(size_t)op], e = start[(size_t)op + 1];
        if (ops->kernel_count[op] == 0 && b == e) continue;
        o.put(first_op ? "\n    {" : ",\n    {");
        first_op = false;
        const std::string name = op_name(names, (uint32_t)op);
        const long long ci = call_index(names, (uint32_t)op);
        o.put("\"operator_id\": ");
        o.str((name + "_" + std::to_string(ci)).c_str());
        o.put(", \"operator_name\": ");
        o.str(name.c_str());
        o.put(", \"call_index\": ");
        o.i64(ci);
        bool fused = false;
        std::vector<std::string> with;
        for (int64_t m = b; m < e; ++m) {
            const int64_t i = member[(size_t)m];
            fused |= is_fused && is_fused[i];
            const uint32_t fw = fused_with ? fused_with[i] : OPATTR_OP_NONE;
            if (fw != OPATTR_OP_NONE && (int64_t)fw < O && fw != (uint32_t)op) {
                const std::string n2 = op_name(names, fw);
                bool seen = false;
                for (const auto &x : with) seen |= x == n2;
                if (!seen) with.push_back(n2);
            }
        }
        o.put(", \"is_fused\": ");
        o.put(fused ? "true" : "false");
        o.put(", \"fused_with\": [");
        for (size_t q = 0; q < with.size(); ++q) {
            if (q) o.put(", ");
            o.str(with[q].c_str());
        }
        o.put("]");
        if (with_kernels) {
            o.put(", \"kernels\": [");
            for (int64_t m = b; m < e; ++m) {
                const int64_t i = member[(size_t)m];
                o.put(m == b ? "\n      " : ",\n      ");
                kernel_record(o, names, kernels, i, tier ? tier[i] : (uint8_t)OPATTR_TIER_NVTX, ncu_idx_of_kernel,
                              counters);
            }
            o.put("]");
        }
        o.put(", \"aggregated\": {\"total_duration_ns\": ");
        o.i64(ops->total_duration_ns[op]);
        o.put(", \"kernel_count\": ");
        o.i64(ops->kernel_count[op]);
        o.put(", \"matched_count\": ");
        o.i64(ops->matched_count[op]);
        for (int c = 0; c < OPATTR_N_COUNTERS; ++c) {
            o.put(", ");
            o.str(COUNTER_FIELD[c]);
            o.put(": ");
            o.f64(ops->agg[(int64_t)c * O + op]);
        }
        o.put("}}");
    }
    o.put("\n  ],\n  \"unattributed_kernels\": [");
    bool first_k = true;
    for (int64_t i = 0; i < K; ++i) {
        if (op_of_kernel[i] != OPATTR_OP_NONE) continue;
        o.put(first_k ? "\n    " : ",\n    ");
        first_k = false;
        kernel_record(o, names, kernels, i, OPATTR_TIER_NONE, ncu_idx_of_kernel, counters);
    }
    o.put("\n  ]\n}\n");
    o.flush();
    const bool ok = o.ok && fclose(o.f) == 0;
    if (bytes_written) *bytes_written = o.total;
    return ok ? OPATTR_OK : OPATTR_E_INVALID_ARG;
}
