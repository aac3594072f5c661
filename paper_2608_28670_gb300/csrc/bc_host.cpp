// bc_host.cpp -- host side of the BaryCache forecast library: the fp64 weight solver,
// the Diff Key memo, the ring-buffer cache context and the C ABI (include/barycache.h).
//
// Paper: BaryCache, Sec. 3.2 (cache context, Eq. 6; Diff Key, Eq. 7; weights, Eqs. 8-12)
// and Sec. 3.3 (full step stores the feature, cache forward applies Eq. 13).
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <string>
#include <unordered_set>
#include <vector>

#include "barycache.h"
#include "bc_internal.h"

namespace {

thread_local std::string t_last_error;

bc_status fail(bc_status s, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
bc_status fail(bc_status s, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    t_last_error = buf;
    return s;
}

bc_status cuda_fail(int err, const char *what) {
    return fail(BC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(static_cast<cudaError_t>(err)));
}

// ------------------------------------------------------------------ weight solver
//
// Both modes are evaluated from the differences d_j = t - s_j only, so that a memo entry
// keyed by the differences returns exactly what a fresh solve would (Eq. 7: the weights
// depend on the schedule through t - s_j alone).

// delta_H of Sec. 3.2 (text between Eqs. 10 and 11); a single node normalises to 1 for
// any delta.
double delta_for_window(int H) {
    if (H <= 2) return 1.0;
    if (H == 3) return 0.95;
    return 0.7;
}

bool params_valid(const bc_params &p) {
    if (p.mode != BC_MODE_EXACT && p.mode != BC_MODE_PAPER) return false;
    if (!std::isfinite(p.delta) || !std::isfinite(p.lambda)) return false;
    if (!(p.clip_C > 0.0) || !(p.eta >= 0.0) || !std::isfinite(p.eta)) return false;
    if (p.lambda < 0.0 || p.lambda > 1.0) return false;
    return true;
}

// Exact polynomial extrapolation, barycentric form:
//   c_j = (w_j / d_j) / sum_k (w_k / d_k),  w_j = 1 / prod_{k!=j} (s_j - s_k),
// with s_j - s_k = d_k - d_j.  A node hit (d_j == 0) is the interpolation property e_j.
bc_status solve_exact(const double *d, int m, double *c) {
    for (int j = 0; j < m; ++j)
        for (int k = j + 1; k < m; ++k)
            if (d[j] == d[k]) return fail(BC_ERR_DUPLICATE_NODE, "two nodes share a timestep");
    for (int j = 0; j < m; ++j) {
        if (d[j] == 0.0) {
            for (int k = 0; k < m; ++k) c[k] = (k == j) ? 1.0 : 0.0;
            return BC_OK;
        }
    }
    double q[BC_MAX_K];
    double sum = 0.0;
    for (int j = 0; j < m; ++j) {
        double prod = 1.0;
        for (int k = 0; k < m; ++k)
            if (k != j) prod *= (d[k] - d[j]);
        q[j] = 1.0 / (prod * d[j]);
        sum += q[j];
    }
    for (int j = 0; j < m; ++j) c[j] = q[j] / sum;
    return BC_OK;
}

// Eqs. 8-12.  Node factors 1/2 at both ends of the window and 1 inside (Eq. 8); raw
// weight with alternating sign, (-1)^j for j counted from 1 (Eq. 9); clip (Eq. 10);
// signed decay power and normalisation (Eq. 11); blend towards x_{f=-1} (Eq. 12, read as
// W = (1 - lambda) alpha + lambda e_1 so that the weights sum to one).
bc_status solve_paper(const double *d, int m, const bc_params &p, double *c) {
    const double delta = p.delta > 0.0 ? p.delta : delta_for_window(m);
    double a[BC_MAX_K];
    double sum = 0.0, mag = 0.0;
    for (int j = 0; j < m; ++j) {
        const double node_factor = (j == 0 || j == m - 1) ? 0.5 : 1.0;
        const double alt = (j % 2 == 0) ? -1.0 : 1.0;  // (-1)^(j+1) for C index j
        double u = node_factor * alt / d[j];
        if (u > p.clip_C) u = p.clip_C;
        if (u < -p.clip_C) u = -p.clip_C;
        const double sg = u < 0.0 ? -1.0 : 1.0;
        a[j] = sg * std::pow(std::fabs(u) + p.eta, delta);
        sum += a[j];
        mag += std::fabs(a[j]);
    }
    if (mag == 0.0 || !(std::fabs(sum) >= 1e-12 * mag))
        return fail(BC_ERR_DEGENERATE_WEIGHTS, "Eq. 11 normaliser vanishes (sum %.3g of %.3g)",
                    sum, mag);
    for (int j = 0; j < m; ++j) c[j] = (1.0 - p.lambda) * (a[j] / sum);
    c[0] += p.lambda;
    return BC_OK;
}

bc_status solve_from_differences(const double *d, int m, const bc_params &p, double *c) {
    for (int j = 0; j < m; ++j)
        if (std::isnan(d[j])) return fail(BC_ERR_INVALID_ARG, "NaN timestep");
    if (p.mode == BC_MODE_EXACT) return solve_exact(d, m, c);
    return solve_paper(d, m, p, c);
}

// ------------------------------------------------------------------ Diff Key memo (Eq. 7)
//
// Key: the weight parameters and every difference t - s_j of the live window (the paper
// prints H-1 differences; all H are needed to fix the weights, so all are keyed).
struct Memo {
    std::map<std::vector<double>, std::vector<double>> table;
    int64_t hits = 0, misses = 0;
    static constexpr size_t kCapacity = 4096;

    bc_status lookup(const double *d, int m, const bc_params &p, double *c) {
        std::vector<double> key = {static_cast<double>(p.mode), p.delta, p.lambda, p.clip_C,
                                   p.eta, static_cast<double>(m)};
        key.insert(key.end(), d, d + m);
        auto it = table.find(key);
        if (it != table.end()) {
            ++hits;
            std::memcpy(c, it->second.data(), sizeof(double) * m);
            return BC_OK;
        }
        ++misses;
        bc_status s = solve_from_differences(d, m, p, c);
        if (s != BC_OK) return s;
        if (table.size() >= kCapacity) table.clear();
        table.emplace(std::move(key), std::vector<double>(c, c + m));
        return BC_OK;
    }
};

// ------------------------------------------------------------------ cache context (Eq. 6)

constexpr uint64_t kAlign = 256;
constexpr uint32_t kMagic = 0xBA7C0DE5u;

int elem_bytes(bc_dtype d) { return d == BC_DTYPE_BF16 ? 2 : 4; }
bool dtype_valid(int d) { return d == BC_DTYPE_F32 || d == BC_DTYPE_BF16; }
uint64_t align_up(uint64_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

bc_status layout(const int64_t *numels, int n_layers, int K, int dtype,
                 std::vector<uint64_t> *offsets, uint64_t *slot_bytes) {
    if (!numels || n_layers < 1) return fail(BC_ERR_INVALID_ARG, "need at least one layer");
    if (K < 1 || K > BC_MAX_K) return fail(BC_ERR_INVALID_ARG, "K=%d outside 1..%d", K, BC_MAX_K);
    if (!dtype_valid(dtype)) return fail(BC_ERR_INVALID_ARG, "unknown dtype %d", dtype);
    const uint64_t eb = elem_bytes(static_cast<bc_dtype>(dtype));
    const uint64_t kLimit = uint64_t(1) << 50;  // 1 PiB: far beyond any device
    uint64_t off = 0;
    if (offsets) offsets->clear();
    for (int l = 0; l < n_layers; ++l) {
        if (numels[l] < 0 || static_cast<uint64_t>(numels[l]) > kLimit / eb)
            return fail(BC_ERR_INVALID_ARG, "layer %d numel %lld out of range", l,
                        static_cast<long long>(numels[l]));
        if (offsets) offsets->push_back(off);
        off += align_up(static_cast<uint64_t>(numels[l]) * eb);
        if (off > kLimit) return fail(BC_ERR_INVALID_ARG, "cache larger than 1 PiB");
    }
    *slot_bytes = off;
    return BC_OK;
}

struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) {
            ok = false;
            return;
        }
        if (prev != dev && cudaSetDevice(dev) != cudaSuccess) ok = false;
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

}  // namespace

struct bc_cache {
    uint32_t magic = kMagic;
    int n_layers = 0;
    int K = 0;
    bc_dtype dtype = BC_DTYPE_BF16;
    bc_params params{};
    int device = 0;
    std::vector<int64_t> numel;
    std::vector<uint64_t> offset;  // byte offset of each layer inside a slot
    uint64_t slot_bytes = 0;
    char *arena = nullptr;
    uint64_t arena_bytes = 0;
    int head = -1;                 // slot index of the newest node
    int count = 0;                 // live nodes (<= K)
    double node_t[BC_MAX_K] = {0, 0, 0, 0};
    Memo memo;
    bc_stats stats{};
    std::vector<bc::LayerEntry> scratch_entries;  // host staging for launch tables
    bc::DeviceTable table;                        // device layer tables (> 1016 layers only):
    bc::DeviceTable push_table;                   //   forecasts, push copies
    double *probe_partials = nullptr;             // device scratch of bc_probe_drift
    uint32_t *status = nullptr;                   // device status word of the forecast kernels
    bool inject_next = false;                     // test hooks (bc_cache_inject_fault):
    bool inject_next_drift = false;               //   next forecast / probe drift / push
    bool inject_next_push = false;
    int kernel = BC_KERNEL_AUTO;                  // bc_kernel

    char *slot_base(int slot) const { return arena + static_cast<uint64_t>(slot) * slot_bytes; }
    int slot_of_node(int j) const { return ((head - j) % K + K) % K; }  // j = 0 newest
    bool overlaps_arena(uint64_t p, uint64_t bytes) const {
        const uint64_t a0 = reinterpret_cast<uint64_t>(arena), a1 = a0 + arena_bytes;
        return bytes != 0 && arena_bytes != 0 && p < a1 && a0 < p + bytes;
    }
};

namespace {

std::mutex g_registry_mu;
std::unordered_set<bc_cache *> g_registry;

bc_status check_handle(bc_handle h) {
    if (!h) return fail(BC_ERR_BAD_HANDLE, "null handle");
    std::lock_guard<std::mutex> lk(g_registry_mu);
    if (!g_registry.count(h) || h->magic != kMagic)
        return fail(BC_ERR_BAD_HANDLE, "handle is not a live cache");
    return BC_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// A device layer table for a cache with more than kLayersLarge layers: n_layers entries of
// device memory, kTableStaging times that of pinned host staging, and one event per staging
// buffer that orders its reuse after the copy that last read it.
bc_status alloc_table(bc::DeviceTable &tb, int n_layers) {
    const size_t bytes = sizeof(bc::LayerEntry) * static_cast<size_t>(n_layers);
    void *dev = nullptr, *host = nullptr;
    cudaEvent_t ev[bc::kTableStaging] = {};
    cudaError_t e = cudaMalloc(&dev, bytes);
    if (e == cudaSuccess) e = cudaHostAlloc(&host, bytes * bc::kTableStaging, cudaHostAllocDefault);
    for (int k = 0; k < bc::kTableStaging && e == cudaSuccess; ++k)
        e = cudaEventCreateWithFlags(&ev[k], cudaEventDisableTiming);
    cudaEvent_t used = nullptr;
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&used, cudaEventDisableTiming);
    if (e != cudaSuccess) {
        cudaGetLastError();
        for (int k = 0; k < bc::kTableStaging; ++k)
            if (ev[k]) cudaEventDestroy(ev[k]);
        if (used) cudaEventDestroy(used);
        if (dev) cudaFree(dev);
        if (host) cudaFreeHost(host);
        return e == cudaErrorMemoryAllocation ? fail(BC_ERR_OOM, "layer table")
                                              : cuda_fail(e, "layer table");
    }
    tb.dev = static_cast<bc::LayerEntry *>(dev);
    tb.host = static_cast<bc::LayerEntry *>(host);
    for (int k = 0; k < bc::kTableStaging; ++k) tb.uploaded[k] = ev[k];
    tb.used = used;
    tb.capacity = n_layers;
    return BC_OK;
}

bc_status alloc_table(bc_cache *h) {
    bc_status s = alloc_table(h->table, h->n_layers);
    if (s == BC_OK) s = alloc_table(h->push_table, h->n_layers);
    return s;
}

cudaError_t free_table(bc::DeviceTable &tb) {
    cudaError_t rc = cudaSuccess;
    auto keep = [&rc](cudaError_t e) {
        if (rc == cudaSuccess && e != cudaSuccess) rc = e;
    };
    if (tb.dev) keep(cudaFree(tb.dev));
    if (tb.host) keep(cudaFreeHost(tb.host));
    for (int k = 0; k < bc::kTableStaging; ++k)
        if (tb.uploaded[k]) keep(cudaEventDestroy(static_cast<cudaEvent_t>(tb.uploaded[k])));
    if (tb.used) keep(cudaEventDestroy(static_cast<cudaEvent_t>(tb.used)));
    tb = bc::DeviceTable{};
    return rc;
}

// Free every device and pinned allocation of the handle (the caller has synchronised).
cudaError_t free_device(bc_cache *h) {
    cudaError_t rc = cudaSuccess;
    auto keep = [&rc](cudaError_t e) {
        if (rc == cudaSuccess && e != cudaSuccess) rc = e;
    };
    if (h->arena) keep(cudaFree(h->arena));
    if (h->probe_partials) keep(cudaFree(h->probe_partials));
    keep(free_table(h->table));
    keep(free_table(h->push_table));
    h->arena = nullptr;
    h->probe_partials = nullptr;
    return rc;
}

// Weights for a forecast at t_new from the live window (through the memo).
bc_status window_weights(bc_cache *h, double t_new, double *c, int *m) {
    if (!std::isfinite(t_new)) return fail(BC_ERR_INVALID_ARG, "non-finite target timestep");
    if (h->count == 0) return fail(BC_ERR_NOT_READY, "forecast before any push");
    double d[BC_MAX_K];
    for (int j = 0; j < h->count; ++j) d[j] = t_new - h->node_t[h->slot_of_node(j)];
    *m = h->count;
    return h->memo.lookup(d, h->count, h->params, c);
}

bc_status check_new_node(bc_cache *h, double t) {
    if (!std::isfinite(t)) return fail(BC_ERR_INVALID_ARG, "non-finite timestep");
    // Nodes that survive this push: all live ones, minus the oldest when the ring is full.
    const int keep = h->count < h->K ? h->count : h->K - 1;
    for (int j = 0; j < keep; ++j)
        if (h->node_t[h->slot_of_node(j)] == t)
            return fail(BC_ERR_DUPLICATE_NODE, "timestep %.17g already cached", t);
    return BC_OK;
}

void rotate_in(bc_cache *h, double t) {
    h->head = (h->head + 1) % h->K;
    h->node_t[h->head] = t;
    if (h->count < h->K) ++h->count;
    ++h->stats.pushes;
}

// Sampler update applied to one layer in the forecast's launch: x <- ca x + cb v_hat + cc z.
struct Update {
    double ca = 1.0, cb = 0.0, cc = 0.0;
    int v_layer = -1;
    void *x = nullptr;
    bc_dtype x_dtype = BC_DTYPE_F32;
    const void *z = nullptr;
};

bool ranges_overlap(uint64_t a, uint64_t an, uint64_t b, uint64_t bn) {
    return an && bn && a < b + bn && b < a + an;
}

// The device layer table for a forecast of n_layers layers, or nullptr when the launch must
// carry its tables in parameter blocks: few enough layers, no table on this handle, or a
// stream that is being captured into a CUDA graph (a graph must hold every table it replays,
// while the device table is rewritten by later calls).
bc::DeviceTable *table_for(bc::DeviceTable &tb, int n_layers, void *stream) {
    if (n_layers <= bc::kLayersLarge || !tb.dev || n_layers > tb.capacity) return nullptr;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(static_cast<cudaStream_t>(stream), &cs) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return cs == cudaStreamCaptureStatusNone ? &tb : nullptr;
}

bc_status forecast_impl(bc_handle h, double t_new, void *const *out_ptrs, bc_dtype out_dtype,
                        const Update &up, void *stream) {
    const int v_layer = up.v_layer;
    void *x = up.x;
    const bc_dtype x_dtype = up.x_dtype;
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!out_ptrs) return fail(BC_ERR_INVALID_ARG, "out_ptrs is NULL");
    if (!dtype_valid(out_dtype)) return fail(BC_ERR_INVALID_ARG, "unknown output dtype");
    const bool euler = v_layer >= 0;
    if (euler) {
        if (v_layer >= h->n_layers) return fail(BC_ERR_INVALID_ARG, "v_layer out of range");
        if (!x) return fail(BC_ERR_INVALID_ARG, "x is NULL");
        if (!dtype_valid(x_dtype)) return fail(BC_ERR_INVALID_ARG, "unknown x dtype");
        if (!aligned16(x)) return fail(BC_ERR_ALIGNMENT, "x is not 16-byte aligned");
        if (up.z && !aligned16(up.z)) return fail(BC_ERR_ALIGNMENT, "z is not 16-byte aligned");
        if (!std::isfinite(up.ca) || !std::isfinite(up.cb) || !std::isfinite(up.cc))
            return fail(BC_ERR_INVALID_ARG, "non-finite update coefficient");
    }
    double c[BC_MAX_K];
    int m = 0;
    s = window_weights(h, t_new, c, &m);
    if (s != BC_OK) return s;

    const uint64_t out_eb = elem_bytes(out_dtype);
    const uint64_t x_bytes =
        euler ? static_cast<uint64_t>(h->numel[v_layer]) * elem_bytes(x_dtype) : 0;
    const uint64_t x0 = reinterpret_cast<uint64_t>(x);
    if (euler && h->overlaps_arena(x0, x_bytes))
        return fail(BC_ERR_INVALID_ARG, "x overlaps the cache arena");
    const uint64_t z0 = reinterpret_cast<uint64_t>(up.z);
    if (euler && up.z && (h->overlaps_arena(z0, x_bytes) || ranges_overlap(z0, x_bytes, x0, x_bytes)))
        return fail(BC_ERR_INVALID_ARG, "z overlaps the cache arena or x");

    auto &entries = h->scratch_entries;
    entries.clear();
    int euler_index = -1;
    for (int l = 0; l < h->n_layers; ++l) {
        void *o = out_ptrs[l];
        if (!o && !(euler && l == v_layer)) continue;
        const uint64_t ob = static_cast<uint64_t>(h->numel[l]) * out_eb;
        if (o) {
            if (!aligned16(o)) return fail(BC_ERR_ALIGNMENT, "output %d not 16-byte aligned", l);
            const uint64_t p = reinterpret_cast<uint64_t>(o);
            if (h->overlaps_arena(p, ob))
                return fail(BC_ERR_INVALID_ARG, "output %d overlaps the cache arena", l);
            if (euler && ranges_overlap(p, ob, x0, x_bytes))
                return fail(BC_ERR_INVALID_ARG, "output %d aliases x", l);
            if (euler && up.z && ranges_overlap(p, ob, z0, x_bytes))
                return fail(BC_ERR_INVALID_ARG, "output %d aliases z", l);
        }
        if (euler && l == v_layer) euler_index = static_cast<int>(entries.size());
        bc::LayerEntry e{};
        e.src = h->offset[l];
        e.dst = reinterpret_cast<uint64_t>(o);
        e.numel = h->numel[l];
        entries.push_back(e);
    }

    bc::LaunchPlan plan{};
    for (int j = 0; j < BC_MAX_K; ++j)
        plan.slot[j] = j < m ? reinterpret_cast<uint64_t>(h->slot_base(h->slot_of_node(j))) : 0;
    bc::kernel_weights(c, m, plan.w, &plan.scale);
    plan.K = m;
    plan.in_dtype = h->dtype;
    plan.out_dtype = out_dtype;
    plan.ca = static_cast<float>(up.ca);
    plan.cb = static_cast<float>(up.cb);
    plan.cc = static_cast<float>(up.cc);
    plan.euler_layer = euler_index;
    plan.x_dtype = x_dtype;
    plan.x = x0;
    plan.z = up.z ? z0 : 0;
    plan.status = h->status;
    plan.inject = h->inject_next ? 1 : 0;
    plan.kernel = h->kernel;
    plan.layers = entries.data();
    plan.n_layers = static_cast<int>(entries.size());

    if (plan.n_layers > 0) {
        DeviceGuard g(h->device);
        if (!g.ok) return fail(BC_ERR_CUDA, "cannot select the cache's device");
        plan.table = table_for(h->table, plan.n_layers, stream);
        const int err = bc::launch_forecast(plan, stream, &h->stats.kernel_launches,
                                                &h->stats.pipeline_launches);
        h->inject_next = false;
        if (err != cudaSuccess) return cuda_fail(err, "forecast launch");
    }
    ++h->stats.forecasts;
    h->stats.memo_hits = h->memo.hits;
    h->stats.memo_misses = h->memo.misses;
    return BC_OK;
}

}  // namespace

// ======================================================================= C ABI
extern "C" {

int bc_version(void) { return 10000; }

const char *bc_status_string(bc_status s) {
    switch (s) {
    case BC_OK: return "ok";
    case BC_ERR_INVALID_ARG: return "invalid argument";
    case BC_ERR_ALIGNMENT: return "device pointer not 16-byte aligned";
    case BC_ERR_OOM: return "device allocation failed";
    case BC_ERR_CUDA: return "CUDA runtime error";
    case BC_ERR_NOT_READY: return "no feature pushed yet";
    case BC_ERR_DUPLICATE_NODE: return "timestep already in the cache window";
    case BC_ERR_DEGENERATE_WEIGHTS: return "weight normaliser vanishes";
    case BC_ERR_BAD_HANDLE: return "bad handle";
    case BC_ERR_DEVICE_TIMEOUT: return "a device pipeline wait timed out";
    }
    return "unknown status";
}

const char *bc_last_error(void) { return t_last_error.c_str(); }

void bc_params_default(bc_params *p) {
    if (!p) return;
    p->mode = BC_MODE_PAPER;
    p->delta = 0.0;
    p->lambda = 0.0;
    p->clip_C = 10.0;
    p->eta = 1e-12;
}

bc_status bc_solve(const double *nodes, int m, double t, const bc_params *p, double *c_out) {
    t_last_error.clear();
    try {
        bc_params prm;
        bc_params_default(&prm);
        if (p) prm = *p;
        if (!nodes || !c_out) return fail(BC_ERR_INVALID_ARG, "null pointer");
        if (m < 1 || m > BC_MAX_K) return fail(BC_ERR_INVALID_ARG, "m=%d outside 1..%d", m, BC_MAX_K);
        if (!params_valid(prm)) return fail(BC_ERR_INVALID_ARG, "invalid weight parameters");
        if (!std::isfinite(t)) return fail(BC_ERR_INVALID_ARG, "non-finite target timestep");
        double d[BC_MAX_K];
        for (int j = 0; j < m; ++j) {
            if (!std::isfinite(nodes[j])) return fail(BC_ERR_INVALID_ARG, "non-finite node");
            d[j] = t - nodes[j];
        }
        return solve_from_differences(d, m, prm, c_out);
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_cache_bytes_for(const int64_t *numels, int n_layers, int K, bc_dtype dtype,
                             int64_t *bytes) {
    t_last_error.clear();
    try {
        if (!bytes) return fail(BC_ERR_INVALID_ARG, "bytes is NULL");
        uint64_t slot = 0;
        bc_status s = layout(numels, n_layers, K, dtype, nullptr, &slot);
        if (s != BC_OK) return s;
        *bytes = static_cast<int64_t>(slot * static_cast<uint64_t>(K));
        return BC_OK;
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_cache_create(const int64_t *numels, int n_layers, int K, bc_dtype dtype,
                          const bc_params *p, bc_handle *out) {
    t_last_error.clear();
    if (!out) return fail(BC_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    bc_cache *h = nullptr;
    try {
        bc_params prm;
        bc_params_default(&prm);
        if (p) prm = *p;
        if (!params_valid(prm)) return fail(BC_ERR_INVALID_ARG, "invalid weight parameters");
        std::vector<uint64_t> offs;
        uint64_t slot = 0;
        bc_status s = layout(numels, n_layers, K, dtype, &offs, &slot);
        if (s != BC_OK) return s;
        h = new bc_cache();
        h->n_layers = n_layers;
        h->K = K;
        h->dtype = dtype;
        h->params = prm;
        h->numel.assign(numels, numels + n_layers);
        h->offset = std::move(offs);
        h->slot_bytes = slot;
        h->arena_bytes = slot * static_cast<uint64_t>(K);
        if (cudaGetDevice(&h->device) != cudaSuccess) {
            delete h;
            cudaGetLastError();
            return fail(BC_ERR_CUDA, "no CUDA device");
        }
        if (h->arena_bytes > 0) {
            void *mem = nullptr;
            cudaError_t e = cudaMalloc(&mem, h->arena_bytes);
            if (e != cudaSuccess) {
                cudaGetLastError();
                delete h;
                if (e == cudaErrorMemoryAllocation)
                    return fail(BC_ERR_OOM, "cannot allocate %llu bytes of cache",
                                static_cast<unsigned long long>(slot * K));
                return cuda_fail(e, "cudaMalloc");
            }
            h->arena = static_cast<char *>(mem);
        }
        {
            void *mem = nullptr;
            // reduction scratch followed by the 4-byte status word (padded to 256 bytes)
            const size_t scratch = sizeof(double) * 2 * bc::kProbeMaxCtas;
            cudaError_t e = cudaMalloc(&mem, scratch + 256);
            if (e == cudaSuccess) e = cudaMemset(static_cast<char *>(mem) + scratch, 0, 256);
            if (e != cudaSuccess) {
                if (mem) cudaFree(mem);
                cudaGetLastError();
                if (h->arena) cudaFree(h->arena);
                delete h;
                return e == cudaErrorMemoryAllocation ? fail(BC_ERR_OOM, "probe scratch")
                                                      : cuda_fail(e, "cudaMalloc");
            }
            h->probe_partials = static_cast<double *>(mem);
            h->status = reinterpret_cast<uint32_t *>(static_cast<char *>(mem) + scratch);
        }
        if (n_layers > bc::kLayersLarge) {
            s = alloc_table(h);
            if (s != BC_OK) {
                free_device(h);
                delete h;
                return s;
            }
        }
        {
            std::lock_guard<std::mutex> lk(g_registry_mu);
            g_registry.insert(h);
        }
        *out = h;
        return BC_OK;
    } catch (const std::bad_alloc &) {
        delete h;
        return fail(BC_ERR_OOM, "host allocation failed");
    } catch (...) {
        delete h;
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_cache_destroy(bc_handle h) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    {
        std::lock_guard<std::mutex> lk(g_registry_mu);
        g_registry.erase(h);
    }
    h->magic = 0;
    bc_status rc = BC_OK;
    if (h->arena || h->probe_partials || h->table.dev || h->push_table.dev) {
        DeviceGuard g(h->device);
        cudaError_t e = cudaDeviceSynchronize();
        if (e == cudaSuccess) e = free_device(h);
        if (e != cudaSuccess) rc = cuda_fail(e, "cudaFree");
    }
    delete h;
    return rc;
}

bc_status bc_cache_info(bc_handle h, int *n_layers, int *K, int *dtype) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (n_layers) *n_layers = h->n_layers;
    if (K) *K = h->K;
    if (dtype) *dtype = static_cast<int>(h->dtype);
    return BC_OK;
}

bc_status bc_cache_bytes(bc_handle h, int64_t *bytes) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!bytes) return fail(BC_ERR_INVALID_ARG, "bytes is NULL");
    *bytes = static_cast<int64_t>(h->arena_bytes);
    return BC_OK;
}

bc_status bc_cache_set_params(bc_handle h, const bc_params *p) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    bc_params prm;
    bc_params_default(&prm);
    if (p) prm = *p;
    if (!params_valid(prm)) return fail(BC_ERR_INVALID_ARG, "invalid weight parameters");
    h->params = prm;
    h->memo.table.clear();
    return BC_OK;
}

bc_status bc_cache_set_kernel(bc_handle h, int kernel) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (kernel != BC_KERNEL_AUTO && kernel != BC_KERNEL_REGISTER && kernel != BC_KERNEL_PIPELINE)
        return fail(BC_ERR_INVALID_ARG, "unknown kernel choice %d", kernel);
    h->kernel = kernel;
    return BC_OK;
}

bc_status bc_cache_reset(bc_handle h) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    h->head = -1;
    h->count = 0;
    return BC_OK;
}

bc_status bc_cache_push(bc_handle h, const void *const *layer_ptrs, double t, void *stream) {
    t_last_error.clear();
    try {
        bc_status s = check_handle(h);
        if (s != BC_OK) return s;
        if (!layer_ptrs) return fail(BC_ERR_INVALID_ARG, "layer_ptrs is NULL");
        s = check_new_node(h, t);
        if (s != BC_OK) return s;
        const int next = (h->head + 1) % h->K;
        const uint64_t eb = elem_bytes(h->dtype);
        auto &entries = h->scratch_entries;
        entries.clear();
        for (int l = 0; l < h->n_layers; ++l) {
            if (h->numel[l] == 0) continue;
            const void *src = layer_ptrs[l];
            if (!src) return fail(BC_ERR_INVALID_ARG, "layer %d source is NULL", l);
            if (!aligned16(src)) return fail(BC_ERR_ALIGNMENT, "layer %d source not 16-byte aligned", l);
            if (h->overlaps_arena(reinterpret_cast<uint64_t>(src), h->numel[l] * eb))
                return fail(BC_ERR_INVALID_ARG, "layer %d source overlaps the cache arena", l);
            bc::LayerEntry e{};
            e.src = reinterpret_cast<uint64_t>(src);
            e.dst = h->offset[l];
            e.numel = h->numel[l];
            entries.push_back(e);
        }
        if (!entries.empty()) {
            DeviceGuard g(h->device);
            if (!g.ok) return fail(BC_ERR_CUDA, "cannot select the cache's device");
            bc::CopyOptions opt{h->kernel, h->status, h->inject_next_push ? 1 : 0,
                                table_for(h->push_table, static_cast<int>(entries.size()),
                                          stream),
                                reinterpret_cast<uint64_t>(h->slot_base(next))};
            const int err = bc::launch_copy(entries.data(), static_cast<int>(entries.size()),
                                            h->dtype, opt, stream, &h->stats.kernel_launches,
                                            &h->stats.pipeline_launches);
            h->inject_next_push = false;
            if (err != cudaSuccess) return cuda_fail(err, "push copy launch");
        }
        rotate_in(h, t);
        return BC_OK;
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_cache_push_flat(bc_handle h, const void *src, double t, void *stream) {
    t_last_error.clear();
    try {
        bc_status s = check_handle(h);
        if (s != BC_OK) return s;
        if (!src) return fail(BC_ERR_INVALID_ARG, "src is NULL");
        if (!aligned16(src)) return fail(BC_ERR_ALIGNMENT, "src is not 16-byte aligned");
        if (h->overlaps_arena(reinterpret_cast<uint64_t>(src), h->slot_bytes))
            return fail(BC_ERR_INVALID_ARG, "src overlaps the cache arena");
        s = check_new_node(h, t);
        if (s != BC_OK) return s;
        if (h->slot_bytes > 0) {
            const int next = (h->head + 1) % h->K;
            bc::LayerEntry e{};
            e.src = reinterpret_cast<uint64_t>(src);
            e.dst = 0;
            e.numel = static_cast<int64_t>(h->slot_bytes / elem_bytes(h->dtype));
            DeviceGuard g(h->device);
            if (!g.ok) return fail(BC_ERR_CUDA, "cannot select the cache's device");
            bc::CopyOptions opt{h->kernel, h->status, h->inject_next_push ? 1 : 0, nullptr,
                                reinterpret_cast<uint64_t>(h->slot_base(next))};
            const int err = bc::launch_copy(&e, 1, h->dtype, opt, stream,
                                            &h->stats.kernel_launches,
                                            &h->stats.pipeline_launches);
            h->inject_next_push = false;
            if (err != cudaSuccess) return cuda_fail(err, "push copy launch");
        }
        rotate_in(h, t);
        return BC_OK;
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_cache_next_slot_ptrs(bc_handle h, void **out_ptrs) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!out_ptrs) return fail(BC_ERR_INVALID_ARG, "out_ptrs is NULL");
    const int next = (h->head + 1) % h->K;
    for (int l = 0; l < h->n_layers; ++l) out_ptrs[l] = h->slot_base(next) + h->offset[l];
    return BC_OK;
}

bc_status bc_cache_commit(bc_handle h, double t) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    s = check_new_node(h, t);
    if (s != BC_OK) return s;
    rotate_in(h, t);
    return BC_OK;
}

bc_status bc_cache_nodes(bc_handle h, double *nodes_out, int *m_out) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!nodes_out || !m_out) return fail(BC_ERR_INVALID_ARG, "null pointer");
    for (int j = 0; j < h->count; ++j) nodes_out[j] = h->node_t[h->slot_of_node(j)];
    *m_out = h->count;
    return BC_OK;
}

bc_status bc_cache_slot_ptrs(bc_handle h, int j, void **out_ptrs) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!out_ptrs) return fail(BC_ERR_INVALID_ARG, "out_ptrs is NULL");
    if (j < 0 || j >= h->count) return fail(BC_ERR_INVALID_ARG, "node %d is not live", j);
    char *base = h->slot_base(h->slot_of_node(j));
    for (int l = 0; l < h->n_layers; ++l) out_ptrs[l] = base + h->offset[l];
    return BC_OK;
}

bc_status bc_coefficients(bc_handle h, double t_new, double *c_out, int *m_out) {
    t_last_error.clear();
    try {
        bc_status s = check_handle(h);
        if (s != BC_OK) return s;
        if (!c_out || !m_out) return fail(BC_ERR_INVALID_ARG, "null pointer");
        s = window_weights(h, t_new, c_out, m_out);
        h->stats.memo_hits = h->memo.hits;
        h->stats.memo_misses = h->memo.misses;
        return s;
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_forecast(bc_handle h, double t_new, void *const *out_ptrs, bc_dtype out_dtype,
                      void *stream) {
    t_last_error.clear();
    try {
        return forecast_impl(h, t_new, out_ptrs, out_dtype, Update{}, stream);
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_forecast_step(bc_handle h, double t_new, double dt, void *const *out_ptrs,
                           bc_dtype out_dtype, int v_layer, void *x, bc_dtype x_dtype,
                           void *stream) {
    t_last_error.clear();
    try {
        if (v_layer < 0) return fail(BC_ERR_INVALID_ARG, "v_layer must name a cached layer");
        if (!std::isfinite(dt)) return fail(BC_ERR_INVALID_ARG, "non-finite dt");
        Update up;
        up.ca = 1.0;
        up.cb = dt;
        up.v_layer = v_layer;
        up.x = x;
        up.x_dtype = x_dtype;
        return forecast_impl(h, t_new, out_ptrs, out_dtype, up, stream);
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_forecast_update(bc_handle h, double t_new, double a, double b, double c,
                             void *const *out_ptrs, bc_dtype out_dtype, int v_layer, void *x,
                             bc_dtype x_dtype, const void *z, void *stream) {
    t_last_error.clear();
    try {
        if (v_layer < 0) return fail(BC_ERR_INVALID_ARG, "v_layer must name a cached layer");
        Update up;
        up.ca = a;
        up.cb = b;
        up.cc = c;
        up.v_layer = v_layer;
        up.x = x;
        up.x_dtype = x_dtype;
        up.z = z;
        return forecast_impl(h, t_new, out_ptrs, out_dtype, up, stream);
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_ddpm_coefficients(double alpha_t, double alpha_bar_t, double *a, double *b,
                               double *c) {
    t_last_error.clear();
    if (!a || !b || !c) return fail(BC_ERR_INVALID_ARG, "null pointer");
    if (!(alpha_t > 0.0 && alpha_t <= 1.0) || !(alpha_bar_t > 0.0 && alpha_bar_t < 1.0))
        return fail(BC_ERR_INVALID_ARG, "need 0 < alpha_t <= 1 and 0 < alpha_bar_t < 1");
    // Eq. 3: mu = (x_t - (1 - alpha_t) / sqrt(1 - alpha_bar_t) * eps) / sqrt(alpha_t);
    // Eq. 2: x_{t-1} ~ N(mu, beta_t I) with beta_t = 1 - alpha_t (the noise scale of Eq. 1).
    const double ra = std::sqrt(alpha_t);
    *a = 1.0 / ra;
    *b = -(1.0 - alpha_t) / (ra * std::sqrt(1.0 - alpha_bar_t));
    *c = std::sqrt(1.0 - alpha_t);
    return BC_OK;
}

bc_status bc_ddim_coefficients(double alpha_bar_t, double alpha_bar_prev, double eta, double *a,
                               double *b, double *c) {
    t_last_error.clear();
    if (!a || !b || !c) return fail(BC_ERR_INVALID_ARG, "null pointer");
    if (!(alpha_bar_t > 0.0 && alpha_bar_t < 1.0) ||
        !(alpha_bar_prev >= alpha_bar_t && alpha_bar_prev <= 1.0) || !(eta >= 0.0) ||
        !std::isfinite(eta))
        return fail(BC_ERR_INVALID_ARG,
                    "need 0 < alpha_bar_t < 1, alpha_bar_t <= alpha_bar_prev <= 1, eta >= 0");
    // DDIM (Song, Meng and Ermon, ICLR 2021, generative process with parameter eta):
    //   x_prev = sqrt(ab_prev) * (x_t - sqrt(1 - ab_t) eps) / sqrt(ab_t)
    //            + sqrt(1 - ab_prev - sigma^2) eps + sigma z,
    //   sigma = eta sqrt((1 - ab_prev) / (1 - ab_t)) sqrt(1 - ab_t / ab_prev).
    const double sigma = eta * std::sqrt((1.0 - alpha_bar_prev) / (1.0 - alpha_bar_t)) *
                         std::sqrt(1.0 - alpha_bar_t / alpha_bar_prev);
    const double dir = 1.0 - alpha_bar_prev - sigma * sigma;
    if (dir < 0.0) return fail(BC_ERR_INVALID_ARG, "eta too large: negative direction variance");
    *a = std::sqrt(alpha_bar_prev / alpha_bar_t);
    *b = std::sqrt(dir) - std::sqrt(alpha_bar_prev * (1.0 - alpha_bar_t) / alpha_bar_t);
    *c = sigma;
    return BC_OK;
}

bc_status bc_cache_layout(bc_handle h, int64_t *offsets) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!offsets) return fail(BC_ERR_INVALID_ARG, "offsets is NULL");
    for (int l = 0; l < h->n_layers; ++l) offsets[l] = static_cast<int64_t>(h->offset[l]);
    offsets[h->n_layers] = static_cast<int64_t>(h->slot_bytes);
    return BC_OK;
}

bc_status bc_forecast_flat(bc_handle h, double t_new, void *out, void *stream) {
    t_last_error.clear();
    try {
        bc_status s = check_handle(h);
        if (s != BC_OK) return s;
        if (!out) return fail(BC_ERR_INVALID_ARG, "out is NULL");
        if (!aligned16(out)) return fail(BC_ERR_ALIGNMENT, "out is not 16-byte aligned");
        if (h->overlaps_arena(reinterpret_cast<uint64_t>(out), h->slot_bytes))
            return fail(BC_ERR_INVALID_ARG, "out overlaps the cache arena");
        double c[BC_MAX_K];
        int m = 0;
        s = window_weights(h, t_new, c, &m);
        if (s != BC_OK) return s;
        if (h->slot_bytes > 0) {
            bc::LayerEntry e{};
            e.src = 0;
            e.dst = reinterpret_cast<uint64_t>(out);
            e.numel = static_cast<int64_t>(h->slot_bytes / elem_bytes(h->dtype));
            bc::LaunchPlan plan{};
            for (int j = 0; j < BC_MAX_K; ++j)
                plan.slot[j] =
                    j < m ? reinterpret_cast<uint64_t>(h->slot_base(h->slot_of_node(j))) : 0;
            bc::kernel_weights(c, m, plan.w, &plan.scale);
            plan.K = m;
            plan.in_dtype = h->dtype;
            plan.out_dtype = h->dtype;
            plan.euler_layer = -1;
            plan.layers = &e;
            plan.n_layers = 1;
            plan.status = h->status;
            plan.inject = h->inject_next ? 1 : 0;
            plan.kernel = h->kernel;
            DeviceGuard g(h->device);
            if (!g.ok) return fail(BC_ERR_CUDA, "cannot select the cache's device");
            const int err = bc::launch_forecast(plan, stream, &h->stats.kernel_launches,
                                                &h->stats.pipeline_launches);
            h->inject_next = false;
            if (err != cudaSuccess) return cuda_fail(err, "forecast launch");
        }
        ++h->stats.forecasts;
        h->stats.memo_hits = h->memo.hits;
        h->stats.memo_misses = h->memo.misses;
        return BC_OK;
    } catch (...) {
        return fail(BC_ERR_INVALID_ARG, "internal exception");
    }
}

bc_status bc_schedule_equal(int n_steps, int interval, int K, uint8_t *is_full) {
    t_last_error.clear();
    if (n_steps < 0 || interval < 1 || K < 0 || (n_steps > 0 && !is_full))
        return fail(BC_ERR_INVALID_ARG, "need n_steps >= 0, interval >= 1, K >= 0");
    for (int i = 0; i < n_steps; ++i) is_full[i] = (i < K || i % interval == 0) ? 1 : 0;
    return BC_OK;
}

bc_status bc_adaptive_init(bc_adaptive *st, double threshold, int K) {
    t_last_error.clear();
    if (!st) return fail(BC_ERR_INVALID_ARG, "state is NULL");
    if (!(threshold >= 0.0) || !std::isfinite(threshold) || K < 0)
        return fail(BC_ERR_INVALID_ARG, "need a finite threshold >= 0 and K >= 0");
    st->threshold = threshold;
    st->accumulated = 0.0;
    st->K = K;
    st->steps = 0;
    st->full_steps = 0;
    return BC_OK;
}

bc_status bc_adaptive_decide(bc_adaptive *st, double drift, int *run_full) {
    t_last_error.clear();
    if (!st || !run_full) return fail(BC_ERR_INVALID_ARG, "null pointer");
    if (!(drift >= 0.0)) return fail(BC_ERR_INVALID_ARG, "drift must be >= 0 (and not NaN)");
    int full;
    if (st->steps < st->K) {
        full = 1;  // the window is still filling
    } else {
        st->accumulated += drift;
        full = st->accumulated >= st->threshold ? 1 : 0;
    }
    if (full) {
        st->accumulated = 0.0;
        ++st->full_steps;
    }
    ++st->steps;
    *run_full = full;
    return BC_OK;
}

bc_status bc_probe_drift(bc_handle h, const void *cur, const void *prev, int64_t n,
                         bc_dtype dtype, double *out, void *stream) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!out || n < 0 || (n > 0 && (!cur || !prev)))
        return fail(BC_ERR_INVALID_ARG, "need device cur, prev (n elements) and out[3]");
    if (!dtype_valid(dtype)) return fail(BC_ERR_INVALID_ARG, "unknown dtype");
    if (!aligned16(cur) || !aligned16(prev))
        return fail(BC_ERR_ALIGNMENT, "probe tensors must be 16-byte aligned");
    DeviceGuard g(h->device);
    if (!g.ok) return fail(BC_ERR_CUDA, "cannot select the cache's device");
    bc::DriftOptions opt{h->kernel, h->status, h->inject_next_drift ? 1 : 0};
    const int err = bc::launch_drift(cur, prev, n, dtype, h->probe_partials, bc::kProbeMaxCtas,
                                     out, opt, stream, &h->stats.kernel_launches,
                                     &h->stats.pipeline_launches);
    h->inject_next_drift = false;
    if (err != cudaSuccess) return cuda_fail(err, "drift launch");
    return BC_OK;
}

bc_status bc_probe_drift_noalloc(const void *cur, const void *prev, int64_t n, bc_dtype dtype,
                                 double *out, void *stream) {
    t_last_error.clear();
    if (!out || n < 0 || (n > 0 && (!cur || !prev)))
        return fail(BC_ERR_INVALID_ARG, "need device cur, prev (n elements) and out[3]");
    if (!dtype_valid(dtype)) return fail(BC_ERR_INVALID_ARG, "unknown dtype");
    const int64_t max_n = bc::static_drift_max_elems(dtype);
    if (n > max_n)
        return fail(BC_ERR_INVALID_ARG,
                    "n = %lld exceeds the no-allocation maximum of %lld elements (1 GiB per "
                    "tensor); use bc_probe_drift with a cache handle",
                    static_cast<long long>(n), static_cast<long long>(max_n));
    if (!aligned16(cur) || !aligned16(prev))
        return fail(BC_ERR_ALIGNMENT, "probe tensors must be 16-byte aligned");
    int64_t launches = 0;
    const int err = bc::launch_drift_static(cur, prev, n, dtype, out, stream, &launches);
    if (err != cudaSuccess) return cuda_fail(err, "no-allocation drift");
    return BC_OK;
}

bc_status bc_cache_check(bc_handle h) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    DeviceGuard g(h->device);
    if (!g.ok) return fail(BC_ERR_CUDA, "cannot select the cache's device");
    uint32_t word = 0;
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess) e = cudaMemcpy(&word, h->status, sizeof word, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "reading the device status");
    if (word == 0) return BC_OK;
    e = cudaMemset(h->status, 0, sizeof word);
    if (e != cudaSuccess) return cuda_fail(e, "clearing the device status");
    return fail(BC_ERR_DEVICE_TIMEOUT,
                "a launch gave up waiting for its shared-memory pipeline (status 0x%x); "
                "outputs of launches since the last check may be incomplete", word);
}

bc_status bc_cache_inject_fault(bc_handle h, int what) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (what < 0 || what > 3) return fail(BC_ERR_INVALID_ARG, "unknown fault %d", what);
    h->inject_next = (what == 1);
    h->inject_next_drift = (what == 2);
    h->inject_next_push = (what == 3);
    return BC_OK;
}

bc_status bc_cache_stats(bc_handle h, bc_stats *out) {
    t_last_error.clear();
    bc_status s = check_handle(h);
    if (s != BC_OK) return s;
    if (!out) return fail(BC_ERR_INVALID_ARG, "out is NULL");
    h->stats.memo_hits = h->memo.hits;
    h->stats.memo_misses = h->memo.misses;
    h->stats.table_uploads = h->table.uploads + h->push_table.uploads;
    *out = h->stats;
    return BC_OK;
}

}  // extern "C"
