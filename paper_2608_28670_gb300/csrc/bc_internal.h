// bc_internal.h -- the layout shared by the host side (bc_host.cpp) and the kernels
// (bc_forecast.cu).  Not part of the public ABI.
#pragma once

#include <cstdint>

#include "barycache.h"

namespace bc {

// Tuning constants of the streaming kernels.  They are compile-time so that the compiler
// unrolls every per-thread loop.  The defaults are the best of a sweep on GB300 (t2v
// workload, K = 2..4): 32-byte history loads, 256-thread CTAs, two CTAs per SM, two
// vectors per thread and slot (four at K = 4).  The BC_* macros exist to build variants
// for tuning sweeps.
#ifndef BC_VEC_BYTES
#define BC_VEC_BYTES 32      // bytes per history vector load (16 or 32)
#endif
#ifndef BC_VECS_PER_THREAD
#define BC_VECS_PER_THREAD 0 // 0: per-K default (vecs_per_thread below)
#endif
#ifndef BC_THREADS
#define BC_THREADS 256
#endif
#ifndef BC_L2_EVICT_FIRST
#define BC_L2_EVICT_FIRST 0  // 1: history loads carry an L2 evict-first cache policy
#endif
#ifndef BC_CTAS_PER_SM
#define BC_CTAS_PER_SM 2     // 0: as many as the occupancy calculator allows
#endif

// Elements of a layer are processed in tiles of kThreads x VPT vectors of kVecBytes
// (VPT = vectors per thread, per history slot); a tile never straddles two layers.
constexpr int kVecBytes = BC_VEC_BYTES;
constexpr int kThreads = BC_THREADS;
static_assert(kVecBytes == 16 || kVecBytes == 32, "vector loads are 16 or 32 bytes");

// Independent vectors per thread and history slot for a K-term forecast (register kernel).
template <int K>
constexpr int kVecsPerThreadFor = BC_VECS_PER_THREAD > 0 ? BC_VECS_PER_THREAD : (K >= 4 ? 4 : 2);
// The push copy streams one source: four 16-byte vectors per thread.
constexpr int kCopyVecsPerThread = 4;

// Layers per launch carried in the kernel's parameter block.  The whole table travels as
// a __grid_constant__ parameter, so a forecast of up to kLayersLarge layers needs no
// device-side table and no host-to-device copy of its own; three table sizes keep the block
// small for the usual few-dozen-layer caches.  A forecast over more layers runs as one
// launch that reads its table from a per-handle device copy (DeviceTable); while its stream
// is being captured into a CUDA graph it issues one parameter-block launch per kLayersLarge
// layers instead, so that the graph holds every table it replays.  Push copies work the same
// way with a table of their own.
constexpr int kLayersSmall = 8;
constexpr int kLayersMedium = 64;
constexpr int kLayersLarge = 1016;

struct LayerEntry {        // 32 bytes
    uint64_t src;          // forecast: byte offset of the layer in every slot;
                           // copy: absolute source address
    uint64_t dst;          // forecast: output address; copy: byte offset of the layer in
                           // the destination slot (its base travels in the launch)
    int64_t numel;         // elements in the layer
    int64_t tile_end;      // exclusive prefix sum of tiles up to this layer
};

// Where a CTA's contiguous tile range starts: the layer holding its first tile and that
// layer's first tile.  Computed by the host for launches whose table is in device memory, so
// that no CTA starts with a binary search of dependent global loads.
struct CtaStart {
    int64_t first;         // first tile of `layer`
    int32_t layer;
    int32_t pad;
};
constexpr int kMaxStartCtas = 512;

template <int CAP>
struct ForecastArgs {
    uint64_t slot[BC_MAX_K];  // slot base address of node j (j = 0 newest)
    float w[BC_MAX_K];        // weights W_j rounded to fp32, divided by `scale`
    float scale;              // power of two >= sum_j |W_j|: the forecast is scale * sum_j w_j F_j
    float ca, cb, cc;         // sampler update x <- ca x + cb v_hat + cc z (update layer)
    int32_t n_layers;
    int32_t euler_layer;      // index into the layer table of the update layer, or -1
    int32_t x_bf16;           // sampler state dtype (and z's): 1 = bf16, 0 = f32
    uint64_t x;               // sampler state address
    uint64_t z;               // noise address (0: no noise term)
    uint32_t *status;         // device status word: bit 0 = a pipeline wait timed out
    int32_t inject;           // test hook: leave the first pipeline stage unarmed
    int64_t total_tiles;
    const LayerEntry *table;  // CAP == 0: the layer table in device memory
    int32_t n_starts;         // CAP == 0: CTAs whose first layer is given in `start`
    CtaStart start[CAP > 0 ? 1 : kMaxStartCtas];  // CAP == 0: layer of each CTA's first tile
    LayerEntry layer[CAP > 0 ? CAP : 1];  // CAP > 0: the layer table itself
};

// Kernel parameter blocks may hold up to 32,764 bytes (CUDA 12.1 and later).
static_assert(sizeof(ForecastArgs<kLayersLarge>) <= 32764, "layer table exceeds the parameter block");

// ------------------------------------------------------------------ host side
// (Everything below is the launchers' host-side view; the kernels see only what is above.)

// A device-memory copy of a launch's layer table, for forecasts and pushes over more layers
// than the parameter block holds (caches of more than kLayersLarge layers have one for each).
// The table is uploaded with one cudaMemcpyAsync on the call's stream, and only when it
// differs from the previous upload: a sampler that reuses its buffers uploads once.  The
// pinned staging is a ring of kTableStaging buffers, each reused only after the copy that
// last read it has run (its event), so the host waits only if that many uploads with
// different tables are still queued ahead of the device.  An event recorded after every
// launch that reads the table makes the next call's stream wait (on the device) until that
// launch is done, before it rewrites the table or reads the copy queued ahead of it.
constexpr int kTableStaging = 4;
struct DeviceTable {
    LayerEntry *dev = nullptr;     // device, `capacity` entries
    LayerEntry *host = nullptr;    // pinned staging: kTableStaging x `capacity` entries
    int capacity = 0;
    int valid = 0;                 // entries of the last upload (0: none yet)
    int last = -1;                 // staging buffer of the last upload
    bool pending[kTableStaging] = {};        // an event was recorded after the buffer's copy
    void *uploaded[kTableStaging] = {};      // cudaEvent_t per staging buffer
    void *used = nullptr;          // cudaEvent_t recorded after the last launch that read `dev`
    bool used_recorded = false;
    int64_t uploads = 0;           // uploads so far
};

// Host-side view of one launch, independent of CAP.
struct LaunchPlan {
    uint64_t slot[BC_MAX_K];
    float w[BC_MAX_K];        // fp32 weights divided by `scale` (see kernel_weights)
    float scale;
    int K;                    // live nodes used (1..BC_MAX_K)
    bc_dtype in_dtype;
    bc_dtype out_dtype;
    float ca, cb, cc;
    int euler_layer;          // index into `layers`, or -1
    bc_dtype x_dtype;
    uint64_t x;
    uint64_t z;
    uint32_t *status;
    int inject;
    int kernel;               // bc_kernel choice: 0 auto, 1 register, 2 pipeline
    const LayerEntry *layers; // tile_end filled by the launcher
    int n_layers;
    DeviceTable *table;       // non-null: more than kLayersLarge layers go in one launch
};

// Kernel weights from the fp64 weights c[0..m-1]: each is rounded to fp32 once, and all are
// divided by the smallest power of two `scale` >= sum_j |fp32(c_j)| (at least 1).  The kernels
// accumulate sum_j w_j F_j and multiply by `scale` at the end.  Scaling by a power of two is
// exact, so wherever the unscaled fp32 sum neither overflows nor enters the subnormal range
// the result is bit for bit the unscaled one; what it buys is that no partial sum exceeds
// max_j |F_j| in magnitude, so finite inputs never overflow in fp32 where the exact
// combination (weights near (3, -3, 1) or (4, -6, 4, -1) on values near the bf16 or fp32
// maximum) is representable.
inline void kernel_weights(const double *c, int m, float *w, float *scale) {
    double sum = 0.0;
    for (int j = 0; j < m; ++j) {
        w[j] = static_cast<float>(c[j]);
        sum += w[j] < 0.0f ? -static_cast<double>(w[j]) : static_cast<double>(w[j]);
    }
    float s = 1.0f;
    while (static_cast<double>(s) < sum && s < 1073741824.0f) s *= 2.0f;
    for (int j = 0; j < m; ++j) w[j] /= s;
    for (int j = m; j < BC_MAX_K; ++j) w[j] = 0.0f;
    *scale = s;
}

// Tiles needed for `numel` elements of `elem_bytes` each, in vectors of `vec_bytes`,
// `tile_vecs` vectors per tile: ceil(numel / (vec_bytes / elem_bytes * tile_vecs)) (the
// vectors a layer needs, rounded up to whole tiles).  The table builders count many layers
// with one tile shape; every shipped shape holds a power of two of elements, so the count is
// a shift rather than a 64-bit division per layer.
struct TileCounter {
    int64_t per_tile;  // elements per tile
    int shift = -1;    // log2(per_tile) when it is a power of two
    TileCounter(int elem_bytes, int vec_bytes, int tile_vecs)
        : per_tile(static_cast<int64_t>(vec_bytes / elem_bytes) * tile_vecs) {
        if ((per_tile & (per_tile - 1)) == 0)
            for (shift = 0; (int64_t{1} << shift) < per_tile; ++shift) {
            }
    }
    int64_t operator()(int64_t numel) const {
        return shift >= 0 ? (numel + per_tile - 1) >> shift : (numel + per_tile - 1) / per_tile;
    }
};
inline int64_t tiles_for(int64_t numel, int elem_bytes, int vec_bytes, int tile_vecs) {
    return TileCounter(elem_bytes, vec_bytes, tile_vecs)(numel);
}

// Enqueue the grouped forecast: one launch, or with more than kLayersLarge layers and no
// device table one launch per group of kLayersLarge.  Returns the CUDA error of the last
// launch; *launches is incremented per launch, *pipeline_launches per launch of the
// shared-memory pipeline kernel.
int launch_forecast(const LaunchPlan &plan, void *stream, int64_t *launches,
                    int64_t *pipeline_launches);
// The same for a given number of live nodes (bc_forecast_k{1,2,3,4}.cu).
int launch_forecast_k1(const LaunchPlan &plan, void *stream, int64_t *launches,
                       int64_t *pipeline_launches);
int launch_forecast_k2(const LaunchPlan &plan, void *stream, int64_t *launches,
                       int64_t *pipeline_launches);
int launch_forecast_k3(const LaunchPlan &plan, void *stream, int64_t *launches,
                       int64_t *pipeline_launches);
int launch_forecast_k4(const LaunchPlan &plan, void *stream, int64_t *launches,
                       int64_t *pipeline_launches);

// Probe drift reduction (bc_probe.cu): at most kProbeMaxCtas partial pairs of scratch.
constexpr int kProbeMaxCtas = 1024;
int probe_ctas();
// The handle's side of a drift launch: kernel choice (bc_kernel), device status word and
// the test hook that leaves the pipeline's first stage unarmed.
struct DriftOptions {
    int kernel;
    uint32_t *status;
    int inject;
};
// Enqueue sum |cur - prev|, sum |prev| and their ratio into out[0..2] (device doubles),
// using partials[0 .. 2 * max_parts) as scratch.  Two launches; *pipeline_launches counts
// the shared-memory pipeline variant of the first.
int launch_drift(const void *cur, const void *prev, int64_t n, bc_dtype dtype, double *partials,
                 int max_parts, double *out, const DriftOptions &opt, void *stream,
                 int64_t *launches, int64_t *pipeline_launches);

// The no-allocation drift (bc_probe.cu): scratch is a file-scope device array of
// kStaticDriftMaxTiles partial pairs (256 KiB), one pair per tile of
// kStaticDriftTileGroups x 256 sixteen-byte groups of the input.
constexpr int64_t kStaticDriftMaxTiles = 16384;
constexpr int kStaticDriftTileGroups = 16;
// Largest probe (elements of dtype) the static scratch can reduce: 1 GiB per tensor.
int64_t static_drift_max_elems(bc_dtype dtype);
// Enqueue the same sums as launch_drift using the static scratch; the first call on a
// device looks up the array's address.  Two launches; *launches incremented per launch.
int launch_drift_static(const void *cur, const void *prev, int64_t n, bc_dtype dtype,
                        double *out, void *stream, int64_t *launches);

// Enqueue the grouped copy used by bc_cache_push (layers[].src absolute, .dst an offset in
// the destination slot opt.dst_base):
// the TMA bulk-copy pipeline for large pushes (or when pinned / injected), else the
// register copy.  *pipeline_launches counts the former.
struct CopyOptions {
    int kernel;               // bc_kernel
    uint32_t *status;         // device status word
    int inject;               // test hook: leave the pipeline's first stage unarmed
    DeviceTable *table;       // non-null: more than kLayersLarge layers go in one launch
    uint64_t dst_base;        // destination slot; layer l lands at dst_base + layers[l].dst
};
int launch_copy(const LayerEntry *layers, int n_layers, bc_dtype dtype, const CopyOptions &opt,
                void *stream, int64_t *launches, int64_t *pipeline_launches);

}  // namespace bc
