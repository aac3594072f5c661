// bc_internal.h -- the layout shared by the host side (bc_host.cpp) and the kernels
// (bc_forecast.cu).  Not part of the public ABI.
#pragma once

#include <cstdint>

#include "barycache.h"

namespace bc {

// Elements of a layer are processed in tiles of kTileVecs 16-byte vectors (kThreads
// threads x kVecsPerThread vectors); a tile never straddles two layers.
constexpr int kThreads = 256;
constexpr int kVecsPerThread = 4;
constexpr int kTileVecs = kThreads * kVecsPerThread;

// Layers per launch carried in the kernel's parameter block.  The whole table travels as
// a __grid_constant__ parameter, so a forecast needs no device-side scratch and no
// host-to-device copy of its own; caches with more layers issue one launch per group.
constexpr int kLayersSmall = 8;
constexpr int kLayersLarge = 240;

struct LayerEntry {        // 32 bytes
    uint64_t src;          // forecast: byte offset of the layer in every slot;
                           // copy: absolute source address
    uint64_t dst;          // output address (forecast) / slot address (copy)
    int64_t numel;         // elements in the layer
    int64_t tile_end;      // exclusive prefix sum of tiles up to this layer
};

template <int CAP>
struct ForecastArgs {
    uint64_t slot[BC_MAX_K];  // slot base address of node j (j = 0 newest)
    float w[BC_MAX_K];        // weights W_j rounded to fp32
    float dt;                 // Euler step (only for the Euler layer)
    int32_t n_layers;
    int32_t euler_layer;      // index into `layer`, or -1
    int32_t x_bf16;           // Euler state dtype: 1 = bf16, 0 = f32
    uint64_t x;               // Euler state address
    int64_t total_tiles;
    LayerEntry layer[CAP];
};

// Host-side view of one launch, independent of CAP.
struct LaunchPlan {
    uint64_t slot[BC_MAX_K];
    float w[BC_MAX_K];
    int K;                    // live nodes used (1..BC_MAX_K)
    bc_dtype in_dtype;
    bc_dtype out_dtype;
    float dt;
    int euler_layer;          // index into `layers`, or -1
    bc_dtype x_dtype;
    uint64_t x;
    const LayerEntry *layers; // tile_end filled by the launcher
    int n_layers;
};

// Tiles needed for `numel` elements of `elem_bytes` each.
inline int64_t tiles_for(int64_t numel, int elem_bytes) {
    const int64_t ev = 16 / elem_bytes;
    const int64_t vecs = (numel + ev - 1) / ev;
    return (vecs + kTileVecs - 1) / kTileVecs;
}

// Enqueue the grouped forecast (one launch per CAP-sized group of layers).  Returns the
// CUDA error of the last launch; *launches is incremented per launch.
int launch_forecast(const LaunchPlan &plan, void *stream, int64_t *launches);

// Enqueue the grouped copy used by bc_cache_push (layers[].src absolute, .dst absolute).
int launch_copy(const LayerEntry *layers, int n_layers, bc_dtype dtype, void *stream,
                int64_t *launches);

}  // namespace bc
