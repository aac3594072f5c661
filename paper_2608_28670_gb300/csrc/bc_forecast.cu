// bc_forecast.cu -- the push's grouped byte-exact copy (Eq. 6: a full step stores its
// features in the evicted slot) and the dispatch of the forecast by history length.
//
// Both copy kernels walk the same kind of layer table as the forecast (carried in the launch's
// parameter block, or for more than kLayersLarge layers in the handle's device table):
//   copy_tma_kernel  TMA bulk loads and stores through a three-stage shared-memory ring, one
//                    warp per SM (large pushes);
//   copy_kernel      16-byte register loads and stores at full occupancy (small pushes).
// Both move bytes, not values (NaN payloads and -0.0 survive), and handle a ragged end of
// fewer than 16 bytes with element accesses.  The forecast kernels are in
// bc_forecast_kernels.cuh, instantiated per history length by bc_forecast_k{1,2,3,4}.cu.
#include "bc_forecast_kernels.cuh"

namespace bc {
namespace {

// Grouped byte-exact copy for the push: layer.src -> slot[0] + layer.dst, numel elements of T.
// Always 16-byte vectors: the caller's source is only guaranteed 16-byte alignment.
template <class T, int CAP>
__global__ void __launch_bounds__(kThreads) copy_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int kVecsPerThread = kCopyVecsPerThread;
    constexpr int kTileVecs = kThreads * kVecsPerThread;
    constexpr int EV = 16 / T::kBytes;
    int l = 0;
    int64_t first = 0;
    if (blockIdx.x < a.total_tiles) find_layer(a, blockIdx.x, l, first);
    LayerEntry L = entry_of(a, l);
    for (int64_t tile = blockIdx.x; tile < a.total_tiles; tile += gridDim.x) {
        if constexpr (CAP == 0) {
            // device-memory table: a grid stride may cross many small layers, so search
            // instead of stepping through every entry
            if (tile >= L.tile_end) {
                find_layer(a, tile, l, first);
                L = entry_of(a, l);
            }
        } else {
            seek_layer(a, tile, l, first);
            L = a.layer[l];
        }
        const int64_t nvec = L.numel / EV;
        const int64_t v0 = (tile - first) * kTileVecs + threadIdx.x;
        const char *src = reinterpret_cast<const char *>(L.src);
        char *dst = reinterpret_cast<char *>(a.slot[0] + L.dst);
        uint4 r[kVecsPerThread];
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) r[u] = ld_stream16(src + v * 16);
        }
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) st_stream16(dst + v * 16, r[u]);
        }
        const int rem = static_cast<int>(L.numel - nvec * EV);
        if (rem != 0 && tile == L.tile_end - 1 && static_cast<int>(threadIdx.x) < rem) {
            const int64_t e = nvec * EV + threadIdx.x;
            using S = typename T::store_t;
            reinterpret_cast<S *>(dst)[e] = reinterpret_cast<const S *>(src)[e];
        }
    }
}

// Grouped byte-exact copy through shared memory by TMA bulk copies (large pushes).  One
// warp per SM walks a contiguous range of tiles; lane 0 loads tile i into a ring stage
// (global -> shared, completing on the stage's mbarrier), writes it out with a bulk store
// (shared -> global, a bulk async-group) and refills the stage of tile i - 1 with tile
// i - 1 + kCopyStages once that tile's store has finished reading shared memory.  The
// ragged end of a layer (fewer than 16 bytes) is copied by the lanes.  Waits on the
// mbarriers are bounded as in the forecast pipeline; a CTA that gives up sets the status
// word, drains what it issued and returns.  Pushing the 43.8 GB video slot: 6.99 TB/s with
// three 32 KiB stages (register copy 6.39; stages x KiB: 4 x 32 6.63, 6 x 32 6.50,
// 2 x 32 4.96, 3 x 24 6.49, 3 x 40 6.85, 3 x 48 6.66, 8 x 16 6.30, 2 x 64 6.43; two
// CTAs per SM of 4 x 16 / 3 x 32 / 6 x 16: 6.56 / 6.52 / 6.49).
#ifndef BC_COPY_STAGES
#define BC_COPY_STAGES 3
#endif
#ifndef BC_COPY_TILE_BYTES
#define BC_COPY_TILE_BYTES 32768
#endif
#ifndef BC_COPY_CTAS_PER_SM
#define BC_COPY_CTAS_PER_SM 1
#endif
constexpr int kCopyStages = BC_COPY_STAGES;
constexpr int kCopyTileBytes = BC_COPY_TILE_BYTES;
constexpr int kCopySmemBytes = kCopyStages * kCopyTileBytes;
constexpr int kCopyMinTilesPerCta = 16;
constexpr int kCopyTmaThreads = 32;

template <class T, int CAP>
__global__ void __launch_bounds__(kCopyTmaThreads)
    copy_tma_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int S = kCopyStages;
    constexpr int kTileGroups = kCopyTileBytes / 16;
    constexpr int EV = 16 / T::kBytes;
    extern __shared__ __align__(128) unsigned char stage_mem[];
    __shared__ __align__(8) uint64_t full[S];
    const int lane = static_cast<int>(threadIdx.x);
    const int64_t per_cta = (a.total_tiles + gridDim.x - 1) / gridDim.x;
    const int64_t t_lo = static_cast<int64_t>(blockIdx.x) * per_cta;
    const int64_t t_hi = t_lo + per_cta < a.total_tiles ? t_lo + per_cta : a.total_tiles;
    if (t_lo >= t_hi) return;
    if (lane == 0) {
        for (int i = 0; i < S; ++i) mbar_init(&full[i], 1);
        mbar_init_fence();
    }
    __syncwarp();

    int pl;                   // lane 0's load cursor
    int64_t pfirst;
    cta_first_layer(a, t_lo, pl, pfirst);
    LayerEntry PL = entry_of(a, pl);
    int64_t issued = 0;
    auto issue = [&](int64_t tile, int stage) {
        if (CAP > 0 || tile >= PL.tile_end) {
            seek_layer(a, tile, pl, pfirst);
            PL = entry_of(a, pl);
        }
        const LayerEntry &L = PL;
        const int64_t g0 = (tile - pfirst) * kTileGroups;
        int64_t ng = L.numel / EV - g0;
        ng = ng > kTileGroups ? kTileGroups : (ng < 0 ? 0 : ng);
        const uint32_t bytes = static_cast<uint32_t>(ng * 16);
        // the test hook (bc_cache_inject_fault) leaves the first stage unarmed
        if (!(a.inject && issued == 0)) {
            mbar_arrive_expect_tx(&full[stage], bytes);
            if (bytes)
                bulk_copy_to_shared(stage_mem + static_cast<size_t>(stage) * kCopyTileBytes,
                                    reinterpret_cast<const char *>(L.src) + g0 * 16, bytes,
                                    &full[stage]);
        }
        ++issued;
    };
    if (lane == 0)
        for (int i = 0; i < S && t_lo + i < t_hi; ++i) issue(t_lo + i, i);

    int l;                    // every lane's store cursor
    int64_t first;
    cta_first_layer(a, t_lo, l, first);
    LayerEntry L = entry_of(a, l);
    for (int64_t tile = t_lo; tile < t_hi; ++tile) {
        const int64_t i = tile - t_lo;
        const int stage = static_cast<int>(i % S);
        int ok = 1;
        if (lane == 0) ok = mbar_wait_bounded(&full[stage], static_cast<uint32_t>((i / S) & 1));
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) {
                if (a.status) atomicOr(a.status, 1u);
                // the stage the test hook left unarmed (the first issued) has no copy
                for (int64_t k = i; k < issued; ++k)
                    if (!(a.inject && k == 0))
                        mbar_wait_bounded(&full[k % S], static_cast<uint32_t>((k / S) & 1));
                bulk_wait_group_all();
            }
            return;
        }
        if (CAP > 0 || tile >= L.tile_end) {
            seek_layer(a, tile, l, first);
            L = entry_of(a, l);
        }
        const int64_t nvec = L.numel / EV;
        if (lane == 0) {
            const int64_t g0 = (tile - first) * kTileGroups;
            int64_t ng = nvec - g0;
            ng = ng > kTileGroups ? kTileGroups : (ng < 0 ? 0 : ng);
            if (ng > 0) {
                fence_proxy_async_shared();
                bulk_store_from_shared(reinterpret_cast<char *>(a.slot[0] + L.dst) + g0 * 16,
                                       stage_mem + static_cast<size_t>(stage) * kCopyTileBytes,
                                       static_cast<uint32_t>(ng * 16));
            }
            bulk_commit_group();
            if (i >= 1 && tile - 1 + S < t_hi) {
                bulk_wait_group_read<1>();  // tile - 1's store no longer reads its stage
                issue(tile - 1 + S, static_cast<int>((i - 1) % S));
            }
        }
        const int rem = static_cast<int>(L.numel - nvec * EV);
        if (rem != 0 && tile == L.tile_end - 1 && lane < rem) {
            const int64_t e = nvec * EV + lane;
            using St = typename T::store_t;
            reinterpret_cast<St *>(a.slot[0] + L.dst)[e] = reinterpret_cast<const St *>(L.src)[e];
        }
    }
    if (lane == 0) bulk_wait_group_all();
}

template <class T, int CAP>
int copy_group(const LayerEntry *layers, int n, const CopyOptions &opt, cudaStream_t s,
               int64_t *launches, int64_t *pipeline_launches) {
    static std::atomic<int> occ{0};
    ForecastArgs<CAP> a;
    memset(&a, 0, sizeof a);
    a.euler_layer = -1;
    a.status = opt.status;
    a.inject = opt.inject;
    a.slot[0] = opt.dst_base;
    // The bulk-copy pipeline needs enough of its 32 KiB tiles per SM to amortise its ring.
    // The layer table is filled with the tile shape of the kernel in question and filled
    // again only if the choice falls on the register copy.
    a.n_layers = n;
    const int sms = sm_count();
    constexpr int kPipeGroups = kCopyTileBytes / 16, kRegGroups = kThreads * kCopyVecsPerThread;
    const bool forced = opt.kernel == BC_KERNEL_PIPELINE || opt.inject;
    const bool weigh = !forced && opt.kernel == BC_KERNEL_AUTO;
    LayerEntry *tab;
    if constexpr (CAP == 0) {
        std::vector<LayerEntry> &v = table_scratch();
        v.resize(static_cast<size_t>(n));
        tab = v.data();
    } else {
        tab = a.layer;
    }
    int tile_groups = forced || weigh ? kPipeGroups : kRegGroups;
    a.total_tiles = fill_entries(tab, layers, n, T::kBytes, 16, tile_groups);
    const bool pipeline =
        forced || (weigh && a.total_tiles >= static_cast<int64_t>(kCopyMinTilesPerCta) * sms);
    if (!pipeline && tile_groups != kRegGroups) {
        tile_groups = kRegGroups;
        a.total_tiles = fill_entries(tab, layers, n, T::kBytes, 16, tile_groups);
    }
    if (a.total_tiles == 0) return cudaSuccess;
    // the launch's error, after recording that a device-table launch reads its table
    auto launched = [&](cudaError_t e) -> int {
        if constexpr (CAP == 0) {
            const int r = table_used(*opt.table, s);
            if (e == cudaSuccess) return r;
        }
        return e;
    };
    if constexpr (CAP == 0) {
        const int err = upload_table(*opt.table, tab, n, s);
        if (err != cudaSuccess) return err;
        a.table = opt.table->dev;
        if (pipeline) {
            const int64_t cap = static_cast<int64_t>(sms) * BC_COPY_CTAS_PER_SM;
            fill_starts(a, tab, n, a.total_tiles < cap ? a.total_tiles : cap);
        }
    }
    if (pipeline) {
        auto kern = copy_tma_kernel<T, CAP>;
        static std::atomic<bool> attr_set[64];
        const int err = ensure_smem_attribute(kern, attr_set, kCopySmemBytes);
        if (err != cudaSuccess) return err;
        const int64_t cap = static_cast<int64_t>(sms) * BC_COPY_CTAS_PER_SM;
        const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
        kern<<<grid, kCopyTmaThreads, kCopySmemBytes, s>>>(a);
        ++*launches;
        ++*pipeline_launches;
        return launched(cudaGetLastError());
    }
    auto kern = copy_kernel<T, CAP>;
    const int64_t cap = static_cast<int64_t>(sms) * resident_ctas(kern, occ, 0);
    const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
    kern<<<grid, kThreads, 0, s>>>(a);
    ++*launches;
    return launched(cudaGetLastError());
}

template <class T>
int copy_all(const LayerEntry *layers, int n_layers, const CopyOptions &opt, cudaStream_t s,
             int64_t *launches, int64_t *pipe) {
    if (n_layers > kLayersLarge && opt.table != nullptr && n_layers <= opt.table->capacity)
        return copy_group<T, 0>(layers, n_layers, opt, s, launches, pipe);
    int err = cudaSuccess;
    for (int base = 0; base < n_layers && err == cudaSuccess; base += kLayersLarge) {
        const int n = n_layers - base < kLayersLarge ? n_layers - base : kLayersLarge;
        if (n <= kLayersSmall)
            err = copy_group<T, kLayersSmall>(layers + base, n, opt, s, launches, pipe);
        else if (n <= kLayersMedium)
            err = copy_group<T, kLayersMedium>(layers + base, n, opt, s, launches, pipe);
        else
            err = copy_group<T, kLayersLarge>(layers + base, n, opt, s, launches, pipe);
    }
    return err;
}

}  // namespace

int launch_forecast(const LaunchPlan &plan, void *stream, int64_t *launches,
                    int64_t *pipeline_launches) {
    switch (plan.K) {
    case 1: return launch_forecast_k1(plan, stream, launches, pipeline_launches);
    case 2: return launch_forecast_k2(plan, stream, launches, pipeline_launches);
    case 3: return launch_forecast_k3(plan, stream, launches, pipeline_launches);
    case 4: return launch_forecast_k4(plan, stream, launches, pipeline_launches);
    default: return cudaErrorInvalidValue;
    }
}

int launch_copy(const LayerEntry *layers, int n_layers, bc_dtype dtype, const CopyOptions &opt,
                void *stream, int64_t *launches, int64_t *pipeline_launches) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == BC_DTYPE_BF16)
        return copy_all<BF16>(layers, n_layers, opt, s, launches, pipeline_launches);
    return copy_all<F32>(layers, n_layers, opt, s, launches, pipeline_launches);
}

}  // namespace bc
