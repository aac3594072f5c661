// bc_forecast.cu -- the device side of the skipped-step forecast (sm_103a).
//
// Eq. 13 applies one weight vector W to the H cached features of every tensor:
//     out[e] = sum_{j=1..H} W_j * F_j[e].
// Per element that is H loads, H fused multiply-adds and one store: about 0.6-0.8 flop
// per byte, far below any compute ridge, so the kernel is a pure HBM stream and tensor
// cores have no role.  The design goals are (1) every cache byte crosses HBM exactly once,
// (2) enough independent 16-byte loads in flight per SM to cover HBM latency, and (3) one
// launch for all cached tensors, so a 60-layer forecast costs one kernel, not sixty.
//
// Work decomposition: every layer is cut into tiles of kTileVecs 16-byte vectors; tiles
// are numbered across layers by a prefix sum carried in the launch's parameter block; a
// persistent grid (SM count x resident CTAs) walks the tile space with a grid stride, so
// neighbouring CTAs stream neighbouring addresses at the same time.  Within a tile a
// thread first issues all H x kVecsPerThread loads, then converts, accumulates in fp32 and
// stores, which keeps up to 16 independent 128-bit loads in flight per thread.
//
// Loads use ld.global.nc with L1::no_allocate (each byte is touched once, L1 reuse is
// nil); stores use st.global.cs (streaming).  Nothing here waits on another CTA, nothing
// allocates, and nothing traps: out-of-range work is never issued because every vector
// index is checked against the layer's length.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <type_traits>

#include "bc_internal.h"

namespace bc {
namespace {

struct F32 {
    using store_t = float;
    static constexpr int kBytes = 4;
};
struct BF16 {
    using store_t = uint16_t;
    static constexpr int kBytes = 2;
};

__device__ __forceinline__ uint4 ld_stream16(const void *p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p));
    return r;
}

// Coherent loads for the Euler state, which the same kernel also writes (the
// non-coherent path is only valid for data that is read-only during the kernel).
__device__ __forceinline__ uint4 ld_plain16(const void *p) {
    uint4 r;
    asm volatile("ld.global.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p)
                 : "memory");
    return r;
}

__device__ __forceinline__ uint2 ld_plain8(const void *p) {
    uint2 r;
    asm volatile("ld.global.v2.u32 {%0, %1}, [%2];" : "=r"(r.x), "=r"(r.y) : "l"(p) : "memory");
    return r;
}

__device__ __forceinline__ void st_stream16(void *p, uint4 v) {
    asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
}

__device__ __forceinline__ void st_stream8(void *p, uint2 v) {
    asm volatile("st.global.cs.v2.u32 [%0], {%1, %2};" ::"l"(p), "r"(v.x), "r"(v.y) : "memory");
}

// bf16 -> fp32 is a 16-bit shift of the bit pattern (exact).
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// fp32 -> bf16, round to nearest even (the CUDA intrinsic), two values per 32-bit word.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    uint32_t u;
    memcpy(&u, &h, sizeof u);
    return u;
}

// Unpack one 16-byte vector of T into EV = 16 / sizeof(T) floats.
template <class T>
__device__ __forceinline__ void unpack16(uint4 r, float *f);
template <>
__device__ __forceinline__ void unpack16<BF16>(uint4 r, float *f) {
    f[0] = bf16_lo(r.x); f[1] = bf16_hi(r.x); f[2] = bf16_lo(r.y); f[3] = bf16_hi(r.y);
    f[4] = bf16_lo(r.z); f[5] = bf16_hi(r.z); f[6] = bf16_lo(r.w); f[7] = bf16_hi(r.w);
}
template <>
__device__ __forceinline__ void unpack16<F32>(uint4 r, float *f) {
    f[0] = __uint_as_float(r.x); f[1] = __uint_as_float(r.y);
    f[2] = __uint_as_float(r.z); f[3] = __uint_as_float(r.w);
}

// Load / store EV consecutive elements of T at element offset `e` (EV is the vector width
// of the history dtype, so the footprint in T is 8, 16 or 32 bytes, naturally aligned).
// Used for the Euler state only, hence the coherent loads.
template <class T, int EV>
__device__ __forceinline__ void load_elems(const char *base, int64_t e, float *f) {
    const char *p = base + e * T::kBytes;
    if constexpr (T::kBytes * EV == 16) {
        unpack16<T>(ld_plain16(p), f);
    } else if constexpr (T::kBytes * EV == 32) {  // f32 x 8
        unpack16<T>(ld_plain16(p), f);
        unpack16<T>(ld_plain16(p + 16), f + 4);
    } else {                                       // bf16 x 4
        uint2 r = ld_plain8(p);
        f[0] = bf16_lo(r.x); f[1] = bf16_hi(r.x); f[2] = bf16_lo(r.y); f[3] = bf16_hi(r.y);
    }
}

template <class T, int EV>
__device__ __forceinline__ void store_elems(char *base, int64_t e, const float *f) {
    char *p = base + e * T::kBytes;
    if constexpr (std::is_same<T, BF16>::value) {
        if constexpr (EV == 8) {
            st_stream16(p, make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]),
                                      pack_bf16x2(f[4], f[5]), pack_bf16x2(f[6], f[7])));
        } else {
            st_stream8(p, make_uint2(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3])));
        }
    } else {
        st_stream16(p, make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]),
                                  __float_as_uint(f[2]), __float_as_uint(f[3])));
        if constexpr (EV == 8) {
            st_stream16(p + 16, make_uint4(__float_as_uint(f[4]), __float_as_uint(f[5]),
                                           __float_as_uint(f[6]), __float_as_uint(f[7])));
        }
    }
}

template <class T>
__device__ __forceinline__ float load_scalar(const char *base, int64_t e) {
    if constexpr (std::is_same<T, BF16>::value) {
        uint16_t h = *reinterpret_cast<const uint16_t *>(base + e * 2);
        return __uint_as_float(static_cast<uint32_t>(h) << 16);
    } else {
        return *reinterpret_cast<const float *>(base + e * 4);
    }
}

template <class T>
__device__ __forceinline__ void store_scalar(char *base, int64_t e, float v) {
    if constexpr (std::is_same<T, BF16>::value) {
        __nv_bfloat16 h = __float2bfloat16_rn(v);
        uint16_t u;
        memcpy(&u, &h, sizeof u);
        *reinterpret_cast<uint16_t *>(base + e * 2) = u;
    } else {
        *reinterpret_cast<float *>(base + e * 4) = v;
    }
}

// Advance the CTA's layer cursor so that `tile` lies in layer `l`.  Tiles only grow, so
// the cursor only moves forward; `first` is the layer's first tile.
template <int CAP>
__device__ __forceinline__ void seek_layer(const ForecastArgs<CAP> &a, int64_t tile, int &l,
                                           int64_t &first) {
    while (tile >= a.layer[l].tile_end) {
        first = a.layer[l].tile_end;
        ++l;
    }
}

// The grouped forecast, optionally with the Euler epilogue on one layer.
template <int K, class TIn, class TOut, int CAP>
__global__ void __launch_bounds__(kThreads)
    forecast_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int EV = 16 / TIn::kBytes;  // elements per 16-byte history vector
    float w[K];
#pragma unroll
    for (int j = 0; j < K; ++j) w[j] = a.w[j];

    int l = 0;
    int64_t first = 0;
    for (int64_t tile = blockIdx.x; tile < a.total_tiles; tile += gridDim.x) {
        seek_layer(a, tile, l, first);
        const LayerEntry &L = a.layer[l];
        const int64_t numel = L.numel;
        const int64_t nvec = numel / EV;
        const int64_t v0 = (tile - first) * kTileVecs + threadIdx.x;
        const char *src[K];
#pragma unroll
        for (int j = 0; j < K; ++j) src[j] = reinterpret_cast<const char *>(a.slot[j] + L.src);
        char *dst = reinterpret_cast<char *>(L.dst);
        const bool euler = (l == a.euler_layer);

        // Issue every load of the tile before using any of them.
        uint4 r[kVecsPerThread][K];
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) {
#pragma unroll
                for (int j = 0; j < K; ++j) r[u][j] = ld_stream16(src[j] + v * 16);
            }
        }
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) {
                float acc[EV], f[EV];
                unpack16<TIn>(r[u][0], f);
#pragma unroll
                for (int e = 0; e < EV; ++e) acc[e] = w[0] * f[e];
#pragma unroll
                for (int j = 1; j < K; ++j) {
                    unpack16<TIn>(r[u][j], f);
#pragma unroll
                    for (int e = 0; e < EV; ++e) acc[e] = fmaf(w[j], f[e], acc[e]);
                }
                if (!euler) {
                    store_elems<TOut, EV>(dst, v * EV, acc);
                } else {
                    if (dst) store_elems<TOut, EV>(dst, v * EV, acc);
                    float x[EV];
                    char *xb = reinterpret_cast<char *>(a.x);
                    if (a.x_bf16) {
                        load_elems<BF16, EV>(xb, v * EV, x);
#pragma unroll
                        for (int e = 0; e < EV; ++e) x[e] = fmaf(a.dt, acc[e], x[e]);
                        store_elems<BF16, EV>(xb, v * EV, x);
                    } else {
                        load_elems<F32, EV>(xb, v * EV, x);
#pragma unroll
                        for (int e = 0; e < EV; ++e) x[e] = fmaf(a.dt, acc[e], x[e]);
                        store_elems<F32, EV>(xb, v * EV, x);
                    }
                }
            }
        }
        // Ragged tail (numel not a multiple of EV): the layer's last tile takes it.
        const int rem = static_cast<int>(numel - nvec * EV);
        if (rem != 0 && tile == L.tile_end - 1 && static_cast<int>(threadIdx.x) < rem) {
            const int64_t e = nvec * EV + threadIdx.x;
            float acc = w[0] * load_scalar<TIn>(src[0], e);
#pragma unroll
            for (int j = 1; j < K; ++j) acc = fmaf(w[j], load_scalar<TIn>(src[j], e), acc);
            if (!euler) {
                store_scalar<TOut>(dst, e, acc);
            } else {
                if (dst) store_scalar<TOut>(dst, e, acc);
                char *xb = reinterpret_cast<char *>(a.x);
                if (a.x_bf16)
                    store_scalar<BF16>(xb, e, fmaf(a.dt, acc, load_scalar<BF16>(xb, e)));
                else
                    store_scalar<F32>(xb, e, fmaf(a.dt, acc, load_scalar<F32>(xb, e)));
            }
        }
    }
}

// Grouped byte-exact copy for the push: layer.src -> layer.dst, numel elements of T.
template <class T, int CAP>
__global__ void __launch_bounds__(kThreads) copy_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int EV = 16 / T::kBytes;
    int l = 0;
    int64_t first = 0;
    for (int64_t tile = blockIdx.x; tile < a.total_tiles; tile += gridDim.x) {
        seek_layer(a, tile, l, first);
        const LayerEntry &L = a.layer[l];
        const int64_t nvec = L.numel / EV;
        const int64_t v0 = (tile - first) * kTileVecs + threadIdx.x;
        const char *src = reinterpret_cast<const char *>(L.src);
        char *dst = reinterpret_cast<char *>(L.dst);
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

// ------------------------------------------------------------------ launch plumbing

int g_sm_count = 0;

int sm_count() {
    if (g_sm_count == 0) {
        int dev = 0, n = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        g_sm_count = n > 0 ? n : 1;
    }
    return g_sm_count;
}

template <class KernelPtr>
int resident_ctas(KernelPtr kern, int &cache) {
    if (cache == 0) {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, kThreads, 0) != cudaSuccess ||
            n < 1)
            n = 1;
        cache = n;
    }
    return cache;
}

template <int CAP>
int64_t fill_table(ForecastArgs<CAP> &a, const LayerEntry *layers, int n, int elem_bytes) {
    int64_t tiles = 0;
    for (int i = 0; i < n; ++i) {
        a.layer[i] = layers[i];
        tiles += tiles_for(layers[i].numel, elem_bytes);
        a.layer[i].tile_end = tiles;
    }
    a.n_layers = n;
    return tiles;
}

template <int K, class TIn, class TOut, int CAP>
int launch_group(const LaunchPlan &p, const LayerEntry *layers, int n, int euler_local,
                 cudaStream_t s, int64_t *launches) {
    static int occ = 0;
    ForecastArgs<CAP> a;
    memset(&a, 0, sizeof a);
    for (int j = 0; j < BC_MAX_K; ++j) {
        a.slot[j] = p.slot[j];
        a.w[j] = p.w[j];
    }
    a.dt = p.dt;
    a.euler_layer = euler_local;
    a.x_bf16 = p.x_dtype == BC_DTYPE_BF16 ? 1 : 0;
    a.x = p.x;
    a.total_tiles = fill_table(a, layers, n, TIn::kBytes);
    if (a.total_tiles == 0) return cudaSuccess;
    auto kern = forecast_kernel<K, TIn, TOut, CAP>;
    const int64_t cap = static_cast<int64_t>(sm_count()) * resident_ctas(kern, occ);
    const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
    kern<<<grid, kThreads, 0, s>>>(a);
    ++*launches;
    return cudaGetLastError();
}

template <int K, class TIn, class TOut>
int launch_all(const LaunchPlan &p, cudaStream_t s, int64_t *launches) {
    int err = cudaSuccess;
    for (int base = 0; base < p.n_layers && err == cudaSuccess; base += kLayersLarge) {
        const int n = p.n_layers - base < kLayersLarge ? p.n_layers - base : kLayersLarge;
        const int eul = (p.euler_layer >= base && p.euler_layer < base + n) ? p.euler_layer - base
                                                                             : -1;
        if (n <= kLayersSmall)
            err = launch_group<K, TIn, TOut, kLayersSmall>(p, p.layers + base, n, eul, s, launches);
        else
            err = launch_group<K, TIn, TOut, kLayersLarge>(p, p.layers + base, n, eul, s, launches);
    }
    return err;
}

template <int K>
int dispatch_dtypes(const LaunchPlan &p, cudaStream_t s, int64_t *launches) {
    const bool in_bf = p.in_dtype == BC_DTYPE_BF16, out_bf = p.out_dtype == BC_DTYPE_BF16;
    if (in_bf && out_bf) return launch_all<K, BF16, BF16>(p, s, launches);
    if (in_bf && !out_bf) return launch_all<K, BF16, F32>(p, s, launches);
    if (!in_bf && out_bf) return launch_all<K, F32, BF16>(p, s, launches);
    return launch_all<K, F32, F32>(p, s, launches);
}

template <class T, int CAP>
int copy_group(const LayerEntry *layers, int n, cudaStream_t s, int64_t *launches) {
    static int occ = 0;
    ForecastArgs<CAP> a;
    memset(&a, 0, sizeof a);
    a.euler_layer = -1;
    a.total_tiles = fill_table(a, layers, n, T::kBytes);
    if (a.total_tiles == 0) return cudaSuccess;
    auto kern = copy_kernel<T, CAP>;
    const int64_t cap = static_cast<int64_t>(sm_count()) * resident_ctas(kern, occ);
    const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
    kern<<<grid, kThreads, 0, s>>>(a);
    ++*launches;
    return cudaGetLastError();
}

template <class T>
int copy_all(const LayerEntry *layers, int n_layers, cudaStream_t s, int64_t *launches) {
    int err = cudaSuccess;
    for (int base = 0; base < n_layers && err == cudaSuccess; base += kLayersLarge) {
        const int n = n_layers - base < kLayersLarge ? n_layers - base : kLayersLarge;
        if (n <= kLayersSmall)
            err = copy_group<T, kLayersSmall>(layers + base, n, s, launches);
        else
            err = copy_group<T, kLayersLarge>(layers + base, n, s, launches);
    }
    return err;
}

}  // namespace

int launch_forecast(const LaunchPlan &plan, void *stream, int64_t *launches) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    switch (plan.K) {
    case 1: return dispatch_dtypes<1>(plan, s, launches);
    case 2: return dispatch_dtypes<2>(plan, s, launches);
    case 3: return dispatch_dtypes<3>(plan, s, launches);
    case 4: return dispatch_dtypes<4>(plan, s, launches);
    default: return cudaErrorInvalidValue;
    }
}

int launch_copy(const LayerEntry *layers, int n_layers, bc_dtype dtype, void *stream,
                int64_t *launches) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == BC_DTYPE_BF16) return copy_all<BF16>(layers, n_layers, s, launches);
    return copy_all<F32>(layers, n_layers, s, launches);
}

}  // namespace bc
