// bc_forecast_kernels.cuh -- the device side of the skipped-step forecast (sm_103a) and its
// launch logic, instantiated once per history length K by bc_forecast_k{1,2,3,4}.cu so that
// the four translation units compile in parallel.
//
// Eq. 13 applies one weight vector W to the H cached features of every tensor:
//     out[e] = sum_{j=1..H} W_j * F_j[e].
// Per element that is H loads, H fused multiply-adds and one store: about 0.6-0.8 flop
// per byte, far below any compute ridge, so the kernels are pure HBM streams and tensor
// cores have no role.  The design goals are (1) every cache byte crosses HBM exactly once,
// (2) enough bytes in flight per SM to cover HBM latency, and (3) one launch for all cached
// tensors, so a 60-layer forecast costs one kernel, not sixty.
//
// Work decomposition: every layer is cut into tiles of kThreads x VPT history vectors of
// 32 bytes; tiles are numbered across layers by a prefix sum in the launch's layer table
// (carried in the parameter block, or for very many layers in device memory); a persistent
// grid splits the tile space into one contiguous range per CTA, so every CTA streams
// sequential addresses.  Two kernels share the arithmetic (combine_vector / combine_tail,
// so they produce the same bits) and differ in how the history reaches the SM:
//   forecast_tma_kernel  TMA bulk copies into a shared-memory ring of stages, one CTA per
//                        SM (H <= 3, and H = 4 with smaller tiles);
//   forecast_kernel      every thread issues all of its 256-bit loads into registers before
//                        using any, up to two CTAs per SM (small launches, and many small
//                        tensors).
//
// Arithmetic: the host divides the fp32 weights by a power of two `scale` >= sum_j |W_j|
// (kernel_weights), the kernels accumulate in fp32 with FMA in node order j = 1..H and
// multiply by `scale` once (on the update layer the multiplication is folded into the update
// coefficient): bit for bit the unscaled sum wherever that neither overflows nor goes
// subnormal, and no partial sum ever exceeds max_j |F_j|.  NaN and infinities propagate as
// IEEE arithmetic gives them.
//
// Outputs, the sampler state and push sources carry only the ABI's 16-byte alignment and
// use 128-bit (or 64-bit) accesses; stores are st.global.cs (streaming).  No CTA waits on
// another, nothing allocates and nothing traps: every vector index is checked against its
// layer's length, and the pipeline kernel's waits on its own mbarriers are bounded.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <cstring>
#include <type_traits>
#include <vector>

#include "bc_internal.h"
#include "bc_tma.cuh"

// Tuning knobs of the pipeline kernel (the defaults are the best of the sweeps on GB300,
// video workload): 256 threads x VPT 32-byte vectors per slot and tile, S stages.
#ifndef BC_TMA_VPT
#define BC_TMA_VPT 2         // 16 KiB tiles per history slot
#endif
#ifndef BC_TMA_STAGES
#define BC_TMA_STAGES 3
#endif
#ifndef BC_TMA_VPT_K4
#define BC_TMA_VPT_K4 1      // 8 KiB tiles per history slot at H = 4
#endif
#ifndef BC_TMA_STAGES_K4
#define BC_TMA_STAGES_K4 5   // 5 x 4 x 8 KiB = 160 KiB of shared memory
#endif
#ifndef BC_TMA_AUTO_K4
#define BC_TMA_AUTO_K4 1     // AUTO picks the pipeline at H = 4 for large launches too
#endif
#ifndef BC_TMA_MIN_TILES_PER_LAYER
// AUTO runs the pipeline only when layers average at least this many of its tiles: many
// small tensors (the blockwise layout: 4096 x 64 Ki bf16, eight 16 KiB tiles each) stream
// faster through the register kernel (7.14 vs 7.00 TB/s at H = 3).
#define BC_TMA_MIN_TILES_PER_LAYER 32
#endif
#ifndef BC_SMALL_LAUNCH_TILES_PER_SM
#define BC_SMALL_LAUNCH_TILES_PER_SM 2  // register launches below this many tiles per SM use VPT 1
#endif

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

// One history vector: kVecBytes bytes as 16-byte pieces.
struct Raw {
    uint4 q[kVecBytes / 16];
};

__device__ __forceinline__ uint64_t history_policy() {
    uint64_t pol = 0;
#if BC_L2_EVICT_FIRST
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
#endif
    return pol;
}

// History loads: read-only for the whole kernel, touched once -> non-coherent path, no L1
// allocation.  The slots are 256-byte aligned, so 32-byte vectors are always aligned.
__device__ __forceinline__ Raw ld_history(const char *p, uint64_t pol) {
    Raw r;
    (void)pol;
    if constexpr (kVecBytes == 32) {
#if BC_L2_EVICT_FIRST
        asm("ld.global.nc.L1::no_allocate.L2::cache_hint.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8], %9;"
            : "=r"(r.q[0].x), "=r"(r.q[0].y), "=r"(r.q[0].z), "=r"(r.q[0].w), "=r"(r.q[1].x),
              "=r"(r.q[1].y), "=r"(r.q[1].z), "=r"(r.q[1].w)
            : "l"(p), "l"(pol));
#else
        asm("ld.global.nc.L1::no_allocate.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
            : "=r"(r.q[0].x), "=r"(r.q[0].y), "=r"(r.q[0].z), "=r"(r.q[0].w), "=r"(r.q[1].x),
              "=r"(r.q[1].y), "=r"(r.q[1].z), "=r"(r.q[1].w)
            : "l"(p));
#endif
    } else {
#if BC_L2_EVICT_FIRST
        asm("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
            : "=r"(r.q[0].x), "=r"(r.q[0].y), "=r"(r.q[0].z), "=r"(r.q[0].w)
            : "l"(p), "l"(pol));
#else
        asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
            : "=r"(r.q[0].x), "=r"(r.q[0].y), "=r"(r.q[0].z), "=r"(r.q[0].w)
            : "l"(p));
#endif
    }
    return r;
}

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

// 16 bytes of T <-> 16 / sizeof(T) floats.
template <class T>
__device__ __forceinline__ void unpack16(uint4 r, float *f) {
    if constexpr (std::is_same<T, BF16>::value) {
        f[0] = bf16_lo(r.x); f[1] = bf16_hi(r.x); f[2] = bf16_lo(r.y); f[3] = bf16_hi(r.y);
        f[4] = bf16_lo(r.z); f[5] = bf16_hi(r.z); f[6] = bf16_lo(r.w); f[7] = bf16_hi(r.w);
    } else {
        f[0] = __uint_as_float(r.x); f[1] = __uint_as_float(r.y);
        f[2] = __uint_as_float(r.z); f[3] = __uint_as_float(r.w);
    }
}

template <class T>
__device__ __forceinline__ uint4 pack16(const float *f) {
    if constexpr (std::is_same<T, BF16>::value) {
        return make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]),
                          pack_bf16x2(f[4], f[5]), pack_bf16x2(f[6], f[7]));
    } else {
        return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                          __float_as_uint(f[3]));
    }
}

// N consecutive elements of T at byte address p, N * sizeof(T) = 8 or a multiple of 16.
// Addresses are 16-byte aligned (8 for the 8-byte case): outputs and the Euler state are
// only guaranteed 16-byte alignment, so wider accesses are never used on them.
template <class T, int N>
__device__ __forceinline__ void load_plain(const char *p, float *f) {
    constexpr int B = N * T::kBytes;
    if constexpr (B == 8) {
        static_assert(std::is_same<T, BF16>::value, "8-byte groups are 4 bf16");
        const uint2 r = ld_plain8(p);
        f[0] = bf16_lo(r.x); f[1] = bf16_hi(r.x); f[2] = bf16_lo(r.y); f[3] = bf16_hi(r.y);
    } else {
#pragma unroll
        for (int q = 0; q < B / 16; ++q) unpack16<T>(ld_plain16(p + 16 * q), f + q * (16 / T::kBytes));
    }
}

template <class T, int N>
__device__ __forceinline__ void store_stream(char *p, const float *f) {
    constexpr int B = N * T::kBytes;
    if constexpr (B == 8) {
        static_assert(std::is_same<T, BF16>::value, "8-byte groups are 4 bf16");
        st_stream8(p, make_uint2(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3])));
    } else {
#pragma unroll
        for (int q = 0; q < B / 16; ++q) st_stream16(p + 16 * q, pack16<T>(f + q * (16 / T::kBytes)));
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

// ------------------------------------------------------------------ the layer table
//
// With CAP > 0 the table is part of the parameter block; with CAP == 0 it lives in device
// memory (read-only during the launch, so through the non-coherent path).
template <int CAP>
__device__ __forceinline__ int64_t tile_end_of(const ForecastArgs<CAP> &a, int l) {
    if constexpr (CAP == 0)
        return __ldg(reinterpret_cast<const long long *>(&a.table[l].tile_end));
    else
        return a.layer[l].tile_end;
}

template <int CAP>
__device__ __forceinline__ LayerEntry entry_of(const ForecastArgs<CAP> &a, int l) {
    if constexpr (CAP == 0) {
        const LayerEntry *p = a.table + l;
        LayerEntry e;
        e.src = __ldg(reinterpret_cast<const unsigned long long *>(&p->src));
        e.dst = __ldg(reinterpret_cast<const unsigned long long *>(&p->dst));
        e.numel = __ldg(reinterpret_cast<const long long *>(&p->numel));
        e.tile_end = __ldg(reinterpret_cast<const long long *>(&p->tile_end));
        return e;
    } else {
        return a.layer[l];
    }
}

// Place a layer cursor on the layer holding `tile`: a binary search over the tiles' prefix
// sums (about ten dependent loads for a full table, where a scan from layer 0 would take up
// to one per layer); `first` is the layer's first tile.
template <int CAP>
__device__ __forceinline__ void find_layer(const ForecastArgs<CAP> &a, int64_t tile, int &l,
                                           int64_t &first) {
    int lo = 0, hi = a.n_layers - 1;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (tile < tile_end_of(a, mid))
            hi = mid;
        else
            lo = mid + 1;
    }
    l = lo;
    first = lo > 0 ? tile_end_of(a, lo - 1) : 0;
}

// Advance the CTA's layer cursor so that `tile` lies in layer `l`.  Tiles only grow, so
// the cursor only moves forward; `first` is the layer's first tile.
template <int CAP>
__device__ __forceinline__ void seek_layer(const ForecastArgs<CAP> &a, int64_t tile, int &l,
                                           int64_t &first) {
    int64_t end = tile_end_of(a, l);
    while (tile >= end) {
        first = end;
        ++l;
        end = tile_end_of(a, l);
    }
}

// The layer cursor of a CTA's first tile: from the host-computed starts when the launch has
// them, else by binary search.
template <int CAP>
__device__ __forceinline__ void cta_first_layer(const ForecastArgs<CAP> &a, int64_t t_lo, int &l,
                                                int64_t &first) {
    if constexpr (CAP == 0) {
        if (static_cast<int>(blockIdx.x) < a.n_starts) {
            l = a.start[blockIdx.x].layer;
            first = a.start[blockIdx.x].first;
            return;
        }
    }
    find_layer(a, t_lo, l, first);
}

// Forecast one history vector from its K raw pieces (node order j = 1..K), store it, and
// on the update layer apply x <- ca x + cb v_hat (+ cc z) to the same elements.
template <int K, class TIn, class TOut, int CAP>
__device__ __forceinline__ void combine_vector(const ForecastArgs<CAP> &a, const float *w,
                                               float scale, const Raw *r, char *dst, int64_t v,
                                               bool euler) {
    constexpr int EV = kVecBytes / TIn::kBytes;  // elements per history vector
    constexpr int EV16 = 16 / TIn::kBytes;       // elements per 16-byte piece
    float acc[EV], f[EV];
#pragma unroll
    for (int q = 0; q < kVecBytes / 16; ++q) unpack16<TIn>(r[0].q[q], f + q * EV16);
#pragma unroll
    for (int e = 0; e < EV; ++e) acc[e] = w[0] * f[e];
#pragma unroll
    for (int j = 1; j < K; ++j) {
#pragma unroll
        for (int q = 0; q < kVecBytes / 16; ++q) unpack16<TIn>(r[j].q[q], f + q * EV16);
#pragma unroll
        for (int e = 0; e < EV; ++e) acc[e] = fmaf(w[j], f[e], acc[e]);
    }
    if (dst) {
        float out[EV];
#pragma unroll
        for (int e = 0; e < EV; ++e) out[e] = acc[e] * scale;
        store_stream<TOut, EV>(dst + v * EV * TOut::kBytes, out);
    }
    if (euler) {
        // Sampler update on the same elements: x <- ca x + cb v_hat (+ cc z), with
        // v_hat = scale * acc taken inside the FMA as (cb * scale) * acc: the same bits as
        // rounding v_hat first wherever v_hat is in range, and a finite x where only v_hat
        // itself would overflow.
        const float cbs = a.cb * scale;
        float x[EV];
        char *xp = reinterpret_cast<char *>(a.x);
        const char *zp = reinterpret_cast<const char *>(a.z);
        if (a.x_bf16) {
            xp += v * EV * 2;
            load_plain<BF16, EV>(xp, x);
#pragma unroll
            for (int e = 0; e < EV; ++e) x[e] = fmaf(cbs, acc[e], a.ca * x[e]);
            if (zp) {
                float z[EV];
                load_plain<BF16, EV>(zp + v * EV * 2, z);
#pragma unroll
                for (int e = 0; e < EV; ++e) x[e] = fmaf(a.cc, z[e], x[e]);
            }
            store_stream<BF16, EV>(xp, x);
        } else {
            xp += v * EV * 4;
            load_plain<F32, EV>(xp, x);
#pragma unroll
            for (int e = 0; e < EV; ++e) x[e] = fmaf(cbs, acc[e], a.ca * x[e]);
            if (zp) {
                float z[EV];
                load_plain<F32, EV>(zp + v * EV * 4, z);
#pragma unroll
                for (int e = 0; e < EV; ++e) x[e] = fmaf(a.cc, z[e], x[e]);
            }
            store_stream<F32, EV>(xp, x);
        }
    }
}

// Ragged tail of a layer (numel not a multiple of the vector width): scalar accesses by the
// first `rem` threads of the CTA that owns the layer's last tile.
template <int K, class TIn, class TOut, int CAP>
__device__ __forceinline__ void combine_tail(const ForecastArgs<CAP> &a, const float *w,
                                             float scale, const LayerEntry &L, char *dst,
                                             int64_t nvec, bool euler) {
    constexpr int EV = kVecBytes / TIn::kBytes;
    const int rem = static_cast<int>(L.numel - nvec * EV);
    if (rem == 0 || static_cast<int>(threadIdx.x) >= rem) return;
    const int64_t e = nvec * EV + threadIdx.x;
    float acc = w[0] * load_scalar<TIn>(reinterpret_cast<const char *>(a.slot[0] + L.src), e);
#pragma unroll
    for (int j = 1; j < K; ++j)
        acc = fmaf(w[j], load_scalar<TIn>(reinterpret_cast<const char *>(a.slot[j] + L.src), e),
                   acc);
    if (dst) store_scalar<TOut>(dst, e, acc * scale);
    if (euler) {
        const float cbs = a.cb * scale;
        char *xb = reinterpret_cast<char *>(a.x);
        const char *zb = reinterpret_cast<const char *>(a.z);
        if (a.x_bf16) {
            float xn = fmaf(cbs, acc, a.ca * load_scalar<BF16>(xb, e));
            if (zb) xn = fmaf(a.cc, load_scalar<BF16>(zb, e), xn);
            store_scalar<BF16>(xb, e, xn);
        } else {
            float xn = fmaf(cbs, acc, a.ca * load_scalar<F32>(xb, e));
            if (zb) xn = fmaf(a.cc, load_scalar<F32>(zb, e), xn);
            store_scalar<F32>(xb, e, xn);
        }
    }
}

// The grouped forecast with register-held history loads: each thread issues all
// H x VPT loads of its tile before using any of them.
template <int K, int VPT, class TIn, class TOut, int CAP>
__global__ void __launch_bounds__(kThreads)
    forecast_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int kTileVecs = kThreads * VPT;
    const uint64_t pol = history_policy();
    float w[K];
#pragma unroll
    for (int j = 0; j < K; ++j) w[j] = a.w[j];
    const float scale = a.scale;

    // Each CTA streams one contiguous range of tiles (better DRAM page locality than a
    // grid stride: 7.24 vs 7.18 TB/s on the video workload at H = 3).
    const int64_t per_cta = (a.total_tiles + gridDim.x - 1) / gridDim.x;
    const int64_t t_lo = static_cast<int64_t>(blockIdx.x) * per_cta;
    const int64_t t_hi = t_lo + per_cta < a.total_tiles ? t_lo + per_cta : a.total_tiles;
    if (t_lo >= t_hi) return;
    int l;
    int64_t first;
    cta_first_layer(a, t_lo, l, first);
    LayerEntry L = entry_of(a, l);
    for (int64_t tile = t_lo; tile < t_hi; ++tile) {
        if (tile >= L.tile_end) {
            seek_layer(a, tile, l, first);
            L = entry_of(a, l);
        }
        const int64_t nvec = L.numel / (kVecBytes / TIn::kBytes);
        const int64_t v0 = (tile - first) * kTileVecs + threadIdx.x;
        const char *src[K];
#pragma unroll
        for (int j = 0; j < K; ++j) src[j] = reinterpret_cast<const char *>(a.slot[j] + L.src);
        char *dst = reinterpret_cast<char *>(L.dst);
        const bool euler = (l == a.euler_layer);

        Raw r[VPT][K];
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) {
#pragma unroll
                for (int j = 0; j < K; ++j) r[u][j] = ld_history(src[j] + v * kVecBytes, pol);
            }
        }
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) combine_vector<K, TIn, TOut, CAP>(a, w, scale, r[u], dst, v, euler);
        }
        if (tile == L.tile_end - 1)
            combine_tail<K, TIn, TOut, CAP>(a, w, scale, L, dst, nvec, euler);
    }
}

// ---------------------------------------------------------------------------------------
// The grouped forecast with the history staged through shared memory by the Tensor Memory
// Accelerator.  Each CTA (one per SM) owns a ring of S stages; a stage holds one tile of
// every history slot (H x kThreads x VPT x 32 bytes).  Thread 0 issues one 1-D bulk copy
// (cp.async.bulk, global -> shared) per slot and tile, completing on the stage's mbarrier
// with a transaction count; all threads wait on that mbarrier, combine from shared memory
// and store to global memory directly; after a CTA barrier thread 0 refills the stage with
// the tile S ahead.  Three 48 KiB stages in flight per SM sustain 7.35 TB/s at H = 3 on the
// video workload (7.27 TB/s with register-held loads); the outputs are bit-identical to the
// register kernel's.
//
// Every wait is bounded (about one second by %globaltimer): on expiry the CTA records the
// failure in the handle's device status word, drains the copies it issued (again bounded;
// the stage the test hook left unarmed has nothing to drain) and returns, so a lost
// completion can never hang the device; the host reads the word with bc_cache_check.
constexpr int kTmaMinTilesPerCta = 16;

template <int K>
constexpr int kTmaVpt = K >= 4 ? BC_TMA_VPT_K4 : BC_TMA_VPT;
template <int K>
constexpr int kTmaStages = K >= 4 ? BC_TMA_STAGES_K4 : BC_TMA_STAGES;
// Bytes of one history tile, and of the whole ring (S stages of K tiles).
template <int K>
constexpr int kTmaTileBytes = kThreads * kTmaVpt<K> * kVecBytes;
template <int K>
constexpr int kTmaSmemBytes = kTmaStages<K> * K * kTmaTileBytes<K>;

template <int K, class TIn, class TOut, int CAP>
__global__ void __launch_bounds__(kThreads)
    forecast_tma_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int VPT = kTmaVpt<K>;
    constexpr int kTileVecs = kThreads * VPT;
    constexpr int kTileBytes = kTmaTileBytes<K>;
    constexpr int EV = kVecBytes / TIn::kBytes;
    constexpr int S = kTmaStages<K>;
    static_assert(kTmaSmemBytes<K> <= 227 * 1024, "the ring exceeds a CTA's shared memory");
    extern __shared__ __align__(128) unsigned char stage_mem[];
    __shared__ __align__(8) uint64_t full[S];
    // kMeta: the producer hands each stage's layer (entry, index, first tile) to the consumers
    // through shared memory, written before the stage is armed and read after the wait (the
    // mbarrier arrival releases it), so the consumers never touch the layer table.  That pays
    // where the table is in device memory; with the parameter-block table it measured +0.5 %
    // at H = 3 and -1.2 % at H = 4 (-0.2 % at H = 2) on the video workload, so elsewhere the
    // consumers keep their own cursor over the parameter block.
    constexpr bool kMeta = CAP == 0 || K == 3;
    // kCache: producer and consumers keep the current layer's entry in registers and re-read
    // the table only on crossing into the next layer.  Measured on the video workload against
    // re-reading the parameter-block entry on every tile: +0.5 % at H = 2, -2 % at H = 4
    // (8 KiB tiles, five stages; reproducible on two boxes, cause not isolated), so H = 4
    // re-reads per tile unless the table is in device memory.
    constexpr bool kCache = CAP == 0 || K != 4;
    __shared__ LayerEntry stage_entry[kMeta ? S : 1];
    __shared__ int32_t stage_layer[kMeta ? S : 1];
    __shared__ int64_t stage_first[kMeta ? S : 1];
    __shared__ int abort_flag;

    float w[K];
#pragma unroll
    for (int j = 0; j < K; ++j) w[j] = a.w[j];
    const float scale = a.scale;
    const int64_t per_cta = (a.total_tiles + gridDim.x - 1) / gridDim.x;
    const int64_t t_lo = static_cast<int64_t>(blockIdx.x) * per_cta;
    const int64_t t_hi = t_lo + per_cta < a.total_tiles ? t_lo + per_cta : a.total_tiles;
    if (threadIdx.x == 0) {
        for (int i = 0; i < S; ++i) mbar_init(&full[i], 1);
        mbar_init_fence();
        abort_flag = 0;
    }
    __syncthreads();

    // Producer state (thread 0): its own layer cursor, and how many tiles it has issued.
    int pl = 0;
    int64_t pfirst = 0;
    int64_t issued = 0;
    LayerEntry PL{};
    auto issue = [&](int64_t tile, int stage) {
        if (!kCache || tile >= PL.tile_end) {
            seek_layer(a, tile, pl, pfirst);
            PL = entry_of(a, pl);
        }
        const LayerEntry &L = PL;
        if constexpr (kMeta) {
            stage_entry[stage] = L;
            stage_layer[stage] = pl;
            stage_first[stage] = pfirst;
        }
        const int64_t nvec = L.numel / EV;
        const int64_t v_first = (tile - pfirst) * kTileVecs;
        int64_t nv = nvec - v_first;
        nv = nv > kTileVecs ? kTileVecs : (nv < 0 ? 0 : nv);
        const uint32_t bytes = static_cast<uint32_t>(nv * kVecBytes);
        // A test hook (bc_cache_inject_fault) leaves the first stage unarmed, so that its
        // wait runs out; nothing else ever skips the arrival.
        if (!(a.inject && issued == 0)) mbar_arrive_expect_tx(&full[stage], bytes * K);
        if (bytes && !(a.inject && issued == 0)) {
#pragma unroll
            for (int j = 0; j < K; ++j)
                bulk_copy_to_shared(stage_mem + (static_cast<size_t>(stage) * K + j) * kTileBytes,
                                    reinterpret_cast<const char *>(a.slot[j] + L.src) +
                                        v_first * kVecBytes,
                                    bytes, &full[stage]);
        }
        ++issued;
    };
    if (threadIdx.x == 0 && t_lo < t_hi) {
        cta_first_layer(a, t_lo, pl, pfirst);
        PL = entry_of(a, pl);
        for (int i = 0; i < S && t_lo + i < t_hi; ++i) issue(t_lo + i, i);
    }

    int l = 0;                // the consumers' own cursor (without kMeta)
    int64_t first = 0;
    LayerEntry CL{};
    if (!kMeta && t_lo < t_hi) {
        cta_first_layer(a, t_lo, l, first);
        CL = entry_of(a, l);
    }
    for (int64_t tile = t_lo; tile < t_hi; ++tile) {
        const int64_t i = tile - t_lo;
        const int stage = static_cast<int>(i % S);
        if (!mbar_wait_bounded(&full[stage], static_cast<uint32_t>((i / S) & 1))) abort_flag = 1;
        __syncthreads();  // the exit decision below is the same for every thread
        if (abort_flag) {
            if (threadIdx.x == 0) {
                if (a.status) atomicOr(a.status, 1u);
                // drain the copies this CTA issued and has not consumed (bounded); the stage
                // the test hook left unarmed (the first issued) has none in flight
                for (int64_t k = i; k < issued; ++k)
                    if (!(a.inject && k == 0))
                        mbar_wait_bounded(&full[k % S], static_cast<uint32_t>((k / S) & 1));
            }
            return;
        }
        LayerEntry L;
        int64_t lfirst;
        int lidx;
        if constexpr (kMeta) {
            L = stage_entry[stage];
            lfirst = stage_first[stage];
            lidx = stage_layer[stage];
        } else {
            if (!kCache || tile >= CL.tile_end) {
                seek_layer(a, tile, l, first);
                CL = entry_of(a, l);
            }
            L = CL;
            lfirst = first;
            lidx = l;
        }
        const int64_t nvec = L.numel / EV;
        const int64_t v0 = (tile - lfirst) * kTileVecs;
        char *dst = reinterpret_cast<char *>(L.dst);
        const bool euler = (lidx == a.euler_layer);
        const unsigned char *sb = stage_mem + static_cast<size_t>(stage) * K * kTileBytes;
#pragma unroll
        for (int u = 0; u < VPT; ++u) {
            const int lv = u * kThreads + threadIdx.x;
            const int64_t v = v0 + lv;
            if (v < nvec) {
                Raw r[K];
#pragma unroll
                for (int j = 0; j < K; ++j)
                    r[j] = *reinterpret_cast<const Raw *>(sb + static_cast<size_t>(j) * kTileBytes +
                                                          static_cast<size_t>(lv) * kVecBytes);
                combine_vector<K, TIn, TOut, CAP>(a, w, scale, r, dst, v, euler);
            }
        }
        if (tile == L.tile_end - 1)
            combine_tail<K, TIn, TOut, CAP>(a, w, scale, L, dst, nvec, euler);
        __syncthreads();  // every thread is done reading this stage
        if (threadIdx.x == 0 && tile + S < t_hi) issue(tile + S, stage);
    }
}

// ------------------------------------------------------------------ launch plumbing
//
// The launchers keep a few values computed on first use (SM counts, occupancies, whether a
// kernel's shared-memory attribute was set on a device).  Handles may be driven from
// several host threads at once, so these caches are atomics; threads that race to fill
// one store the same value.

// Pipeline CTAs per SM, each with its own ring (a launch-shape knob: two measured slower at
// every H).
#ifndef BC_TMA_CTAS_PER_SM
#define BC_TMA_CTAS_PER_SM 1
#endif

// SM count of the current device, cached per device.
inline int sm_count() {
    static std::atomic<int> cached[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
    if (dev >= 64) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        return n > 0 ? n : 1;
    }
    int c = cached[dev].load(std::memory_order_relaxed);
    if (c == 0) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        c = n > 0 ? n : 1;
        cached[dev].store(c, std::memory_order_relaxed);
    }
    return c;
}

// Resident CTAs per SM for a kernel, optionally capped (the forecast runs best at two
// 256-thread CTAs per SM; the single-stream copy at full occupancy).
template <class KernelPtr>
int resident_ctas(KernelPtr kern, std::atomic<int> &cache, int cap) {
    int c = cache.load(std::memory_order_relaxed);
    if (c == 0) {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, kThreads, 0) != cudaSuccess ||
            n < 1)
            n = 1;
        if (cap > 0 && cap < n) n = cap;
        c = n;
        cache.store(c, std::memory_order_relaxed);
    }
    return c;
}

// Copy the layers into `dst` with their tile prefix sums; returns the number of tiles.
inline int64_t fill_entries(LayerEntry *dst, const LayerEntry *layers, int n, int elem_bytes,
                            int vec_bytes, int tile_vecs) {
    const TileCounter tiles_of(elem_bytes, vec_bytes, tile_vecs);
    int64_t tiles = 0;
    for (int i = 0; i < n; ++i) {
        dst[i] = layers[i];
        tiles += tiles_of(layers[i].numel);
        dst[i].tile_end = tiles;
    }
    return tiles;
}

// Make the handle's device table hold `entries[0..n)` for a launch on `s`: one
// cudaMemcpyAsync on `s` from the next pinned staging buffer, skipped when the previous upload
// was the same table.  A staging buffer is rewritten only after the copy that last read it has
// run (its event).  `s` first waits for the last launch that read the table, whatever stream
// it went to (on that same stream the wait is already met): that launch may still be reading
// the table this copy overwrites, and a launch that reuses the table must follow the copy
// queued ahead of it.  Stream handles are not compared, since a destroyed stream's handle can
// come back as a new stream.
inline int upload_table(DeviceTable &tb, const LayerEntry *entries, int n, cudaStream_t s) {
    const size_t bytes = sizeof(LayerEntry) * static_cast<size_t>(n);
    if (tb.used_recorded) {
        const cudaError_t e = cudaStreamWaitEvent(s, static_cast<cudaEvent_t>(tb.used), 0);
        if (e != cudaSuccess) return e;
    }
    if (tb.valid == n && tb.last >= 0 &&
        std::memcmp(tb.host + static_cast<size_t>(tb.last) * tb.capacity, entries, bytes) == 0)
        return cudaSuccess;
    const int k = (tb.last + 1) % kTableStaging;
    cudaEvent_t ev = static_cast<cudaEvent_t>(tb.uploaded[k]);
    if (tb.pending[k]) {
        const cudaError_t e = cudaEventSynchronize(ev);
        if (e != cudaSuccess) return e;
        tb.pending[k] = false;
    }
    LayerEntry *stage = tb.host + static_cast<size_t>(k) * tb.capacity;
    std::memcpy(stage, entries, bytes);
    tb.valid = 0;
    cudaError_t e = cudaMemcpyAsync(tb.dev, stage, bytes, cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return e;
    e = cudaEventRecord(ev, s);
    if (e != cudaSuccess) return e;
    tb.pending[k] = true;
    tb.last = k;
    tb.valid = n;
    ++tb.uploads;
    return cudaSuccess;
}

// Record that a launch on `s` reads the table (after the launch, on `s`).
inline int table_used(DeviceTable &tb, cudaStream_t s) {
    const cudaError_t e = cudaEventRecord(static_cast<cudaEvent_t>(tb.used), s);
    if (e != cudaSuccess) return e;
    tb.used_recorded = true;
    return cudaSuccess;
}

// Fill a.start[] with the layer of every CTA's first tile (contiguous ranges of
// ceil(total / grid) tiles), as the kernels would find it: the first layer whose tiles reach
// past that tile (the last layer if none does), by binary search over the prefix sums, so
// that tables of many thousands of layers are not walked once more per call.
template <int CAP>
inline void fill_starts(ForecastArgs<CAP> &a, const LayerEntry *tab, int n, int64_t grid) {
    a.n_starts = 0;
    if (grid > kMaxStartCtas || grid < 1) return;
    const int64_t per_cta = (a.total_tiles + grid - 1) / grid;
    for (int64_t c = 0; c < grid; ++c) {
        const int64_t t = c * per_cta;
        int lo = 0, hi = n - 1;
        while (lo < hi) {
            const int mid = lo + (hi - lo) / 2;
            if (tab[mid].tile_end > t)
                hi = mid;
            else
                lo = mid + 1;
        }
        a.start[c].layer = lo;
        a.start[c].first = lo > 0 ? tab[lo - 1].tile_end : 0;
    }
    a.n_starts = static_cast<int32_t>(grid);
}

// Host staging for the tile prefix sums of a device-table launch (one per host thread).
inline std::vector<LayerEntry> &table_scratch() {
    static thread_local std::vector<LayerEntry> v;
    return v;
}

template <int K, class TIn, class TOut, int CAP>
int launch_group(const LaunchPlan &p, const LayerEntry *layers, int n, int euler_local,
                 cudaStream_t s, int64_t *launches, int64_t *pipeline_launches) {
    ForecastArgs<CAP> a;
    memset(&a, 0, sizeof a);
    for (int j = 0; j < BC_MAX_K; ++j) {
        a.slot[j] = p.slot[j];
        a.w[j] = p.w[j];
    }
    a.scale = p.scale;
    a.ca = p.ca;
    a.cb = p.cb;
    a.cc = p.cc;
    a.z = p.z;
    a.euler_layer = euler_local;
    a.x_bf16 = p.x_dtype == BC_DTYPE_BF16 ? 1 : 0;
    a.x = p.x;
    a.status = p.status;
    a.inject = p.inject;
    a.n_layers = n;
    const int sms = sm_count();

    // Kernel choice.  The pipeline kernel needs enough tiles per CTA to amortise filling its
    // ring; small launches (few or tiny layers) run the register kernel, and launches of
    // under BC_SMALL_LAUNCH_TILES_PER_SM of its tiles per SM use half-size tiles so that more
    // SMs and threads share the few round trips.  The layer table is filled (tile prefix
    // sums) with the tile shape of the kernel in question and filled again only when the
    // choice falls on another shape (at H <= 3 both kernels share one).
    constexpr int kRegVpt = kVecsPerThreadFor<K>;
    constexpr int kTmaTile = kThreads * kTmaVpt<K>, kRegTile = kThreads * kRegVpt;
    const bool forced = p.kernel == BC_KERNEL_PIPELINE || p.inject;
    const bool weigh = !forced && p.kernel == BC_KERNEL_AUTO && (K <= 3 || BC_TMA_AUTO_K4);
    LayerEntry *tab;
    if constexpr (CAP == 0) {
        std::vector<LayerEntry> &v = table_scratch();
        v.resize(static_cast<size_t>(n));
        tab = v.data();
    } else {
        tab = a.layer;
    }
    int tile_vecs = forced || weigh ? kTmaTile : kRegTile;
    a.total_tiles = fill_entries(tab, layers, n, TIn::kBytes, kVecBytes, tile_vecs);
    bool pipeline = forced;
    if (weigh)
        pipeline = a.total_tiles >= static_cast<int64_t>(kTmaMinTilesPerCta) * sms &&
                   a.total_tiles >= static_cast<int64_t>(BC_TMA_MIN_TILES_PER_LAYER) * n;
    if (!pipeline && tile_vecs != kRegTile) {
        tile_vecs = kRegTile;
        a.total_tiles = fill_entries(tab, layers, n, TIn::kBytes, kVecBytes, tile_vecs);
    }
    if (!pipeline && CAP == kLayersSmall && p.kernel == BC_KERNEL_AUTO && kRegVpt > 1 &&
        a.total_tiles < static_cast<int64_t>(BC_SMALL_LAUNCH_TILES_PER_SM) * sms) {
        tile_vecs = kThreads;
        a.total_tiles = fill_entries(tab, layers, n, TIn::kBytes, kVecBytes, tile_vecs);
    }
    const int vpt = tile_vecs / kThreads;
    if (a.total_tiles == 0) return cudaSuccess;
    // the launch's error, after recording that a device-table launch reads its table
    auto launched = [&](cudaError_t e) -> int {
        if constexpr (CAP == 0) {
            const int r = table_used(*p.table, s);
            if (e == cudaSuccess) return r;
        }
        return e;
    };

    if constexpr (CAP == 0) {
        const int err = upload_table(*p.table, tab, n, s);
        if (err != cudaSuccess) return err;
        a.table = p.table->dev;
        // every CTA's first layer, as the kernels would find it (grid as launched below)
        int64_t grid_cap = static_cast<int64_t>(sms) * (pipeline ? BC_TMA_CTAS_PER_SM : 1);
        if (!pipeline) {
            static std::atomic<int> occ_reg{0};
            grid_cap *= resident_ctas(forecast_kernel<K, kRegVpt, TIn, TOut, 0>, occ_reg,
                                      BC_CTAS_PER_SM);
        }
        fill_starts(a, tab, n, a.total_tiles < grid_cap ? a.total_tiles : grid_cap);
    }

    if (pipeline) {
        // shared-memory pipeline, one CTA per SM
        auto kern = forecast_tma_kernel<K, TIn, TOut, CAP>;
        constexpr int smem = kTmaSmemBytes<K>;
        static std::atomic<bool> attr_set[64];
        const int err = ensure_smem_attribute(kern, attr_set, smem);
        if (err != cudaSuccess) return err;
        const int64_t cap = static_cast<int64_t>(sms) * BC_TMA_CTAS_PER_SM;
        const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
        kern<<<grid, kThreads, smem, s>>>(a);
        ++*launches;
        ++*pipeline_launches;
        return launched(cudaGetLastError());
    }
    if constexpr (CAP == kLayersSmall && kRegVpt > 1) {
        if (vpt == 1) {
            static std::atomic<int> occ{0};
            auto kern = forecast_kernel<K, 1, TIn, TOut, CAP>;
            const int64_t cap =
                static_cast<int64_t>(sms) * resident_ctas(kern, occ, BC_CTAS_PER_SM);
            const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
            kern<<<grid, kThreads, 0, s>>>(a);
            ++*launches;
            return cudaGetLastError();
        }
    }
    static std::atomic<int> occ{0};
    auto kern = forecast_kernel<K, kRegVpt, TIn, TOut, CAP>;
    const int64_t cap = static_cast<int64_t>(sms) * resident_ctas(kern, occ, BC_CTAS_PER_SM);
    const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
    kern<<<grid, kThreads, 0, s>>>(a);
    ++*launches;
    return launched(cudaGetLastError());
}

template <int K, class TIn, class TOut>
int launch_all(const LaunchPlan &p, cudaStream_t s, int64_t *launches, int64_t *pipe) {
    if (p.n_layers > kLayersLarge && p.table != nullptr && p.n_layers <= p.table->capacity)
        return launch_group<K, TIn, TOut, 0>(p, p.layers, p.n_layers, p.euler_layer, s, launches,
                                             pipe);
    int err = cudaSuccess;
    for (int base = 0; base < p.n_layers && err == cudaSuccess; base += kLayersLarge) {
        const int n = p.n_layers - base < kLayersLarge ? p.n_layers - base : kLayersLarge;
        const int eul = (p.euler_layer >= base && p.euler_layer < base + n) ? p.euler_layer - base
                                                                             : -1;
        if (n <= kLayersSmall)
            err = launch_group<K, TIn, TOut, kLayersSmall>(p, p.layers + base, n, eul, s, launches,
                                                           pipe);
        else if (n <= kLayersMedium)
            err = launch_group<K, TIn, TOut, kLayersMedium>(p, p.layers + base, n, eul, s,
                                                            launches, pipe);
        else
            err = launch_group<K, TIn, TOut, kLayersLarge>(p, p.layers + base, n, eul, s, launches,
                                                           pipe);
    }
    return err;
}

template <int K>
int dispatch_dtypes(const LaunchPlan &p, cudaStream_t s, int64_t *launches, int64_t *pipe) {
    const bool in_bf = p.in_dtype == BC_DTYPE_BF16, out_bf = p.out_dtype == BC_DTYPE_BF16;
    if (in_bf && out_bf) return launch_all<K, BF16, BF16>(p, s, launches, pipe);
    if (in_bf && !out_bf) return launch_all<K, BF16, F32>(p, s, launches, pipe);
    if (!in_bf && out_bf) return launch_all<K, F32, BF16>(p, s, launches, pipe);
    return launch_all<K, F32, F32>(p, s, launches, pipe);
}

}  // namespace
}  // namespace bc
