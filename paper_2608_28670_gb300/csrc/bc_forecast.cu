// bc_forecast.cu -- the device side of the skipped-step forecast (sm_103a).
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
// 32 bytes; tiles are numbered across layers by a prefix sum carried in the launch's
// parameter block; a persistent grid splits the tile space into one contiguous range per
// CTA, so every CTA streams sequential addresses.  Two kernels share the arithmetic
// (combine_vector / combine_tail, so they produce the same bits) and differ in how the
// history reaches the SM:
//   forecast_tma_kernel  H <= 3: TMA bulk copies into a three-stage shared-memory ring,
//                        one CTA per SM (7.33 TB/s at H = 3 on the 60-layer video
//                        workload);
//   forecast_kernel      H = 4 and small launches: every thread issues all of its 256-bit
//                        loads into registers before using any, two CTAs per SM (7.24 TB/s
//                        at H = 3, 7.21 at H = 4).
// The path from 6.96 TB/s (128-bit register loads, three CTAs per SM, grid stride) to
// these numbers came from sweeps of vector width, vectors per thread, CTA size and count,
// cache hints, tile order, ring depth and store path on that workload.
//
// The file also holds the push's grouped byte-exact copy on the same layer tables:
// copy_tma_kernel (TMA bulk loads and stores through a three-stage ring, one warp per SM;
// large pushes) and copy_kernel (16-byte register copies; small pushes).
//
// Outputs, the sampler state and push sources carry only the ABI's 16-byte alignment and
// use 128-bit (or 64-bit) accesses; stores are st.global.cs (streaming).  No CTA waits on
// another, nothing allocates and nothing traps: every vector index is checked against its
// layer's length, and the pipeline kernel's waits on its own mbarriers are bounded.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <type_traits>

#include "bc_internal.h"
#include "bc_tma.cuh"

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

// Place a layer cursor on the layer holding `tile`: a binary search over the tiles' prefix
// sums (about ten dependent parameter loads for a full table, where a scan from layer 0
// would take up to one per layer); `first` is the layer's first tile.
template <int CAP>
__device__ __forceinline__ void find_layer(const ForecastArgs<CAP> &a, int64_t tile, int &l,
                                           int64_t &first) {
    int lo = 0, hi = a.n_layers - 1;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (tile < a.layer[mid].tile_end)
            hi = mid;
        else
            lo = mid + 1;
    }
    l = lo;
    first = lo > 0 ? a.layer[lo - 1].tile_end : 0;
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

// Forecast one history vector from its K raw pieces (node order j = 1..K), store it, and
// on the update layer apply x <- ca x + cb v_hat (+ cc z) to the same elements.
template <int K, class TIn, class TOut, int CAP>
__device__ __forceinline__ void combine_vector(const ForecastArgs<CAP> &a, const float *w,
                                               const Raw *r, char *dst, int64_t v, bool euler) {
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
    if (dst) store_stream<TOut, EV>(dst + v * EV * TOut::kBytes, acc);
    if (euler) {
        // Sampler update on the same elements: x <- ca x + cb v_hat (+ cc z).
        float x[EV];
        char *xp = reinterpret_cast<char *>(a.x);
        const char *zp = reinterpret_cast<const char *>(a.z);
        if (a.x_bf16) {
            xp += v * EV * 2;
            load_plain<BF16, EV>(xp, x);
#pragma unroll
            for (int e = 0; e < EV; ++e) x[e] = fmaf(a.cb, acc[e], a.ca * x[e]);
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
            for (int e = 0; e < EV; ++e) x[e] = fmaf(a.cb, acc[e], a.ca * x[e]);
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
                                             const LayerEntry &L, char *dst, int64_t nvec,
                                             bool euler) {
    constexpr int EV = kVecBytes / TIn::kBytes;
    const int rem = static_cast<int>(L.numel - nvec * EV);
    if (rem == 0 || static_cast<int>(threadIdx.x) >= rem) return;
    const int64_t e = nvec * EV + threadIdx.x;
    float acc = w[0] * load_scalar<TIn>(reinterpret_cast<const char *>(a.slot[0] + L.src), e);
#pragma unroll
    for (int j = 1; j < K; ++j)
        acc = fmaf(w[j], load_scalar<TIn>(reinterpret_cast<const char *>(a.slot[j] + L.src), e),
                   acc);
    if (dst) store_scalar<TOut>(dst, e, acc);
    if (euler) {
        char *xb = reinterpret_cast<char *>(a.x);
        const char *zb = reinterpret_cast<const char *>(a.z);
        if (a.x_bf16) {
            float xn = fmaf(a.cb, acc, a.ca * load_scalar<BF16>(xb, e));
            if (zb) xn = fmaf(a.cc, load_scalar<BF16>(zb, e), xn);
            store_scalar<BF16>(xb, e, xn);
        } else {
            float xn = fmaf(a.cb, acc, a.ca * load_scalar<F32>(xb, e));
            if (zb) xn = fmaf(a.cc, load_scalar<F32>(zb, e), xn);
            store_scalar<F32>(xb, e, xn);
        }
    }
}

// The grouped forecast with register-held history loads (used at H = 4, where the
// shared-memory pipeline below does not pay): each thread issues all H x VPT loads of its
// tile before using any of them.
template <int K, class TIn, class TOut, int CAP>
__global__ void __launch_bounds__(kThreads)
    forecast_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int kVecsPerThread = kVecsPerThreadFor<K>;
    constexpr int kTileVecs = kThreads * kVecsPerThread;
    const uint64_t pol = history_policy();
    float w[K];
#pragma unroll
    for (int j = 0; j < K; ++j) w[j] = a.w[j];

    // Each CTA streams one contiguous range of tiles (better DRAM page locality than a
    // grid stride: 7.24 vs 7.18 TB/s on the video workload at H = 3).
    const int64_t per_cta = (a.total_tiles + gridDim.x - 1) / gridDim.x;
    const int64_t t_lo = static_cast<int64_t>(blockIdx.x) * per_cta;
    const int64_t t_hi = t_lo + per_cta < a.total_tiles ? t_lo + per_cta : a.total_tiles;
    if (t_lo >= t_hi) return;
    int l;
    int64_t first;
    find_layer(a, t_lo, l, first);
    for (int64_t tile = t_lo; tile < t_hi; ++tile) {
        seek_layer(a, tile, l, first);
        const LayerEntry &L = a.layer[l];
        const int64_t nvec = L.numel / (kVecBytes / TIn::kBytes);
        const int64_t v0 = (tile - first) * kTileVecs + threadIdx.x;
        const char *src[K];
#pragma unroll
        for (int j = 0; j < K; ++j) src[j] = reinterpret_cast<const char *>(a.slot[j] + L.src);
        char *dst = reinterpret_cast<char *>(L.dst);
        const bool euler = (l == a.euler_layer);

        Raw r[kVecsPerThread][K];
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) {
#pragma unroll
                for (int j = 0; j < K; ++j) r[u][j] = ld_history(src[j] + v * kVecBytes, pol);
            }
        }
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
            const int64_t v = v0 + u * kThreads;
            if (v < nvec) combine_vector<K, TIn, TOut, CAP>(a, w, r[u], dst, v, euler);
        }
        if (tile == L.tile_end - 1) combine_tail<K, TIn, TOut, CAP>(a, w, L, dst, nvec, euler);
    }
}

// ---------------------------------------------------------------------------------------
// The grouped forecast with the history staged through shared memory by the Tensor Memory
// Accelerator (H <= 3).  Each CTA (one per SM) owns a ring of kTmaStages stages; a stage
// holds one tile of every history slot (H x 16 KiB).  Thread 0 issues one 1-D bulk copy
// (cp.async.bulk, global -> shared) per slot and tile, completing on the stage's mbarrier
// with a transaction count; all threads wait on that mbarrier, combine from shared memory
// and store to global memory directly; after a CTA barrier thread 0 refills the stage with
// the tile kTmaStages ahead.  Three 48 KiB stages in flight per SM sustain 7.35 TB/s at
// H = 3 on the video workload (7.27 TB/s with register-held loads); the outputs are
// bit-identical to the register kernel's.
//
// Every wait is bounded (about one second by %globaltimer): on expiry the CTA records the
// failure in the handle's device status word, drains the copies it issued (again bounded)
// and returns, so a lost completion can never hang the device; the host reads the word
// with bc_cache_check.
constexpr int kTmaStages = 3;
constexpr int kTmaMinTilesPerCta = 16;

// Bytes of one history tile, and of the whole ring (kTmaStages stages of K tiles).
template <int K>
constexpr int kTmaTileBytes = kThreads * kVecsPerThreadFor<K> * kVecBytes;
template <int K>
constexpr int kTmaSmemBytes = kTmaStages * K * kTmaTileBytes<K>;

template <int K, class TIn, class TOut, int CAP>
__global__ void __launch_bounds__(kThreads)
    forecast_tma_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int kVecsPerThread = kVecsPerThreadFor<K>;
    constexpr int kTileVecs = kThreads * kVecsPerThread;
    constexpr int kTileBytes = kTmaTileBytes<K>;
    constexpr int EV = kVecBytes / TIn::kBytes;
    constexpr int S = kTmaStages;
    extern __shared__ __align__(128) unsigned char stage_mem[];
    __shared__ __align__(8) uint64_t full[S];
    __shared__ int abort_flag;

    float w[K];
#pragma unroll
    for (int j = 0; j < K; ++j) w[j] = a.w[j];
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
    auto issue = [&](int64_t tile, int stage) {
        seek_layer(a, tile, pl, pfirst);
        const LayerEntry &L = a.layer[pl];
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
        find_layer(a, t_lo, pl, pfirst);
        for (int i = 0; i < S && t_lo + i < t_hi; ++i) issue(t_lo + i, i);
    }

    int l = 0;
    int64_t first = 0;
    if (t_lo < t_hi) find_layer(a, t_lo, l, first);
    for (int64_t tile = t_lo; tile < t_hi; ++tile) {
        const int64_t i = tile - t_lo;
        const int stage = static_cast<int>(i % S);
        if (!mbar_wait_bounded(&full[stage], static_cast<uint32_t>((i / S) & 1))) abort_flag = 1;
        __syncthreads();  // the exit decision below is the same for every thread
        if (abort_flag) {
            if (threadIdx.x == 0) {
                if (a.status) atomicOr(a.status, 1u);
                // drain the copies this CTA issued and has not consumed (bounded)
                for (int64_t k = i; k < issued; ++k)
                    mbar_wait_bounded(&full[k % S], static_cast<uint32_t>((k / S) & 1));
            }
            return;
        }
        seek_layer(a, tile, l, first);
        const LayerEntry &L = a.layer[l];
        const int64_t nvec = L.numel / EV;
        const int64_t v0 = (tile - first) * kTileVecs;
        char *dst = reinterpret_cast<char *>(L.dst);
        const bool euler = (l == a.euler_layer);
        const unsigned char *sb = stage_mem + static_cast<size_t>(stage) * K * kTileBytes;
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
            const int lv = u * kThreads + threadIdx.x;
            const int64_t v = v0 + lv;
            if (v < nvec) {
                Raw r[K];
#pragma unroll
                for (int j = 0; j < K; ++j)
                    r[j] = *reinterpret_cast<const Raw *>(sb + static_cast<size_t>(j) * kTileBytes +
                                                          static_cast<size_t>(lv) * kVecBytes);
                combine_vector<K, TIn, TOut, CAP>(a, w, r, dst, v, euler);
            }
        }
        if (tile == L.tile_end - 1) combine_tail<K, TIn, TOut, CAP>(a, w, L, dst, nvec, euler);
        __syncthreads();  // every thread is done reading this stage
        if (threadIdx.x == 0 && tile + S < t_hi) issue(tile + S, stage);
    }
}

// Grouped byte-exact copy for the push: layer.src -> layer.dst, numel elements of T.
// Always 16-byte vectors: the caller's source is only guaranteed 16-byte alignment.
template <class T, int CAP>
__global__ void __launch_bounds__(kThreads) copy_kernel(const __grid_constant__ ForecastArgs<CAP> a) {
    constexpr int kVecsPerThread = kCopyVecsPerThread;
    constexpr int kTileVecs = kThreads * kVecsPerThread;
    constexpr int EV = 16 / T::kBytes;
    int l = 0;
    int64_t first = 0;
    if (blockIdx.x < a.total_tiles) find_layer(a, blockIdx.x, l, first);
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
    find_layer(a, t_lo, pl, pfirst);
    int64_t issued = 0;
    auto issue = [&](int64_t tile, int stage) {
        seek_layer(a, tile, pl, pfirst);
        const LayerEntry &L = a.layer[pl];
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
    find_layer(a, t_lo, l, first);
    for (int64_t tile = t_lo; tile < t_hi; ++tile) {
        const int64_t i = tile - t_lo;
        const int stage = static_cast<int>(i % S);
        int ok = 1;
        if (lane == 0) ok = mbar_wait_bounded(&full[stage], static_cast<uint32_t>((i / S) & 1));
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
            if (lane == 0) {
                if (a.status) atomicOr(a.status, 1u);
                for (int64_t k = i; k < issued; ++k)
                    mbar_wait_bounded(&full[k % S], static_cast<uint32_t>((k / S) & 1));
                bulk_wait_group_all();
            }
            return;
        }
        seek_layer(a, tile, l, first);
        const LayerEntry &L = a.layer[l];
        const int64_t nvec = L.numel / EV;
        if (lane == 0) {
            const int64_t g0 = (tile - first) * kTileGroups;
            int64_t ng = nvec - g0;
            ng = ng > kTileGroups ? kTileGroups : (ng < 0 ? 0 : ng);
            if (ng > 0) {
                fence_proxy_async_shared();
                bulk_store_from_shared(reinterpret_cast<char *>(L.dst) + g0 * 16,
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
            reinterpret_cast<St *>(L.dst)[e] = reinterpret_cast<const St *>(L.src)[e];
        }
    }
    if (lane == 0) bulk_wait_group_all();
}

// ------------------------------------------------------------------ launch plumbing
//
// The launchers keep a few values computed on first use (SM counts, occupancies, whether a
// kernel's shared-memory attribute was set on a device).  Handles may be driven from
// several host threads at once, so these caches are atomics; threads that race to fill
// one store the same value.

// SM count of the current device, cached per device.
int sm_count() {
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


template <int CAP>
int64_t fill_table(ForecastArgs<CAP> &a, const LayerEntry *layers, int n, int elem_bytes,
                   int vec_bytes, int tile_vecs) {
    int64_t tiles = 0;
    for (int i = 0; i < n; ++i) {
        a.layer[i] = layers[i];
        tiles += tiles_for(layers[i].numel, elem_bytes, vec_bytes, tile_vecs);
        a.layer[i].tile_end = tiles;
    }
    a.n_layers = n;
    return tiles;
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
    a.ca = p.ca;
    a.cb = p.cb;
    a.cc = p.cc;
    a.z = p.z;
    a.euler_layer = euler_local;
    a.x_bf16 = p.x_dtype == BC_DTYPE_BF16 ? 1 : 0;
    a.x = p.x;
    a.status = p.status;
    a.inject = p.inject;
    a.total_tiles =
        fill_table(a, layers, n, TIn::kBytes, kVecBytes, kThreads * kVecsPerThreadFor<K>);
    if (a.total_tiles == 0) return cudaSuccess;
    // The pipeline kernel (H <= 3) needs enough tiles per CTA to amortise filling its ring;
    // small launches (few or tiny layers) run the register kernel.
    bool pipeline = false;
    if constexpr (K <= 3)
        pipeline = p.kernel == BC_KERNEL_PIPELINE || p.inject ||
                   (p.kernel == BC_KERNEL_AUTO &&
                    a.total_tiles >= static_cast<int64_t>(kTmaMinTilesPerCta) * sm_count());
    if constexpr (K <= 3) {
      if (pipeline) {
        // shared-memory pipeline, one CTA per SM
        auto kern = forecast_tma_kernel<K, TIn, TOut, CAP>;
        constexpr int smem = kTmaSmemBytes<K>;
        static std::atomic<bool> attr_set[64];
        const int err = ensure_smem_attribute(kern, attr_set, smem);
        if (err != cudaSuccess) return err;
        const int64_t cap = sm_count();
        const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
        kern<<<grid, kThreads, smem, s>>>(a);
        ++*launches;
        ++*pipeline_launches;
        return cudaGetLastError();
      }
    }
    static std::atomic<int> occ{0};
    auto kern = forecast_kernel<K, TIn, TOut, CAP>;
    const int64_t cap =
        static_cast<int64_t>(sm_count()) * resident_ctas(kern, occ, BC_CTAS_PER_SM);
    const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
    kern<<<grid, kThreads, 0, s>>>(a);
    ++*launches;
    return cudaGetLastError();
}

template <int K, class TIn, class TOut>
int launch_all(const LaunchPlan &p, cudaStream_t s, int64_t *launches, int64_t *pipe) {
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

template <class T, int CAP>
int copy_group(const LayerEntry *layers, int n, const CopyOptions &opt, cudaStream_t s,
               int64_t *launches, int64_t *pipeline_launches) {
    static std::atomic<int> occ{0};
    ForecastArgs<CAP> a;
    memset(&a, 0, sizeof a);
    a.euler_layer = -1;
    a.status = opt.status;
    a.inject = opt.inject;
    // The bulk-copy pipeline needs enough of its 32 KiB tiles per SM to amortise its ring.
    a.total_tiles = fill_table(a, layers, n, T::kBytes, 16, kCopyTileBytes / 16);
    if (a.total_tiles == 0) return cudaSuccess;
    const bool pipeline =
        opt.kernel == BC_KERNEL_PIPELINE || opt.inject ||
        (opt.kernel == BC_KERNEL_AUTO &&
         a.total_tiles >= static_cast<int64_t>(kCopyMinTilesPerCta) * sm_count());
    if (pipeline) {
        auto kern = copy_tma_kernel<T, CAP>;
        static std::atomic<bool> attr_set[64];
        const int err = ensure_smem_attribute(kern, attr_set, kCopySmemBytes);
        if (err != cudaSuccess) return err;
        const int64_t cap = static_cast<int64_t>(sm_count()) * BC_COPY_CTAS_PER_SM;
        const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
        kern<<<grid, kCopyTmaThreads, kCopySmemBytes, s>>>(a);
        ++*launches;
        ++*pipeline_launches;
        return cudaGetLastError();
    }
    a.total_tiles = fill_table(a, layers, n, T::kBytes, 16, kThreads * kCopyVecsPerThread);
    auto kern = copy_kernel<T, CAP>;
    const int64_t cap = static_cast<int64_t>(sm_count()) * resident_ctas(kern, occ, 0);
    const int grid = static_cast<int>(a.total_tiles < cap ? a.total_tiles : cap);
    kern<<<grid, kThreads, 0, s>>>(a);
    ++*launches;
    return cudaGetLastError();
}

template <class T>
int copy_all(const LayerEntry *layers, int n_layers, const CopyOptions &opt, cudaStream_t s,
             int64_t *launches, int64_t *pipe) {
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
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    switch (plan.K) {
    case 1: return dispatch_dtypes<1>(plan, s, launches, pipeline_launches);
    case 2: return dispatch_dtypes<2>(plan, s, launches, pipeline_launches);
    case 3: return dispatch_dtypes<3>(plan, s, launches, pipeline_launches);
    case 4: return dispatch_dtypes<4>(plan, s, launches, pipeline_launches);
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
