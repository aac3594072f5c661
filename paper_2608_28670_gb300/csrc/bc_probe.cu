// bc_probe.cu -- relative L1 drift of a feature probe between two consecutive steps, the
// signal of the adaptive schedule (Sec. 4.5: a full step is triggered once the
// accumulated relative change of a feature probe exceeds a threshold).
//
//     drift = sum_e |cur[e] - prev[e]| / sum_e |prev[e]|
//
// Two launches with a fixed reduction order, so the result is bitwise reproducible for a
// given device: (1) a persistent grid streams both tensors once in 16-byte groups, each
// thread sums a group in fp32 and accumulates the group sums with compensated (Kahan) fp32
// addition, so the error stays near two fp32 ulps however long the stream is, without
// touching GB300's slow fp64 pipe per element; every CTA adds its threads' sums with a
// fixed compensated fp32 shuffle tree, converts once per warp to fp64 and writes its two
// partial sums to scratch; (2) one CTA adds the partials in a fixed order and writes
// {sum |d|, sum |prev|, ratio}.  HBM-bound: 2 * n * sizeof(T) bytes, no atomics.
// The first launch comes in two forms: drift_partials (register loads, four groups in
// flight per thread, grid stride; small probes) and drift_tma_partials (one CTA per SM
// streaming a contiguous range of tiles through a five-stage TMA ring in shared memory;
// large probes), whose only waits are on its own mbarriers and are bounded.  On a 365 M
// element bf16 probe pair: 6.98 TB/s with five 2 x 16 KiB stages (four: 6.91, three: 6.75,
// six: 6.80, 2 x 32 KiB stages x 2 / x 3: 6.91 / 6.73, eight 2 x 8 KiB: 5.16), register
// loads 6.84.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "bc_internal.h"
#include "bc_tma.cuh"

namespace bc {
namespace {

constexpr int kProbeThreads = 256;

__device__ __forceinline__ uint4 ld_nc16(const void *p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p));
    return r;
}

template <bool kBf16>
__device__ __forceinline__ void unpack(uint4 r, float *f) {
    if constexpr (kBf16) {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    } else {
        f[0] = __uint_as_float(r.x); f[1] = __uint_as_float(r.y);
        f[2] = __uint_as_float(r.z); f[3] = __uint_as_float(r.w);
    }
}

template <bool kBf16>
__device__ __forceinline__ float load1(const char *p, int64_t e) {
    if constexpr (kBf16)
        return __uint_as_float(static_cast<uint32_t>(reinterpret_cast<const uint16_t *>(p)[e]) << 16);
    return reinterpret_cast<const float *>(p)[e];
}

// Compensated fp32 accumulator (Kahan): the rounding error of every addition is carried
// into the next, so a long sum keeps about fp32 precision.  Inputs are sums of |x| >= 0.
struct Kahan {
    float s = 0.0f, c = 0.0f;
    __device__ __forceinline__ void add(float x) {
        const float y = x - c;
        const float t = s + y;
        c = (t - s) - y;
        s = t;
    }
};

// Sum |c - p| and |p| over one 16-byte group of each tensor (fp32, fixed order).
template <bool kBf16>
__device__ __forceinline__ void group_sums(uint4 rc, uint4 rp, float &gd, float &gp) {
    constexpr int ev = kBf16 ? 8 : 4;
    float c[8], p[8];
    unpack<kBf16>(rc, c);
    unpack<kBf16>(rp, p);
    gd = 0.0f;
    gp = 0.0f;
#pragma unroll
    for (int e = 0; e < ev; ++e) {
        gd += fabsf(c[e] - p[e]);
        gp += fabsf(p[e]);
    }
}

constexpr int kGroupsInFlight = 4;

// Fixed-order tree sums of two doubles per thread over the CTA (kProbeThreads threads):
// a shuffle tree within each warp, then warp 0 sums the warps' results the same way, so
// the order never changes (bitwise reproducible) and the CTA waits at three barriers, not
// at one per tree level (the fp64 adds are on GB300's slow fp64 pipe, so every level is
// latency on the critical path).  `sh` holds at least 2 x (kProbeThreads / 32) doubles.
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
    return v;  // lane 0
}

__device__ __forceinline__ void block_sum2(double &a, double &b, double *sh) {
    constexpr int kWarps = kProbeThreads / 32;
    const int w = static_cast<int>(threadIdx.x) / 32, lane = static_cast<int>(threadIdx.x) % 32;
    a = warp_sum(a);
    b = warp_sum(b);
    if (lane == 0) {
        sh[w] = a;
        sh[kWarps + w] = b;
    }
    __syncthreads();
    if (w == 0) {
        double ra = lane < kWarps ? sh[lane] : 0.0;
        double rb = lane < kWarps ? sh[kWarps + lane] : 0.0;
        ra = warp_sum(ra);
        rb = warp_sum(rb);
        if (lane == 0) {
            sh[0] = ra;
            sh[1] = rb;
        }
    }
    __syncthreads();
    a = sh[0];
    b = sh[1];
    __syncthreads();  // `sh` may be written again right after
}

// A compensated fp32 value hi + lo.  Two of them add with Knuth's error-free TwoSum on the
// high parts (the rounding error of hi_a + hi_b is recovered exactly) and a plain sum of the
// low parts, so a tree of them keeps about twice fp32's precision on the fast fp32 pipe.
struct F2 {
    float hi, lo;
};

__device__ __forceinline__ F2 f2_add(F2 a, F2 b) {
    const float s = a.hi + b.hi;
    const float bv = s - a.hi;
    const float e = (a.hi - (s - bv)) + (b.hi - bv);
    return {s, (a.lo + b.lo) + e};
}

__device__ __forceinline__ F2 warp_sum_f2(F2 v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const F2 u{__shfl_down_sync(0xffffffffu, v.hi, o), __shfl_down_sync(0xffffffffu, v.lo, o)};
        v = f2_add(v, u);
    }
    return v;  // lane 0
}

// CTA sums of every thread's two Kahan accumulators, in a fixed order: a compensated fp32
// shuffle tree within each warp, one conversion to fp64 per warp, and thread 0 adds the
// warps' sums in warp order.  The results are valid in thread 0.  The only fp64 work is the
// per-warp conversion and eight additions: GB300 issues about two fp64 operations per cycle
// per SM, so a per-thread fp64 tree costs microseconds per launch.  `sh` holds at least
// 2 x (kProbeThreads / 32) doubles.
__device__ __forceinline__ void block_sum_kahan(const Kahan &a, const Kahan &b, double *sh,
                                                double &ra, double &rb) {
    constexpr int kWarps = kProbeThreads / 32;
    const int w = static_cast<int>(threadIdx.x) / 32, lane = static_cast<int>(threadIdx.x) % 32;
    const F2 va = warp_sum_f2({a.s, -a.c});  // a Kahan sum is s - c
    const F2 vb = warp_sum_f2({b.s, -b.c});
    if (lane == 0) {
        sh[w] = static_cast<double>(va.hi) + static_cast<double>(va.lo);
        sh[kWarps + w] = static_cast<double>(vb.hi) + static_cast<double>(vb.lo);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double sa = 0.0, sb = 0.0;
        for (int i = 0; i < kWarps; ++i) {
            sa += sh[i];
            sb += sh[kWarps + i];
        }
        ra = sa;
        rb = sb;
    }
    __syncthreads();  // `sh` may be written again right after
}

template <bool kBf16>
__global__ void __launch_bounds__(kProbeThreads)
    drift_partials(const char *cur, const char *prev, int64_t n, double *partials) {
    __shared__ double sh[kProbeThreads];
    constexpr int ev = kBf16 ? 8 : 4;
    const int64_t nvec = n / ev;
    Kahan sd, sp;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * kProbeThreads * kGroupsInFlight;
    for (int64_t base = static_cast<int64_t>(blockIdx.x) * kProbeThreads * kGroupsInFlight +
                        threadIdx.x;
         base < nvec; base += stride) {
        uint4 rc[kGroupsInFlight], rp[kGroupsInFlight];
#pragma unroll
        for (int u = 0; u < kGroupsInFlight; ++u) {
            const int64_t g = base + static_cast<int64_t>(u) * kProbeThreads;
            if (g < nvec) {
                rc[u] = ld_nc16(cur + g * 16);
                rp[u] = ld_nc16(prev + g * 16);
            }
        }
#pragma unroll
        for (int u = 0; u < kGroupsInFlight; ++u) {
            const int64_t g = base + static_cast<int64_t>(u) * kProbeThreads;
            if (g < nvec) {
                float gd, gp;
                group_sums<kBf16>(rc[u], rp[u], gd, gp);
                sd.add(gd);
                sp.add(gp);
            }
        }
    }
    if (blockIdx.x == 0) {  // ragged tail: fewer than one 16-byte group
        const int64_t e = nvec * ev + threadIdx.x;
        if (e < n) {
            const float c = load1<kBf16>(cur, e), p = load1<kBf16>(prev, e);
            sd.add(fabsf(c - p));
            sp.add(fabsf(p));
        }
    }
    double bd = 0.0, bp = 0.0;
    block_sum_kahan(sd, sp, sh, bd, bp);
    if (threadIdx.x == 0) {
        partials[2 * blockIdx.x] = bd;
        partials[2 * blockIdx.x + 1] = bp;
    }
}

// ---- shared-memory pipeline form: a stage holds one tile (kDriftTileBytes) of each
// tensor; thread 0 refills a stage with the tile kDriftStages ahead once every thread has
// read it (five stages: 160 KiB of shared memory).  A wait that runs out sets bit 0 of the status word, stores NaN partials (so the
// drift reads NaN), drains the copies in flight and returns.
#ifndef BC_DRIFT_STAGES
#define BC_DRIFT_STAGES 5
#endif
#ifndef BC_DRIFT_TILE_BYTES
#define BC_DRIFT_TILE_BYTES 16384
#endif
constexpr int kDriftStages = BC_DRIFT_STAGES;
constexpr int kDriftTileBytes = BC_DRIFT_TILE_BYTES;
constexpr int kDriftSmemBytes = kDriftStages * 2 * kDriftTileBytes;
constexpr int kDriftMinTilesPerCta = 16;

template <bool kBf16>
__global__ void __launch_bounds__(kProbeThreads)
    drift_tma_partials(const char *cur, const char *prev, int64_t n, double *partials,
                       uint32_t *status, int inject) {
    constexpr int S = kDriftStages;
    constexpr int kTileGroups = kDriftTileBytes / 16;
    constexpr int ev = kBf16 ? 8 : 4;
    extern __shared__ __align__(128) unsigned char stage_mem[];
    __shared__ __align__(8) uint64_t full[S];
    __shared__ double sh[kProbeThreads];
    __shared__ int abort_flag;
    const int64_t nvec = n / ev;
    const int64_t ntiles = (nvec + kTileGroups - 1) / kTileGroups;
    const int64_t per_cta = (ntiles + gridDim.x - 1) / gridDim.x;
    const int64_t t_lo = static_cast<int64_t>(blockIdx.x) * per_cta;
    const int64_t t_hi = t_lo + per_cta < ntiles ? t_lo + per_cta : ntiles;
    if (threadIdx.x == 0) {
        for (int i = 0; i < S; ++i) mbar_init(&full[i], 1);
        mbar_init_fence();
        abort_flag = 0;
    }
    __syncthreads();

    int64_t issued = 0;                 // thread 0 only
    auto issue = [&](int64_t tile, int stage) {
        const int64_t g0 = tile * kTileGroups;
        const int64_t ng = nvec - g0 < kTileGroups ? nvec - g0 : kTileGroups;
        const uint32_t bytes = static_cast<uint32_t>(ng * 16);
        unsigned char *dst = stage_mem + static_cast<size_t>(stage) * 2 * kDriftTileBytes;
        if (!(inject && issued == 0)) {   // the test hook leaves the first stage unarmed
            mbar_arrive_expect_tx(&full[stage], 2 * bytes);
            bulk_copy_to_shared(dst, cur + g0 * 16, bytes, &full[stage]);
            bulk_copy_to_shared(dst + kDriftTileBytes, prev + g0 * 16, bytes, &full[stage]);
        }
        ++issued;
    };
    if (threadIdx.x == 0)
        for (int i = 0; i < S && t_lo + i < t_hi; ++i) issue(t_lo + i, i);

    Kahan sd, sp;
    for (int64_t tile = t_lo; tile < t_hi; ++tile) {
        const int64_t i = tile - t_lo;
        const int stage = static_cast<int>(i % S);
        if (!mbar_wait_bounded(&full[stage], static_cast<uint32_t>((i / S) & 1))) abort_flag = 1;
        __syncthreads();  // the exit decision below is the same for every thread
        if (abort_flag) {
            if (threadIdx.x == 0) {
                if (status) atomicOr(status, 1u);
                const double nan = __longlong_as_double(0x7ff8000000000000LL);
                partials[2 * blockIdx.x] = nan;
                partials[2 * blockIdx.x + 1] = nan;
                // the stage the test hook left unarmed (the first issued) has no copy
                for (int64_t k = i; k < issued; ++k)
                    if (!(inject && k == 0))
                        mbar_wait_bounded(&full[k % S], static_cast<uint32_t>((k / S) & 1));
            }
            return;
        }
        const int64_t g0 = tile * kTileGroups;
        const int ng = static_cast<int>(nvec - g0 < kTileGroups ? nvec - g0 : kTileGroups);
        const unsigned char *sb = stage_mem + static_cast<size_t>(stage) * 2 * kDriftTileBytes;
        for (int g = threadIdx.x; g < ng; g += kProbeThreads) {
            const uint4 rc = *reinterpret_cast<const uint4 *>(sb + static_cast<size_t>(g) * 16);
            const uint4 rp = *reinterpret_cast<const uint4 *>(sb + kDriftTileBytes +
                                                              static_cast<size_t>(g) * 16);
            float gd, gp;
            group_sums<kBf16>(rc, rp, gd, gp);
            sd.add(gd);
            sp.add(gp);
        }
        __syncthreads();  // every thread is done reading this stage
        if (threadIdx.x == 0 && tile + S < t_hi) issue(tile + S, stage);
    }
    if (blockIdx.x == 0) {  // ragged tail: fewer than one 16-byte group
        const int64_t e = nvec * ev + threadIdx.x;
        if (e < n) {
            const float c = load1<kBf16>(cur, e), p = load1<kBf16>(prev, e);
            sd.add(fabsf(c - p));
            sp.add(fabsf(p));
        }
    }
    double bd = 0.0, bp = 0.0;
    block_sum_kahan(sd, sp, sh, bd, bp);
    if (threadIdx.x == 0) {
        partials[2 * blockIdx.x] = bd;
        partials[2 * blockIdx.x + 1] = bp;
    }
}

__global__ void __launch_bounds__(kProbeThreads)
    drift_final(const double *partials, int nparts, double *out) {
    __shared__ double sh[kProbeThreads];
    double sd = 0.0, sp = 0.0;
    for (int i = threadIdx.x; i < nparts; i += kProbeThreads) {
        sd += partials[2 * i];
        sp += partials[2 * i + 1];
    }
    block_sum2(sd, sp, sh);
    if (threadIdx.x == 0) {
        out[0] = sd;
        out[1] = sp;
        // 0 for an unchanged zero probe, +inf for a change of a zero probe, NaN if either
        // sum is NaN (a NaN in the probe, or a pipeline wait that gave up)
        double r = __longlong_as_double(0x7ff8000000000000LL);
        if (sp > 0.0)
            r = sd / sp;
        else if (sp == 0.0 && sd == 0.0)
            r = 0.0;
        else if (sp == 0.0 && sd > 0.0)
            r = __longlong_as_double(0x7ff0000000000000LL);
        out[2] = r;
    }
}

}  // namespace

int probe_ctas() {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int n = (sms > 0 ? sms : 1) * 4;
    return n < kProbeMaxCtas ? n : kProbeMaxCtas;
}

namespace {

int sm_count_of_current_device() {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms > 0 ? sms : 1;
}

// Launch the pipeline form on one CTA per SM (at most max_parts, at most one per tile).
template <bool kBf16>
int launch_drift_tma(const char *cur, const char *prev, int64_t n, int64_t ntiles,
                     double *partials, int max_parts, const DriftOptions &opt, cudaStream_t s,
                     int *grid_out) {
    auto kern = drift_tma_partials<kBf16>;
    static std::atomic<bool> attr_set[64];
    const int err = ensure_smem_attribute(kern, attr_set, kDriftSmemBytes);
    if (err != cudaSuccess) return err;
    int64_t grid = sm_count_of_current_device();
    if (grid > max_parts) grid = max_parts;
    if (grid > ntiles) grid = ntiles;
    if (grid < 1) grid = 1;
    kern<<<static_cast<int>(grid), kProbeThreads, kDriftSmemBytes, s>>>(cur, prev, n, partials,
                                                                        opt.status, opt.inject);
    *grid_out = static_cast<int>(grid);
    return cudaGetLastError();
}

}  // namespace

int launch_drift(const void *cur, const void *prev, int64_t n, bc_dtype dtype, double *partials,
                 int max_parts, double *out, const DriftOptions &opt, void *stream,
                 int64_t *launches, int64_t *pipeline_launches) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int ev = dtype == BC_DTYPE_BF16 ? 8 : 4;
    const int64_t nvec = n / ev;
    const char *c = static_cast<const char *>(cur);
    const char *p = static_cast<const char *>(prev);
    const int64_t ntiles = (nvec + kDriftTileBytes / 16 - 1) / (kDriftTileBytes / 16);
    const bool pipeline =
        ntiles > 0 && (opt.kernel == BC_KERNEL_PIPELINE || opt.inject ||
                       (opt.kernel == BC_KERNEL_AUTO &&
                        ntiles >= static_cast<int64_t>(kDriftMinTilesPerCta) *
                                      sm_count_of_current_device()));
    int grid = 0;
    int err = cudaSuccess;
    if (pipeline) {
        err = dtype == BC_DTYPE_BF16
                  ? launch_drift_tma<true>(c, p, n, ntiles, partials, max_parts, opt, s, &grid)
                  : launch_drift_tma<false>(c, p, n, ntiles, partials, max_parts, opt, s, &grid);
        if (err != cudaSuccess) return err;
        ++*pipeline_launches;
    } else {
        // one CTA per kProbeThreads x kGroupsInFlight groups: no CTA without data
        constexpr int64_t kCtaGroups = static_cast<int64_t>(kProbeThreads) * kGroupsInFlight;
        int64_t want = (nvec + kCtaGroups - 1) / kCtaGroups;
        if (want < 1) want = 1;
        grid = probe_ctas();
        if (grid > max_parts) grid = max_parts;
        if (want < grid) grid = static_cast<int>(want);
        if (dtype == BC_DTYPE_BF16)
            drift_partials<true><<<grid, kProbeThreads, 0, s>>>(c, p, n, partials);
        else
            drift_partials<false><<<grid, kProbeThreads, 0, s>>>(c, p, n, partials);
        err = cudaGetLastError();
        if (err != cudaSuccess) return err;
    }
    ++*launches;
    drift_final<<<1, kProbeThreads, 0, s>>>(partials, grid, out);
    ++*launches;
    return cudaGetLastError();
}

}  // namespace bc

// ---------------------------------------------------------------------------------------
// No-allocation variant (bc_probe_drift_noalloc).
//
// For callers that must not allocate device memory themselves nor have the library do it
// for them, the scratch of the reduction lives in a file-scope device array that exists
// for as long as the library is loaded, on every device that loads it.  Unlike the handle
// variant above (one partial per CTA of a device-sized grid), this variant writes one
// partial pair per fixed tile of the input, so its scratch need grows with the input and
// is bounded by the array: kStaticDriftMaxTiles tiles of kStaticDriftTileGroups x 256
// sixteen-byte groups, i.e. 1 GiB per probe tensor.  Every partial the final pass reads is
// written earlier in the same call, so nothing needs clearing between calls; calls that
// overlap on the device share the array and race.
static __device__ __align__(256) double g_drift_scratch[2 * bc::kStaticDriftMaxTiles];

namespace bc {
namespace {

template <bool kBf16>
__global__ void __launch_bounds__(kProbeThreads)
    drift_tile_partials(const char *cur, const char *prev, int64_t n, int64_t ntiles,
                        double *partials) {
    __shared__ double sh[kProbeThreads];
    constexpr int ev = kBf16 ? 8 : 4;
    const int64_t nvec = n / ev;
    const int rem = static_cast<int>(n - nvec * ev);
    constexpr int64_t kTileGroups = static_cast<int64_t>(kStaticDriftTileGroups) * kProbeThreads;
    static_assert(kStaticDriftTileGroups % kGroupsInFlight == 0, "whole rounds per tile");
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        Kahan sd, sp;
        for (int r = 0; r < kStaticDriftTileGroups; r += kGroupsInFlight) {
            uint4 rc[kGroupsInFlight], rp[kGroupsInFlight];
            const int64_t g0 = tile * kTileGroups + static_cast<int64_t>(r) * kProbeThreads +
                               threadIdx.x;
#pragma unroll
            for (int u = 0; u < kGroupsInFlight; ++u) {
                const int64_t g = g0 + static_cast<int64_t>(u) * kProbeThreads;
                if (g < nvec) {
                    rc[u] = ld_nc16(cur + g * 16);
                    rp[u] = ld_nc16(prev + g * 16);
                }
            }
#pragma unroll
            for (int u = 0; u < kGroupsInFlight; ++u) {
                const int64_t g = g0 + static_cast<int64_t>(u) * kProbeThreads;
                if (g < nvec) {
                    float gd, gp;
                    group_sums<kBf16>(rc[u], rp[u], gd, gp);
                    sd.add(gd);
                    sp.add(gp);
                } else if (g == nvec && rem > 0) {  // the ragged last group, element by element
                    float gd = 0.0f, gp = 0.0f;
                    for (int e = 0; e < rem; ++e) {
                        const float c = load1<kBf16>(cur, nvec * ev + e);
                        const float p = load1<kBf16>(prev, nvec * ev + e);
                        gd += fabsf(c - p);
                        gp += fabsf(p);
                    }
                    sd.add(gd);
                    sp.add(gp);
                }
            }
        }
        double bd = 0.0, bp = 0.0;
        block_sum_kahan(sd, sp, sh, bd, bp);
        if (threadIdx.x == 0) {
            partials[2 * tile] = bd;
            partials[2 * tile + 1] = bp;
        }
    }
}

std::mutex g_static_mu;
constexpr int kMaxDevices = 64;

// The looked-up address of g_drift_scratch per device, with the id of the context it was
// looked up in: a context created later on the same device (after cudaDeviceReset, say)
// loads the library's module afresh, at a possibly different address.
struct StaticScratch {
    double *ptr = nullptr;
    unsigned long long ctx = 0;
};
StaticScratch g_static_scratch[kMaxDevices];

// Unique id of the calling thread's current context (the driver's cuCtxGetId, reached through
// the runtime's entry-point query so that the library does not link the driver API), or 0
// when no context is current or the query is unavailable.  Called with g_static_mu held.
unsigned long long current_context_id() {
    using GetCurrent = CUresult (*)(CUcontext *);
    using GetId = CUresult (*)(CUcontext, unsigned long long *);
    static bool tried = false;
    static GetCurrent get_current = nullptr;
    static GetId get_id = nullptr;
    if (!tried) {
        tried = true;
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrent>(f);
        f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<GetId>(f);
        cudaGetLastError();
    }
    if (!get_current || !get_id) return 0;
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
    if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of g_drift_scratch on the current device.  In host code the array's name
// only stands in for the symbol, so the address is looked up with cudaGetSymbolAddress, with
// that device current: on the first no-allocation call on a device, and again whenever the
// device's current context is not the one the address was looked up in (or cannot be told).
int static_scratch(double **out) {
    int dev = 0;
    int err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_static_mu);
    StaticScratch &sc = g_static_scratch[dev];
    const unsigned long long ctx = current_context_id();
    if (sc.ptr && ctx != 0 && sc.ctx == ctx) {
        *out = sc.ptr;
        return cudaSuccess;
    }
    void *p = nullptr;
    err = cudaGetSymbolAddress(&p, g_drift_scratch);
    if (err != cudaSuccess) {
        cudaGetLastError();  // reported once, by return value
        return err;
    }
    sc.ptr = static_cast<double *>(p);
    sc.ctx = current_context_id();  // the lookup made the device's context current
    *out = sc.ptr;
    return cudaSuccess;
}

}  // namespace

int64_t static_drift_max_elems(bc_dtype dtype) {
    const int64_t ev = dtype == BC_DTYPE_BF16 ? 8 : 4;
    return kStaticDriftMaxTiles * kStaticDriftTileGroups * kProbeThreads * ev;
}

int launch_drift_static(const void *cur, const void *prev, int64_t n, bc_dtype dtype,
                        double *out, void *stream, int64_t *launches) {
    double *scratch = nullptr;
    int err = static_scratch(&scratch);
    if (err != cudaSuccess) return err;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t ev = dtype == BC_DTYPE_BF16 ? 8 : 4;
    const int64_t groups = (n + ev - 1) / ev;
    constexpr int64_t kTileGroups = static_cast<int64_t>(kStaticDriftTileGroups) * kProbeThreads;
    int64_t ntiles = (groups + kTileGroups - 1) / kTileGroups;
    if (ntiles < 1) ntiles = 1;
    if (ntiles > kStaticDriftMaxTiles) return cudaErrorInvalidValue;  // the caller checks first
    int64_t grid = probe_ctas();
    if (grid > ntiles) grid = ntiles;
    if (dtype == BC_DTYPE_BF16)
        drift_tile_partials<true><<<static_cast<int>(grid), kProbeThreads, 0, s>>>(
            static_cast<const char *>(cur), static_cast<const char *>(prev), n, ntiles, scratch);
    else
        drift_tile_partials<false><<<static_cast<int>(grid), kProbeThreads, 0, s>>>(
            static_cast<const char *>(cur), static_cast<const char *>(prev), n, ntiles, scratch);
    ++*launches;
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    drift_final<<<1, kProbeThreads, 0, s>>>(scratch, static_cast<int>(ntiles), out);
    ++*launches;
    return cudaGetLastError();
}

}  // namespace bc
