// bc_probe.cu -- relative L1 drift of a feature probe between two consecutive steps, the
// signal of the adaptive schedule (Sec. 4.5: a full step is triggered once the
// accumulated relative change of a feature probe exceeds a threshold).
//
//     drift = sum_e |cur[e] - prev[e]| / sum_e |prev[e]|
//
// Two launches with a fixed reduction order, so the result is bitwise reproducible for a
// given device: (1) a persistent grid streams both tensors once in 16-byte groups (four
// groups of loads in flight per thread), each thread sums a group in fp32 and accumulates
// the group sums with compensated (Kahan) fp32 addition, so the error stays near two fp32
// ulps however long the stream is, without touching GB300's slow fp64 pipe per element;
// every CTA adds its threads' sums in fp64 and writes its two partial sums to scratch;
// (2) one CTA adds the partials in index order and writes {sum |d|, sum |prev|, ratio}.
// HBM-bound: 2 * n * sizeof(T) bytes.  No atomics, no waits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "bc_internal.h"

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
    __device__ __forceinline__ double value() const {
        return static_cast<double>(s) - static_cast<double>(c);
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

// Fixed-order tree sum of one double per thread over the CTA (kProbeThreads threads).
__device__ __forceinline__ double block_sum(double v, double *sh) {
    sh[threadIdx.x] = v;
    __syncthreads();
    for (int s = kProbeThreads / 2; s > 0; s >>= 1) {
        if (static_cast<int>(threadIdx.x) < s) sh[threadIdx.x] += sh[threadIdx.x + s];
        __syncthreads();
    }
    const double r = sh[0];
    __syncthreads();
    return r;
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
    const double bd = block_sum(sd.value(), sh);
    const double bp = block_sum(sp.value(), sh);
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
    sd = block_sum(sd, sh);
    sp = block_sum(sp, sh);
    if (threadIdx.x == 0) {
        out[0] = sd;
        out[1] = sp;
        out[2] = sp > 0.0 ? sd / sp : (sd > 0.0 ? __longlong_as_double(0x7ff0000000000000LL) : 0.0);
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

int launch_drift(const void *cur, const void *prev, int64_t n, bc_dtype dtype, double *partials,
                 int max_parts, double *out, void *stream, int64_t *launches) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int ev = dtype == BC_DTYPE_BF16 ? 8 : 4;
    const int64_t nvec = n / ev;
    int64_t want = (nvec + kProbeThreads - 1) / kProbeThreads;
    if (want < 1) want = 1;
    int grid = probe_ctas();
    if (grid > max_parts) grid = max_parts;
    if (want < grid) grid = static_cast<int>(want);
    if (dtype == BC_DTYPE_BF16)
        drift_partials<true><<<grid, kProbeThreads, 0, s>>>(
            static_cast<const char *>(cur), static_cast<const char *>(prev), n, partials);
    else
        drift_partials<false><<<grid, kProbeThreads, 0, s>>>(
            static_cast<const char *>(cur), static_cast<const char *>(prev), n, partials);
    ++*launches;
    int err = cudaGetLastError();
    if (err != cudaSuccess) return err;
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
        const double bd = block_sum(sd.value(), sh);
        const double bp = block_sum(sp.value(), sh);
        if (threadIdx.x == 0) {
            partials[2 * tile] = bd;
            partials[2 * tile + 1] = bp;
        }
    }
}

std::mutex g_static_mu;
constexpr int kMaxDevices = 64;
double *g_static_scratch[kMaxDevices] = {};

// Device address of g_drift_scratch on the current device.  In host code the array's name
// only stands in for the symbol, so the address is looked up with cudaGetSymbolAddress,
// once per device, with that device current (the first no-allocation call on it).
int static_scratch(double **out) {
    int dev = 0;
    int err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_static_mu);
    if (!g_static_scratch[dev]) {
        void *p = nullptr;
        err = cudaGetSymbolAddress(&p, g_drift_scratch);
        if (err != cudaSuccess) return err;
        g_static_scratch[dev] = static_cast<double *>(p);
    }
    *out = g_static_scratch[dev];
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
