// bc_probe.cu -- relative L1 drift of a feature probe between two consecutive steps, the
// signal of the adaptive schedule (Sec. 4.5: a full step is triggered once the
// accumulated relative change of a feature probe exceeds a threshold).
//
//     drift = sum_e |cur[e] - prev[e]| / sum_e |prev[e]|
//
// Two launches with a fixed reduction order, so the result is bitwise reproducible for a
// given device: (1) a persistent grid streams both tensors once in 16-byte groups, each
// thread sums a group in fp32 and accumulates the group sums in fp64 (fp64 per element
// would outrun GB300's fp64 rate), and every CTA writes its two partial sums to scratch;
// (2) one CTA adds the partials in index order and writes {sum |d|, sum |prev|, ratio}.
// HBM-bound: 2 * n * sizeof(T) bytes.  No atomics, no waits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

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

__device__ __forceinline__ void unpack(uint4 r, float *f, bool bf16) {
    if (bf16) {
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

__device__ __forceinline__ float load1(const char *p, int64_t e, bool bf16) {
    if (bf16) return __uint_as_float(static_cast<uint32_t>(reinterpret_cast<const uint16_t *>(p)[e]) << 16);
    return reinterpret_cast<const float *>(p)[e];
}

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

__global__ void __launch_bounds__(kProbeThreads)
    drift_partials(const char *cur, const char *prev, int64_t n, int bf16, double *partials) {
    __shared__ double sh[kProbeThreads];
    const int ev = bf16 ? 8 : 4;
    const int64_t nvec = n / ev;
    double sd = 0.0, sp = 0.0;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * kProbeThreads;
    for (int64_t v = static_cast<int64_t>(blockIdx.x) * kProbeThreads + threadIdx.x; v < nvec;
         v += stride) {
        float c[8], p[8];
        unpack(ld_nc16(cur + v * 16), c, bf16);
        unpack(ld_nc16(prev + v * 16), p, bf16);
        float gd = 0.0f, gp = 0.0f;
        for (int e = 0; e < ev; ++e) {
            gd += fabsf(c[e] - p[e]);
            gp += fabsf(p[e]);
        }
        sd += gd;
        sp += gp;
    }
    if (blockIdx.x == 0) {  // ragged tail: fewer than one 16-byte group
        const int64_t e = nvec * ev + threadIdx.x;
        if (e < n) {
            const float c = load1(cur, e, bf16), p = load1(prev, e, bf16);
            sd += fabsf(c - p);
            sp += fabsf(p);
        }
    }
    sd = block_sum(sd, sh);
    sp = block_sum(sp, sh);
    if (threadIdx.x == 0) {
        partials[2 * blockIdx.x] = sd;
        partials[2 * blockIdx.x + 1] = sp;
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
    drift_partials<<<grid, kProbeThreads, 0, s>>>(static_cast<const char *>(cur),
                                                  static_cast<const char *>(prev), n,
                                                  dtype == BC_DTYPE_BF16 ? 1 : 0, partials);
    ++*launches;
    int err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    drift_final<<<1, kProbeThreads, 0, s>>>(partials, grid, out);
    ++*launches;
    return cudaGetLastError();
}

}  // namespace bc
