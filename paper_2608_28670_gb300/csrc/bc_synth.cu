// bc_synth.cu -- seeded synthetic feature trajectories for tests and benchmarks.
//
// Built into its own library (libbc_synth.so) and holding none of the forecast's
// arithmetic: it only writes input tensors.  Every element e of tensor `tensor_id` follows
// a random polynomial trajectory in the (normalised) timestep tau,
//     F(e, tau) = amp(e) * sum_{d=0..degree} a_d(e) tau^d + noise_std * z(e, step_id),
// with a_d, z ~ N(0, 1).  amp(e) is outlier_scale for a seeded fraction `outlier_frac` of
// channels (channel = e mod hidden) and 1 otherwise.
//
// Random numbers: Philox4x32-10, the counter-based generator of Salmon, Moraes, Dror and
// Shaw, "Parallel random numbers: as easy as 1, 2, 3" (SC 2011), keyed by the 64-bit seed,
// with the element index and tensor/step ids as the counter; normals by the Box-Muller
// transform.  The output depends only on (seed, tensor_id, step_id, e), never on the launch
// shape, so any sub-range can be regenerated.
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include <cstdint>
#include <cstring>

namespace {

struct U4 {
    uint32_t x, y, z, w;
};

__device__ __forceinline__ U4 philox4x32_10(U4 c, uint32_t k0, uint32_t k1) {
    const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;  // round multipliers
    const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;  // Weyl key increments
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(M0, c.x), lo0 = M0 * c.x;
        const uint32_t hi1 = __umulhi(M1, c.z), lo1 = M1 * c.z;
        c = U4{hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0};
        k0 += W0;
        k1 += W1;
    }
    return c;
}

// Uniform in (0, 1): 24 random bits centred in their bin, never 0 or 1.
__device__ __forceinline__ float unit(uint32_t u) {
    return (static_cast<float>(u >> 8) + 0.5f) * (1.0f / 16777216.0f);
}

__device__ __forceinline__ void box_muller(uint32_t a, uint32_t b, float &z0, float &z1) {
    const float r = sqrtf(-2.0f * logf(unit(a)));
    float s, c;
    sincospif(2.0f * unit(b), &s, &c);
    z0 = r * c;
    z1 = r * s;
}

struct Recipe {
    uint32_t k0, k1;
    uint32_t tensor_id, step_id;
    float tau;
    int degree;
    float noise_std;
    int64_t hidden;
    float outlier_frac, outlier_scale;
};

__device__ __forceinline__ float trajectory(const Recipe &r, int64_t e) {
    const uint32_t elo = static_cast<uint32_t>(e), ehi = static_cast<uint32_t>(e >> 32);
    const U4 coef = philox4x32_10(U4{elo, ehi, r.tensor_id, 0u}, r.k0, r.k1);
    float a[4];
    box_muller(coef.x, coef.y, a[0], a[1]);
    box_muller(coef.z, coef.w, a[2], a[3]);
    float v = 0.0f;
    for (int d = r.degree; d >= 0; --d) v = v * r.tau + a[d];  // Horner
    if (r.outlier_frac > 0.0f) {
        const int64_t ch = e % r.hidden;
        const U4 h = philox4x32_10(U4{static_cast<uint32_t>(ch), 0u, 0xFFFFFFFFu, 0u}, r.k0, r.k1);
        if (unit(h.x) < r.outlier_frac) v *= r.outlier_scale;
    }
    if (r.noise_std != 0.0f) {
        const U4 nz = philox4x32_10(U4{elo, ehi, r.tensor_id, 1u + r.step_id}, r.k0, r.k1);
        float z0, z1;
        box_muller(nz.x, nz.y, z0, z1);
        v += r.noise_std * z0;
    }
    return v;
}

__global__ void fill_f32(float *dst, int64_t n, Recipe r) {
    for (int64_t e = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; e < n;
         e += int64_t(gridDim.x) * blockDim.x)
        dst[e] = trajectory(r, e);
}

__global__ void fill_bf16(__nv_bfloat16 *dst, int64_t n, Recipe r) {
    for (int64_t e = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; e < n;
         e += int64_t(gridDim.x) * blockDim.x)
        dst[e] = __float2bfloat16_rn(trajectory(r, e));
}

}  // namespace

extern "C" {

// Fill `n` elements at device address `dst` (dtype 0 = f32, 1 = bf16) on `stream`.
// Returns a cudaError_t value (0 = success); sizes and pointers are checked.
int bcs_fill(void *dst, int dtype, int64_t n, uint64_t seed, uint32_t tensor_id,
             uint32_t step_id, double tau, int degree, double noise_std, int64_t hidden,
             double outlier_frac, double outlier_scale, void *stream) {
    if (n < 0 || (n > 0 && !dst) || degree < 0 || degree > 3 || hidden < 1 ||
        (dtype != 0 && dtype != 1))
        return static_cast<int>(cudaErrorInvalidValue);
    if (n == 0) return 0;
    Recipe r{};
    r.k0 = static_cast<uint32_t>(seed);
    r.k1 = static_cast<uint32_t>(seed >> 32);
    r.tensor_id = tensor_id;
    r.step_id = step_id;
    r.tau = static_cast<float>(tau);
    r.degree = degree;
    r.noise_std = static_cast<float>(noise_std);
    r.hidden = hidden;
    r.outlier_frac = static_cast<float>(outlier_frac);
    r.outlier_scale = static_cast<float>(outlier_scale);
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (n + 255) / 256;
    const int64_t cap = static_cast<int64_t>(sms > 0 ? sms : 1) * 16;
    const int grid = static_cast<int>(want < cap ? want : cap);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (dtype == 0)
        fill_f32<<<grid, 256, 0, s>>>(static_cast<float *>(dst), n, r);
    else
        fill_bf16<<<grid, 256, 0, s>>>(static_cast<__nv_bfloat16 *>(dst), n, r);
    return static_cast<int>(cudaGetLastError());
}

}  // extern "C"
