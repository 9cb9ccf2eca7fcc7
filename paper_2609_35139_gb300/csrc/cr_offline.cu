// Offline preparation kernels (bandwidth-bound):
//   canon_kernel    chunk-cache canonicalisation, K^c_t = R_M(q_t)^{-1} K_t with
//                   V as stored (Sec. 4.1, "Chunk-cache preparation")
//   sigma_*_kernel  per-coordinate RMS statistics over corpus caches: sigma_stale
//                   from stale caches, sigma_Delta from joint - stale residual
//                   targets (Sec. 4.2, "Normalization and objective")
#include <cuda_bf16.h>

#include "cr_internal.h"
#include "cr_ptx.cuh"

namespace cr {
namespace {

struct Freq {
    float f[64];
};

__device__ __forceinline__ void load8(const uint16_t* p, float* v) {
    const uint4 w = *reinterpret_cast<const uint4*>(p);
    const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        v[2 * i] = __uint_as_float(u[i] << 16);
        v[2 * i + 1] = __uint_as_float(u[i] & 0xFFFF0000u);
    }
}
__device__ __forceinline__ void load8(const float* p, float* v) {
    const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void store8(uint16_t* p, const float* v) {
    *reinterpret_cast<uint4*>(p) = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                              pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
}
__device__ __forceinline__ void store8(float* p, const float* v) {
    reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

// One thread per (token, group of 8 rotation pairs, quarter of the layers): the
// 8 angles q_t * f_d are computed once and applied to that group in the K
// segments of the thread's layers (rotate-half pairs (d, d + d_h/2) inside
// each d_h-wide segment, by -q_t f_d: (a, b) -> (a cos + b sin, b cos - a sin)),
// one rounding to the cache dtype.  With dir = -1 the sine changes sign and the
// rotation is by +q_t f_d, R_M itself (the stale cache's re-rotation of K to
// request positions, Sec. 2.2).  Two segments are loaded before either is
// rotated, for memory-level parallelism.
template <typename T>
__global__ void __launch_bounds__(256) canon_kernel(T* kv, int64_t n, const int32_t* __restrict__ pos,
                                                    int L, int H, int dh,
                                                    const __grid_constant__ Freq f, float dir) {
    pdl_launch_dependents();
    pdl_wait();
    const int groups = dh / 16;
    constexpr int kParts = 4;   // layer ranges per (token, group)
    const int64_t D = static_cast<int64_t>(2) * L * H * dh;
    const int64_t work = n * groups * kParts;
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < work;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int part = static_cast<int>(idx % kParts);
        const int64_t tg = idx / kParts;
        const int64_t t = tg / groups;
        const int g = static_cast<int>(tg - t * groups);
        const float q = static_cast<float>(__ldg(pos + t));
        float c[8], s[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            sincos_prod(q, f.f[g * 8 + i], &s[i], &c[i]);
            s[i] *= dir;
        }
        T* row = kv + t * D;
        // the K segments (layer l, head h) of this part, l in [l0, l1)
        const int l0 = part * L / kParts, l1 = (part + 1) * L / kParts;
        const int nseg = (l1 - l0) * H;
        for (int k = 0; k < nseg; k += 2) {
            const int k2 = (k + 1 < nseg) ? k + 1 : k;
            T* seg0 = row + (static_cast<int64_t>(2 * (l0 + k / H)) * H + k % H) * dh;
            T* seg1 = row + (static_cast<int64_t>(2 * (l0 + k2 / H)) * H + k2 % H) * dh;
            float a0[8], b0[8], a1[8], b1[8];
            load8(seg0 + g * 8, a0);
            load8(seg0 + dh / 2 + g * 8, b0);
            load8(seg1 + g * 8, a1);
            load8(seg1 + dh / 2 + g * 8, b1);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float x0 = a0[i], y0 = b0[i], x1 = a1[i], y1 = b1[i];
                a0[i] = x0 * c[i] + y0 * s[i];
                b0[i] = y0 * c[i] - x0 * s[i];
                a1[i] = x1 * c[i] + y1 * s[i];
                b1[i] = y1 * c[i] - x1 * s[i];
            }
            store8(seg0 + g * 8, a0);
            store8(seg0 + dh / 2 + g * 8, b0);
            if (k2 != k) {
                store8(seg1 + g * 8, a1);
                store8(seg1 + dh / 2 + g * 8, b1);
            }
        }
    }
}

// Partial sums of squares: block (x, y) covers 2048 coordinates (8 per thread)
// over the 64-token slice y; part[y][j].  With b, the squares of a - b.
template <typename T>
__global__ void __launch_bounds__(256) sigma_partial_kernel(const T* __restrict__ a, const T* __restrict__ b,
                                                            int64_t n, int64_t D, float* __restrict__ part) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t col = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) * 8;
    if (col >= D) return;
    const int64_t t0 = static_cast<int64_t>(blockIdx.y) * kSigmaSlice;
    const int64_t t1 = t0 + kSigmaSlice < n ? t0 + kSigmaSlice : n;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    int64_t t = t0;
    // four rows in flight, added in row order (the sum's order is fixed)
    for (; t + 4 <= t1; t += 4) {
        float x[4][8];
#pragma unroll
        for (int u = 0; u < 4; ++u) load8(a + (t + u) * D + col, x[u]);
        if (b) {
            float y[4][8];
#pragma unroll
            for (int u = 0; u < 4; ++u) load8(b + (t + u) * D + col, y[u]);
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int i = 0; i < 8; ++i) x[u][i] -= y[u][i];
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = fmaf(x[u][i], x[u][i], acc[i]);
    }
    for (; t < t1; ++t) {
        float x[8];
        load8(a + t * D + col, x);
        if (b) {
            float y[8];
            load8(b + t * D + col, y);
#pragma unroll
            for (int i = 0; i < 8; ++i) x[i] -= y[i];
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = fmaf(x[i], x[i], acc[i]);
    }
    store8(part + static_cast<int64_t>(blockIdx.y) * D + col, acc);
}

// sumsq[j] += sum over slices, in slice order (deterministic), in fp64.
__global__ void __launch_bounds__(256) sigma_reduce_kernel(const float* __restrict__ part, int slices,
                                                           int64_t D, double* sumsq) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t j = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; j < D;
         j += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        double s = 0.0;
        for (int k = 0; k < slices; ++k) s += static_cast<double>(part[static_cast<int64_t>(k) * D + j]);
        sumsq[j] += s;
    }
}

__global__ void __launch_bounds__(256) sigma_finalize_kernel(const double* __restrict__ sumsq, int64_t D,
                                                             double inv_count, float* __restrict__ sigma) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t j = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; j < D;
         j += static_cast<int64_t>(gridDim.x) * blockDim.x)
        sigma[j] = static_cast<float>(sqrt(sumsq[j] * inv_count));
}

}  // namespace

cr_status launch_canonicalize(void* kv, bool f32, int64_t n, const int32_t* pos, int L, int H, int dh,
                              const float* inv_freq_host, cudaStream_t st, float dir) {
    if (n <= 0) return CR_OK;
    if (dh != 64 && dh != 128) return CR_ERR_UNSUPPORTED;
    Freq f{};
    for (int i = 0; i < dh / 2; ++i) f.f[i] = inv_freq_host[i];
    const int64_t work = n * (dh / 16) * 4;
    int64_t blocks = (work + 255) / 256;
    if (blocks > static_cast<int64_t>(num_sms()) * 16) blocks = static_cast<int64_t>(num_sms()) * 16;
    const dim3 grid(static_cast<unsigned>(blocks)), block(256);
    if (f32)
        return launch_pdl(canon_kernel<float>, grid, block, 0, st, static_cast<float*>(kv), n, pos, L, H,
                          dh, f, dir);
    return launch_pdl(canon_kernel<uint16_t>, grid, block, 0, st, static_cast<uint16_t*>(kv), n, pos, L,
                      H, dh, f, dir);
}

cr_status launch_sigma_accumulate(const void* a, const void* b, bool f32, int64_t n, int64_t D,
                                  float* part, double* sumsq, cudaStream_t st) {
    if (n <= 0) return CR_OK;
    const int64_t slices = (n + kSigmaSlice - 1) / kSigmaSlice;
    const dim3 grid(static_cast<unsigned>((D / 8 + 255) / 256), static_cast<unsigned>(slices));
    cr_status s;
    if (f32)
        s = launch_pdl(sigma_partial_kernel<float>, grid, dim3(256), 0, st, static_cast<const float*>(a),
                       static_cast<const float*>(b), n, D, part);
    else
        s = launch_pdl(sigma_partial_kernel<uint16_t>, grid, dim3(256), 0, st,
                       static_cast<const uint16_t*>(a), static_cast<const uint16_t*>(b), n, D, part);
    if (s != CR_OK) return s;
    int64_t blocks = (D + 255) / 256;
    if (blocks > static_cast<int64_t>(num_sms()) * 8) blocks = static_cast<int64_t>(num_sms()) * 8;
    return launch_pdl(sigma_reduce_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st,
                      static_cast<const float*>(part), static_cast<int>(slices), D, sumsq);
}

cr_status launch_sigma_finalize(const double* sumsq, int64_t D, int64_t count, float* sigma,
                                cudaStream_t st) {
    int64_t blocks = (D + 255) / 256;
    if (blocks > static_cast<int64_t>(num_sms()) * 8) blocks = static_cast<int64_t>(num_sms()) * 8;
    return launch_pdl(sigma_finalize_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, sumsq,
                      D, 1.0 / static_cast<double>(count), sigma);
}

}  // namespace cr
