// Training-step kernels (Sec. 4.2, App. A): the bandwidth-bound pieces of the
// backward pass and of the optimizer (the backward's matrix products run in
// the tcgen05 GEMM, launch_gemm_lay).
//   row_scale_kernel     c_request of every row, for the loss head's epilogue
//   rowsq_kernel         per row: the loss head's partial sums of r^2 in order
//   loss_reduce_kernel   per request, rows summed in order (fp64): the loss
//   colsum_kernel        column sums in a fixed order (bias, LayerNorm grads)
//   ln_backward_kernel   LayerNorm backward per row, plus dy * x_hat per element
//   gelu_backward_kernel dpre = dg * (Phi(pre) + pre phi(pre))
//   rope_backward_kernel the repairer RoPE's transpose on dQ, dK
//   sqnorm_*             squared L2 norm of the gradient (fp64, fixed order)
//   adamw_kernel         clipping coefficient, AdamW, bf16 mirror of the weights
//   seg_grad_kernel      the segment weights' gradient out of the grouped GEMM's blocks
#include <cuda_bf16.h>

#include "cr_internal.h"
#include "cr_ptx.cuh"

namespace cr {
namespace {

__device__ __forceinline__ uint16_t f32_to_bf16(float x) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

// the request of row t: req_start[r] <= t < req_start[r + 1]
__device__ __forceinline__ int request_of(const LossParams& p, int64_t t) {
    int r0 = 0, r1 = p.n_req - 1;
    while (r0 < r1) {
        const int mid = (r0 + r1 + 1) >> 1;
        if (p.req_start[mid] <= t) r0 = mid;
        else r1 = mid - 1;
    }
    return r0;
}


// The loss weight c of each row's request: dL/dr = c r.
__global__ void row_scale_kernel(const __grid_constant__ LossParams p, int64_t n, float* __restrict__ out) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x)
        out[t] = p.scale[request_of(p, t)];
}

// Per row, the loss head's nparts partial sums of r^2 (part[j][row], one per
// column tile and epilogue column group) added in a fixed order: block of 8
// warps over 32 rows (a lane per row), warp w adds parts [w P/8, (w+1) P/8) in
// order, eight loads in flight, then the warps' sums in warp order.
__global__ void __launch_bounds__(256)
    rowsq_kernel(const float* __restrict__ part, int64_t rows, int nparts, float* __restrict__ rowsq) {
    pdl_launch_dependents();
    pdl_wait();
    const int lane = static_cast<int>(threadIdx.x & 31), w = static_cast<int>(threadIdx.x >> 5);
    const int64_t t = static_cast<int64_t>(blockIdx.x) * 32 + lane;
    const int per = (nparts + 7) / 8;
    const int j0 = w * per, j1 = min(nparts, j0 + per);
    float s = 0.0f;
    if (t < rows) {
#pragma unroll 8
        for (int j = j0; j < j1; ++j) s += part[static_cast<int64_t>(j) * rows + t];
    }
    __shared__ float red[8][32];
    red[w][lane] = s;
    __syncthreads();
    if (w == 0 && t < rows) {
        float a = 0.0f;
#pragma unroll
        for (int k = 0; k < 8; ++k) a += red[k][lane];
        rowsq[t] = a;
    }
}


// One block per request: each thread sums a fixed stride of the request's rows
// (fp64), then a fixed tree; the result divided by N_r D n_req (the mean over
// requests).  loss_total_kernel adds the requests in order.
__global__ void __launch_bounds__(256)
    loss_reduce_kernel(const float* __restrict__ rowsq, const __grid_constant__ LossParams p, int64_t D,
                       double* __restrict__ per_req) {
    pdl_launch_dependents();
    pdl_wait();
    const int r = blockIdx.x;
    double s = 0.0;
    for (int64_t t = p.req_start[r] + threadIdx.x; t < p.req_start[r + 1]; t += blockDim.x)
        s += static_cast<double>(rowsq[t]);
    __shared__ double red[256];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int k = 128; k > 0; k >>= 1) {
        if (static_cast<int>(threadIdx.x) < k) red[threadIdx.x] += red[threadIdx.x + k];
        __syncthreads();
    }
    if (threadIdx.x == 0)
        per_req[r] = red[0] / (static_cast<double>(p.req_start[r + 1] - p.req_start[r]) * D * p.n_req);
}

__global__ void loss_total_kernel(const double* __restrict__ per_req, int n_req, float* __restrict__ loss_out) {
    pdl_launch_dependents();
    pdl_wait();
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    double l = 0.0;
    for (int r = 0; r < n_req; ++r) l += per_req[r];
    loss_out[0] = static_cast<float>(l);
}

// Column sums in a fixed order, one launch: block (x, y) sums rows
// [kColSlice y, kColSlice (y + 1)) of the 64 columns [64 x, 64 x + 64), two
// adjacent columns per lane: warp w of 8 adds rows w, w + 8, ... in row order
// (eight loads in flight), the warps' sums are added in warp order into
// partial[y][c], and the last block of column block x to finish (elected by a
// counter, after a fence) adds the slices in order and resets the counter.
// The order of the additions never depends on timing.  kOut16: an fp32 input
// is also written rounded to bf16 (round to nearest even) into a16 [rows,
// cols], the operand of the backward's GEMMs, from the same read.  cols and
// lda are even.
constexpr int kColSlice = 256;
__device__ __forceinline__ float2 ld2(const float* p, int64_t i) {
    return *reinterpret_cast<const float2*>(p + i);
}
__device__ __forceinline__ float2 ld2(const uint16_t* p, int64_t i) {
    const uint32_t v = *reinterpret_cast<const uint32_t*>(p + i);
    return make_float2(__uint_as_float(v << 16), __uint_as_float(v & 0xFFFF0000u));
}
template <typename T, bool kOut16>
__global__ void __launch_bounds__(256)
    colsum_kernel(const T* __restrict__ a, int64_t rows, int64_t cols, int64_t lda,
                  uint16_t* __restrict__ a16, float* part, float* __restrict__ out, int accumulate,
                  unsigned* __restrict__ counters) {
    pdl_launch_dependents();
    pdl_wait();
    const int lane = static_cast<int>(threadIdx.x & 31), w = static_cast<int>(threadIdx.x >> 5);
    const int64_t c = static_cast<int64_t>(blockIdx.x) * 64 + 2 * lane;
    const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kColSlice;
    const int64_t r1 = min(rows, r0 + kColSlice);
    float s0 = 0.0f, s1 = 0.0f;
    if (c < cols) {
#pragma unroll 8
        for (int64_t r = r0 + w; r < r1; r += 8) {
            const float2 v = ld2(a, r * lda + c);
            s0 += v.x;
            s1 += v.y;
            if constexpr (kOut16) *reinterpret_cast<uint32_t*>(a16 + r * cols + c) = pack_bf16x2(v.x, v.y);
        }
    }
    __shared__ float2 red[8][32];
    red[w][lane] = make_float2(s0, s1);
    __syncthreads();
    if (w == 0 && c < cols) {
        float t0 = 0.0f, t1 = 0.0f;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            t0 += red[k][lane].x;
            t1 += red[k][lane].y;
        }
        *reinterpret_cast<float2*>(part + static_cast<int64_t>(blockIdx.y) * cols + c) = make_float2(t0, t1);
    }
    __threadfence();
    __syncthreads();
    __shared__ bool last;
    if (threadIdx.x == 0) last = atomicAdd(&counters[blockIdx.x], 1u) == gridDim.y - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    if (w == 0 && c < cols) {
        float t0 = 0.0f, t1 = 0.0f;
        for (int64_t y = 0; y < gridDim.y; ++y) {
            const float2 v = __ldcg(reinterpret_cast<const float2*>(part + y * cols + c));
            t0 += v.x;
            t1 += v.y;
        }
        out[c] = accumulate ? out[c] + t0 : t0;
        out[c + 1] = accumulate ? out[c + 1] + t1 : t1;
    }
    if (threadIdx.x == 0) counters[blockIdx.x] = 0u;
}

// LayerNorm backward, one warp per row of D (a multiple of 32, at most 1024)
// values: with x_hat = (x - mean) rstd and g = dy gamma,
//   dx = rstd (g - mean(g) - x_hat mean(g x_hat))  (+ add, if given)
// and gprod = dy x_hat per element (its column sums are dgamma).
__global__ void __launch_bounds__(256)
    ln_backward_kernel(const float* __restrict__ x, const float* __restrict__ gamma,
                       const float* __restrict__ dy, const float* __restrict__ add, float eps, int64_t N,
                       int D, float* __restrict__ dx, float* __restrict__ gprod) {
    pdl_launch_dependents();
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t row = blockIdx.x * static_cast<int64_t>(blockDim.x / 32) + (threadIdx.x >> 5);
    if (row >= N) return;
    const float* xr = x + row * D;
    const float* dr = dy + row * D;
    const int per = D / 32;   // <= 32
    float xv[32], gv[32];
    float s = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
        if (i < per) {
            xv[i] = xr[i * 32 + lane];
            s += xv[i];
        }
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mean = s / D;
    float v = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
        if (i < per) {
            const float d = xv[i] - mean;
            v = fmaf(d, d, v);
        }
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const float rstd = rsqrtf(v / D + eps);
    float sg = 0.0f, sgx = 0.0f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
        if (i < per) {
            const int c = i * 32 + lane;
            const float dyv = dr[c];
            xv[i] = (xv[i] - mean) * rstd;
            gv[i] = dyv * __ldg(gamma + c);
            sg += gv[i];
            sgx = fmaf(gv[i], xv[i], sgx);
            gprod[row * D + c] = dyv * xv[i];
        }
    for (int o = 16; o > 0; o >>= 1) {
        sg += __shfl_xor_sync(0xffffffffu, sg, o);
        sgx += __shfl_xor_sync(0xffffffffu, sgx, o);
    }
    const float mg = sg / D, mgx = sgx / D;
#pragma unroll
    for (int i = 0; i < 32; ++i)
        if (i < per) {
            const int64_t k = row * D + i * 32 + lane;
            float d = rstd * (gv[i] - mg - xv[i] * mgx);
            if (add) d += add[k];
            dx[k] = d;
        }
}

// dpre = dg * GELU'(pre), GELU'(x) = Phi(x) + x phi(x), in place on dg.
__global__ void __launch_bounds__(256)
    gelu_backward_kernel(float* __restrict__ dg, const float* __restrict__ pre, int64_t n) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const float x = pre[i];
        const float Phi = 0.5f * erfcf(-x * 0.70710678118654752f);
        const float phi = 0.39894228040143268f * expf(-0.5f * x * x);
        dg[i] *= fmaf(x, phi, Phi);
    }
}

// The repairer RoPE rotated q and k of every head by angle p_t f_i (pairs
// (i, i + d/2)); its transpose rotates the gradients back:
//   (a, b) -> (a cos + b sin, b cos - a sin).  dqkv [N, 3 d_b] fp32, Q and K
// columns [0, 2 d_b); table [d/2, N] (cos, sin) of the forward, angle-major.
__global__ void __launch_bounds__(256)
    rope_backward_kernel(float* __restrict__ dqkv, const float2* __restrict__ table, int64_t N, int db,
                         int hd) {
    pdl_launch_dependents();
    pdl_wait();
    const int half = hd / 2;
    const int64_t pairs_per_row = static_cast<int64_t>(2 * db / hd) * half;   // Q and K heads
    const int64_t total = N * pairs_per_row;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t t = i / pairs_per_row;
        const int64_t rem = i - t * pairs_per_row;
        const int64_t h = rem / half;
        const int j = static_cast<int>(rem - h * half);
        const float2 cs = table[static_cast<int64_t>(j) * N + t];
        float* base = dqkv + t * 3 * db + h * hd;
        const float a = base[j], b = base[j + half];
        base[j] = a * cs.x + b * cs.y;
        base[j + half] = b * cs.x - a * cs.y;
    }
}

// out[i] = in[i] * scale[i % cols] (dW_seg: the cache's 1 / sigma_stale per column)
__global__ void __launch_bounds__(256)
    seg_grad_kernel(const float* __restrict__ blocks, float* __restrict__ g, int64_t S, int64_t d_seg,
                    int64_t dh, const float* __restrict__ sigma) {
    pdl_launch_dependents();
    pdl_wait();
    // blocks [S d_h, 128]: row s d_h + d of segment s holds sum_t kv[t, s d_h + d] dy[t, c]
    // for the 128 columns c of its group; segment s's own d_seg columns start at
    // (s mod (128 / d_seg)) d_seg.  g = [S][d_seg][d_h], divided by sigma_stale.
    const int64_t n = S * d_seg * dh;
    const int64_t spg = 128 / d_seg;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t s = i / (d_seg * dh);
        const int64_t r = i - s * d_seg * dh;
        const int64_t j = r / dh, d = r - j * dh;
        const int64_t row = s * dh + d;
        g[i] = __ldg(blocks + row * 128 + (s % spg) * d_seg + j) / __ldg(sigma + row);
    }
}

// Squared norm of the flat gradient: fp64 partial per CTA over a fixed range,
// then the partials in order.  coef = min(1, max_norm / (norm + 1e-6)).
constexpr int kNormCtas = 1024;
__global__ void __launch_bounds__(256)
    sqnorm_partial_kernel(const float* __restrict__ g, int64_t n, double* __restrict__ part) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t per = (n + gridDim.x - 1) / gridDim.x;
    const int64_t a = blockIdx.x * per, b = min(n, a + per);
    float s = 0.0f;
    for (int64_t i = a + threadIdx.x; i < b; i += blockDim.x) s = fmaf(g[i], g[i], s);
    __shared__ double red[256];
    red[threadIdx.x] = static_cast<double>(s);
    __syncthreads();
    for (int k = 128; k > 0; k >>= 1) {
        if (static_cast<int>(threadIdx.x) < k) red[threadIdx.x] += red[threadIdx.x + k];
        __syncthreads();
    }
    if (threadIdx.x == 0) part[blockIdx.x] = red[0];
}

__global__ void __launch_bounds__(256)
    sqnorm_reduce_kernel(const double* __restrict__ part, int n_part, float max_norm,
                         float* __restrict__ stats) {
    pdl_launch_dependents();
    pdl_wait();
    // a fixed-order tree over the partials (each thread a fixed stride of them)
    __shared__ double red[256];
    double t = 0.0;
    for (int i = threadIdx.x; i < n_part; i += blockDim.x) t += part[i];
    red[threadIdx.x] = t;
    __syncthreads();
    for (int k = 128; k > 0; k >>= 1) {
        if (static_cast<int>(threadIdx.x) < k) red[threadIdx.x] += red[threadIdx.x + k];
        __syncthreads();
    }
    if (threadIdx.x != 0) return;
    const double norm = sqrt(red[0]);
    stats[1] = static_cast<float>(norm);
    stats[2] = static_cast<float>(fmin(1.0, static_cast<double>(max_norm) / (norm + 1e-6)));
    stats[3] = 0.0f;
}

// AdamW on the flat parameter vector with the clipped gradient coef * g:
//   theta <- theta (1 - lr wd); m <- b1 m + (1 - b1) g; v <- b2 v + (1 - b2) g^2;
//   theta <- theta - lr (m / bc1) / (sqrt(v / bc2) + eps);  bf16 mirror rewritten.
__global__ void __launch_bounds__(256)
    adamw_kernel(float* __restrict__ p, float* __restrict__ m, float* __restrict__ v, const float* __restrict__ g,
                 uint16_t* __restrict__ pb, int64_t n, const __grid_constant__ AdamWParams hp,
                 const float* __restrict__ stats) {
    pdl_launch_dependents();
    pdl_wait();
    const float coef = stats[2];
    for (int64_t q = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; q < n / 4;
         q += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        float4 P4 = reinterpret_cast<float4*>(p)[q], M4 = reinterpret_cast<float4*>(m)[q];
        float4 V4 = reinterpret_cast<float4*>(v)[q];
        const float4 G4 = reinterpret_cast<const float4*>(g)[q];
        float* pp = &P4.x;
        float* mm = &M4.x;
        float* vv = &V4.x;
        const float* gg = &G4.x;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float gi = gg[k] * coef;
            const float th = pp[k] * (1.0f - hp.lr * hp.wd);
            mm[k] = hp.b1 * mm[k] + (1.0f - hp.b1) * gi;
            vv[k] = hp.b2 * vv[k] + (1.0f - hp.b2) * gi * gi;
            const float upd = (mm[k] / hp.bc1) / (sqrtf(vv[k] / hp.bc2) + hp.eps);
            pp[k] = th - hp.lr * upd;
        }
        reinterpret_cast<float4*>(p)[q] = P4;
        reinterpret_cast<float4*>(m)[q] = M4;
        reinterpret_cast<float4*>(v)[q] = V4;
        reinterpret_cast<uint2*>(pb)[q] = make_uint2(
            static_cast<uint32_t>(f32_to_bf16(P4.x)) | (static_cast<uint32_t>(f32_to_bf16(P4.y)) << 16),
            static_cast<uint32_t>(f32_to_bf16(P4.z)) | (static_cast<uint32_t>(f32_to_bf16(P4.w)) << 16));
    }
}


dim3 grid_for(int64_t n, int64_t cap_per_sm = 16) {
    int64_t b = (n + 255) / 256;
    const int64_t cap = static_cast<int64_t>(num_sms()) * cap_per_sm;
    if (b > cap) b = cap;
    if (b < 1) b = 1;
    return dim3(static_cast<unsigned>(b));
}

}  // namespace

cr_status launch_loss_head(const uint16_t* yf, const uint16_t* w_out, const float* b_out,
                           const float* sigma_delta, const uint16_t* stale, const uint16_t* joint, int64_t N,
                           int64_t D, int64_t db, const LossParams& p, uint16_t* dz, float* row_scale,
                           float* part, float* rowsq, float* loss_out, double* per_req, unsigned* status,
                           cudaStream_t st) {
    cr_status s = launch_pdl(row_scale_kernel, grid_for(N), dim3(256), 0, st, p, N, row_scale);
    if (s != CR_OK) return s;
    GemmParams gh{};
    gh.status = status;
    gh.bias = b_out;
    gh.sigma = sigma_delta;
    gh.loss_joint = joint;
    gh.loss_dz = dz;
    gh.row_scale = row_scale;
    gh.loss_part = part;
    if ((s = launch_gemm(yf, db, w_out, N, D, db, EPI_KV_LOSS, gh, const_cast<uint16_t*>(stale), D, st)) != CR_OK)
        return s;
    const int nparts = static_cast<int>(2 * (D / 128));
    s = launch_pdl(rowsq_kernel, dim3(static_cast<unsigned>((N + 31) / 32)), dim3(256), 0, st,
                   static_cast<const float*>(part), N, nparts, rowsq);
    if (s != CR_OK) return s;
    s = launch_pdl(loss_reduce_kernel, dim3(static_cast<unsigned>(p.n_req)), dim3(256), 0, st,
                   static_cast<const float*>(rowsq), p, D, per_req);
    if (s != CR_OK) return s;
    return launch_pdl(loss_total_kernel, dim3(1), dim3(32), 0, st, static_cast<const double*>(per_req), p.n_req,
                      loss_out);
}

size_t colsum_scratch_floats(int64_t rows, int64_t cols) {
    return static_cast<size_t>((rows + kColSlice - 1) / kColSlice) * static_cast<size_t>(cols);
}

size_t colsum_counters(int64_t cols) { return static_cast<size_t>((cols + 31) / 32); }

cr_status launch_colsum_bf16(const float* a, int64_t rows, int64_t cols, uint16_t* a16, float* out,
                             float* scratch, unsigned* counters, cudaStream_t st) {
    const int64_t slices = (rows + kColSlice - 1) / kColSlice;
    if (slices > 65535) return CR_ERR_UNSUPPORTED;
    if ((cols & 1) != 0) return CR_ERR_UNSUPPORTED;
    const dim3 g1(static_cast<unsigned>((cols + 63) / 64), static_cast<unsigned>(slices));
    return launch_pdl(colsum_kernel<float, true>, g1, dim3(256), 0, st, a, rows, cols, cols, a16, scratch, out,
                      0, counters);
}

cr_status launch_colsum(const void* a, bool bf16, int64_t rows, int64_t cols, int64_t lda, float* out,
                        bool accumulate, float* scratch, unsigned* counters, cudaStream_t st) {
    const int64_t slices = (rows + kColSlice - 1) / kColSlice;
    if (slices > 65535) return CR_ERR_UNSUPPORTED;
    if ((cols & 1) != 0 || (lda & 1) != 0) return CR_ERR_UNSUPPORTED;
    const dim3 g1(static_cast<unsigned>((cols + 63) / 64), static_cast<unsigned>(slices));
    uint16_t* none = nullptr;
    return bf16 ? launch_pdl(colsum_kernel<uint16_t, false>, g1, dim3(256), 0, st,
                             static_cast<const uint16_t*>(a), rows, cols, lda, none, scratch, out,
                             accumulate ? 1 : 0, counters)
                : launch_pdl(colsum_kernel<float, false>, g1, dim3(256), 0, st, static_cast<const float*>(a),
                             rows, cols, lda, none, scratch, out, accumulate ? 1 : 0, counters);
}

cr_status launch_ln_backward(const float* x, const float* gamma, const float* dy, const float* add, float eps,
                             int64_t N, int D, float* dx, float* gprod, cudaStream_t st) {
    if (D % 32 != 0 || D > 1024) return CR_ERR_UNSUPPORTED;
    return launch_pdl(ln_backward_kernel, dim3(static_cast<unsigned>((N + 7) / 8)), dim3(256), 0, st, x, gamma,
                      dy, add, eps, N, D, dx, gprod);
}

cr_status launch_gelu_backward(float* dg, const float* pre, int64_t n, cudaStream_t st) {
    return launch_pdl(gelu_backward_kernel, grid_for(n), dim3(256), 0, st, dg, pre, n);
}

cr_status launch_rope_backward(float* dqkv, const float2* table, int64_t N, int db, int hd, cudaStream_t st) {
    return launch_pdl(rope_backward_kernel, grid_for(N * db), dim3(256), 0, st, dqkv, table, N, db, hd);
}

cr_status launch_seg_grad(const float* blocks, float* g, int64_t S, int64_t dseg, int64_t dh,
                          const float* sigma, cudaStream_t st) {
    if (128 % dseg != 0) return CR_ERR_UNSUPPORTED;
    const int64_t n = S * dseg * dh;
    return launch_pdl(seg_grad_kernel, grid_for(n), dim3(256), 0, st, blocks, g, S, dseg, dh, sigma);
}

size_t sqnorm_scratch_doubles() { return kNormCtas; }

cr_status launch_clip_adamw(float* p, float* m, float* v, const float* g, uint16_t* pb, int64_t n,
                            const AdamWParams& hp, float max_norm, double* scratch, float* stats,
                            cudaStream_t st) {
    cr_status s = launch_pdl(sqnorm_partial_kernel, dim3(kNormCtas), dim3(256), 0, st, g, n, scratch);
    if (s != CR_OK) return s;
    s = launch_pdl(sqnorm_reduce_kernel, dim3(1), dim3(256), 0, st, static_cast<const double*>(scratch),
                   kNormCtas, max_norm, stats);
    if (s != CR_OK) return s;
    if (n % 4 != 0) return CR_ERR_UNSUPPORTED;
    return launch_pdl(adamw_kernel, grid_for(n / 4), dim3(256), 0, st, p, m, v, g, pb, n, hp,
                      static_cast<const float*>(stats));
}

}  // namespace cr
