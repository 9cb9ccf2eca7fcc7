// Bandwidth-bound kernels of the repair path:
//   gather_kernel     stale-cache assembly (Sec. 4.1, "Chunk-cache
//                     preparation": canonical chunk caches concatenated in
//                     document order; a pure copy, K is not rotated)
//   gather_emb_kernel the same for the embeddings and chunk map alone
//   layernorm_kernel  LayerNorm of the residual stream (optionally adding the
//                     block's reinjection P_b(s) first, Sec. 4.1 eq. for h^b)
//   to_bf16_kernel    fp32 cache/embedding -> bf16 operands for the tensor cores
//   split_bf16_kernel fp32 -> two-term bf16 operand (hi, lo) for the tensor cores
#include <cuda_bf16.h>

#include "cr_internal.h"
#include "cr_ptx.cuh"

namespace cr {
namespace {

// One CTA per output row (grid-stride).  A row is one token's D_KV cache
// values plus its d_model embedding values, each copied with 16-byte vectors,
// four loads in flight per thread before the matching stores.
__global__ void __launch_bounds__(512) gather_kernel(const __grid_constant__ GatherParams p) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t t = blockIdx.x; t < p.n_tokens; t += gridDim.x) {
        int lo = 0, hi = p.n_seg - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (p.seg[mid].dst_row <= t)
                lo = mid;
            else
                hi = mid - 1;
        }
        const GatherSeg& sg = p.seg[lo];
        const int64_t off = t - sg.dst_row;
        const int64_t src = sg.src_row + off;
        if (off < 0 || off >= sg.len || src < 0 || src >= p.n_pool_tokens) {
            if (threadIdx.x == 0) report(p.status, CR_DEV_INDEX, 1);
            continue;
        }
        if (threadIdx.x == 0) {
            p.chunk_id[t] = sg.chunk_local;
            p.pos[t] = static_cast<int32_t>(sg.local_start + off);
            p.chunk_end[t] = sg.local_start + sg.len;
        }
        for (int part = 0; part < 2; ++part) {
            const int64_t rb = part == 0 ? p.kv_row_bytes : p.emb_row_bytes;
            const uint4* s = reinterpret_cast<const uint4*>((part == 0 ? p.kv_pool : p.emb_pool) + src * rb);
            uint4* d = reinterpret_cast<uint4*>((part == 0 ? p.kv_out : p.emb_out) + t * rb);
            const int64_t nv = rb >> 4;
            for (int64_t base = threadIdx.x; base < nv; base += 4 * blockDim.x) {
                uint4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int64_t i = base + u * blockDim.x;
                    if (i < nv) v[u] = __ldcs(s + i);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int64_t i = base + u * blockDim.x;
                    if (i < nv) d[i] = v[u];
                }
            }
        }
    }
    if (blockIdx.x == 0 && static_cast<int>(threadIdx.x) <= p.n_req)
        p.cu_seqlens[threadIdx.x] = p.cu_seqlens_host[threadIdx.x];
}

// The same assembly without the cache rows (they go with the segment
// projection, which reads them from the pool): embedding rows and the chunk
// map, one warp per output row, eight 16-byte loads in flight per lane before
// the stores.
__global__ void __launch_bounds__(256) gather_emb_kernel(const __grid_constant__ GatherParams p) {
    pdl_launch_dependents();
    pdl_wait();
    const int wpb = static_cast<int>(blockDim.x >> 5);
    const int lane = static_cast<int>(threadIdx.x & 31);
    for (int64_t t = static_cast<int64_t>(blockIdx.x) * wpb + (threadIdx.x >> 5); t < p.n_tokens;
         t += static_cast<int64_t>(gridDim.x) * wpb) {
        int lo = 0, hi = p.n_seg - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (p.seg[mid].dst_row <= t)
                lo = mid;
            else
                hi = mid - 1;
        }
        const GatherSeg& sg = p.seg[lo];
        const int64_t off = t - sg.dst_row;
        const int64_t src = sg.src_row + off;
        if (off < 0 || off >= sg.len || src < 0 || src >= p.n_pool_tokens) {
            if (lane == 0) report(p.status, CR_DEV_INDEX, 2);
            continue;
        }
        if (lane == 0) {
            p.chunk_id[t] = sg.chunk_local;
            p.pos[t] = static_cast<int32_t>(sg.local_start + off);
            p.chunk_end[t] = sg.local_start + sg.len;
        }
        const uint4* s = reinterpret_cast<const uint4*>(p.emb_pool + src * p.emb_row_bytes);
        uint4* d = reinterpret_cast<uint4*>(p.emb_out + t * p.emb_row_bytes);
        const int64_t nv = p.emb_row_bytes >> 4;
        for (int64_t base = lane; base < nv; base += 8 * 32) {
            uint4 v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int64_t i = base + u * 32;
                if (i < nv) v[u] = __ldcs(s + i);
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int64_t i = base + u * 32;
                if (i < nv) d[i] = v[u];
            }
        }
    }
    if (blockIdx.x == 0)
        for (int i = static_cast<int>(threadIdx.x); i <= p.n_req; i += static_cast<int>(blockDim.x))
            p.cu_seqlens[i] = p.cu_seqlens_host[i];
}


// A row of D = 128 VPL values is held by WPR warps (WPR = 2 when VPL is even):
// each lane keeps VPL / WPR float4 of it in registers, so that a CTA of 256
// threads keeps 8 / WPR rows in flight with few registers per thread (many
// resident warps hide the memory latency).  Two-pass statistics from the
// registers (mean, then mean squared deviation: biased variance); the WPR
// warps of a row exchange their partial sums through shared memory.  gamma and
// beta are read after the statistics (they stay in L1).
template <int VPL, int WPR>
__global__ void __launch_bounds__(256) layernorm_kernel(const float* x,
                                                        const float* __restrict__ add,
                                                        int64_t ld_add, float* x_out,
                                                        const float* __restrict__ g,
                                                        const float* __restrict__ b, float eps,
                                                        int64_t M, uint16_t* __restrict__ u) {
    constexpr int D = VPL * 128;
    constexpr int HV = VPL / WPR;            // float4 per lane
    constexpr int RPB = 8 / WPR;             // rows per CTA
    static_assert(VPL % WPR == 0, "a row splits into whole float4 columns per warp");
    __shared__ float red[2][8];
    pdl_launch_dependents();
    pdl_wait();
    const int warp = static_cast<int>(threadIdx.x >> 5);
    const int part = warp % WPR;             // this warp's part of the row
    const int64_t row = static_cast<int64_t>(blockIdx.x) * RPB + warp / WPR;
    const int lane = threadIdx.x & 31;
    const bool live = row < M;
    const int64_t rr = live ? row : 0;       // rows past M read row 0 and write nothing
    const int c0 = part * (D / 4 / WPR);     // first float4 of this part
    float4 v[HV];
    const float4* xr = reinterpret_cast<const float4*>(x + rr * D) + c0;
#pragma unroll
    for (int k = 0; k < HV; ++k) v[k] = xr[lane + 32 * k];
    if (add) {
        float4 av[HV];
        const float4* ar = reinterpret_cast<const float4*>(add + rr * ld_add) + c0;
#pragma unroll
        for (int k = 0; k < HV; ++k) av[k] = ar[lane + 32 * k];
        float4* xo = reinterpret_cast<float4*>(x_out + rr * D) + c0;
#pragma unroll
        for (int k = 0; k < HV; ++k) {
            v[k].x += av[k].x;
            v[k].y += av[k].y;
            v[k].z += av[k].z;
            v[k].w += av[k].w;
            if (live) xo[lane + 32 * k] = v[k];
        }
    }
    // the row's sum over its WPR warps (the same order in every warp of the row)
    auto row_sum = [&](float s, int slot) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if constexpr (WPR == 1) {
            return s;
        } else {
            if (lane == 0) red[slot][warp] = s;
            __syncthreads();
            const int w0 = warp - part;
            float t = red[slot][w0];
#pragma unroll
            for (int q = 1; q < WPR; ++q) t += red[slot][w0 + q];
            return t;
        }
    };
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < HV; ++k) s += (v[k].x + v[k].y) + (v[k].z + v[k].w);
    const float mean = row_sum(s, 0) * (1.0f / D);
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < HV; ++k) {
        const float a = v[k].x - mean, bb = v[k].y - mean, c = v[k].z - mean, d = v[k].w - mean;
        q += (a * a + bb * bb) + (c * c + d * d);
    }
    const float rstd = rsqrtf(row_sum(q, 1) * (1.0f / D) + eps);
    if (!live) return;
    const float4* g4 = reinterpret_cast<const float4*>(g) + c0;
    const float4* b4 = reinterpret_cast<const float4*>(b) + c0;
    uint2* ur = reinterpret_cast<uint2*>(u + row * D) + c0;
#pragma unroll
    for (int k = 0; k < HV; ++k) {
        const float4 gg = __ldg(g4 + lane + 32 * k), bq = __ldg(b4 + lane + 32 * k);
        uint2 w;
        w.x = pack_bf16x2((v[k].x - mean) * rstd * gg.x + bq.x, (v[k].y - mean) * rstd * gg.y + bq.y);
        w.y = pack_bf16x2((v[k].z - mean) * rstd * gg.z + bq.z, (v[k].w - mean) * rstd * gg.w + bq.w);
        ur[lane + 32 * k] = w;
    }
}

__global__ void to_bf16_kernel(const float* __restrict__ x, int64_t n, uint16_t* __restrict__ y) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const __nv_bfloat16 b = __float2bfloat16_rn(x[i]);
        y[i] = *reinterpret_cast<const uint16_t*>(&b);
    }
}

// Two-term bf16 operand of an fp32 matrix: x [rows, cols] fp32 (contiguous)
// -> out row r = [hi (cols) | lo (cols)], hi = rn(x), lo = rn(x - hi); eight
// values per thread.  cols is a multiple of 8.
__global__ void split_bf16_kernel(const float* __restrict__ x, int64_t rows, int64_t cols,
                                  uint16_t* __restrict__ out) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t c8 = cols >> 3;
    const int64_t n8 = rows * c8;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n8;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t r = i / c8, c = (i - r * c8) << 3;
        const float4* src = reinterpret_cast<const float4*>(x + r * cols + c);
        const float4 a = src[0], b = src[1];
        uint32_t h[4], l[4];
        split_bf16x2(a.x, a.y, &h[0], &l[0]);
        split_bf16x2(a.z, a.w, &h[1], &l[1]);
        split_bf16x2(b.x, b.y, &h[2], &l[2]);
        split_bf16x2(b.z, b.w, &h[3], &l[3]);
        uint16_t* o = out + r * 2 * cols + c;
        *reinterpret_cast<uint4*>(o) = make_uint4(h[0], h[1], h[2], h[3]);
        *reinterpret_cast<uint4*>(o + cols) = make_uint4(l[0], l[1], l[2], l[3]);
    }
}

struct InvFreq {
    float f[64];
};

// (cos, sin) of pos[t] * inv_freq[q] for every token and pair index, the angle's
// product rounding folded back in (same arithmetic as the in-epilogue path).
// Angle-major: entry q * n + t, so that the rows of a tile read it coalesced.
__global__ void rope_table_kernel(const int32_t* __restrict__ pos, int64_t n, int half,
                                  const __grid_constant__ InvFreq f, float2* __restrict__ table) {
    pdl_launch_dependents();
    pdl_wait();
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n * half;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int q = static_cast<int>(i / n);
        const int64_t t = i - static_cast<int64_t>(q) * n;
        float s, c;
        sincos_prod(static_cast<float>(__ldg(pos + t)), f.f[q], &s, &c);
        table[i] = make_float2(c, s);
    }
}

}  // namespace

cr_status launch_rope_table(const int32_t* pos, int64_t n, int half_dim, const float* inv_freq_host,
                            float2* table, cudaStream_t st) {
    if (n <= 0) return CR_OK;
    if (half_dim < 1 || half_dim > 64) return CR_ERR_UNSUPPORTED;
    InvFreq f{};
    for (int i = 0; i < half_dim; ++i) f.f[i] = inv_freq_host[i];
    int64_t blocks = (n * half_dim + 255) / 256;
    if (blocks > static_cast<int64_t>(num_sms()) * 8) blocks = static_cast<int64_t>(num_sms()) * 8;
    return launch_pdl(rope_table_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, pos, n,
                      half_dim, f, table);
}

// The pool row of every request token (the gather's segment table); per
// 128-row box of the request the pool row of its first token when all 128 rows
// lie in one chunk (a contiguous pool range), else -1; and the same per 8-row
// group, for the boxes that straddle chunks (16 groups per box, -1 for groups
// past the request's end).
__global__ void __launch_bounds__(256) src_rows_kernel(const __grid_constant__ GatherParams p,
                                                       int64_t* __restrict__ src_row,
                                                       int64_t* __restrict__ box_src,
                                                       int64_t* __restrict__ grp_src) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t n_box = (p.n_tokens + 127) / 128;
    const int64_t n_grp = 16 * n_box;
    const int64_t n = p.n_tokens > n_grp ? p.n_tokens : n_grp;
    auto seg_of = [&](int64_t t) {
        int lo = 0, hi = p.n_seg - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (p.seg[mid].dst_row <= t)
                lo = mid;
            else
                hi = mid - 1;
        }
        return lo;
    };
    // first row of rows [t0, t0 + len) in the pool when they are one chunk's, else -1
    auto run_src = [&](int64_t t0, int64_t len) -> int64_t {
        const int64_t t1 = t0 + len - 1;
        if (t1 >= p.n_tokens) return -1;
        const GatherSeg& sg = p.seg[seg_of(t0)];
        const bool one = t1 < sg.dst_row + sg.len && t0 >= sg.dst_row;
        return one ? sg.src_row + (t0 - sg.dst_row) : -1;
    };
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        if (i < p.n_tokens) {
            const GatherSeg& sg = p.seg[seg_of(i)];
            const int64_t off = i - sg.dst_row;
            if (off < 0 || off >= sg.len || sg.src_row + off >= p.n_pool_tokens) {
                report(p.status, CR_DEV_INDEX, 3);
                src_row[i] = 0;
            } else {
                src_row[i] = sg.src_row + off;
            }
        }
        if (i < n_box) box_src[i] = run_src(128 * i, 128);
        if (i < n_grp) grp_src[i] = run_src(8 * i, 8);
    }
}

cr_status launch_src_rows(const GatherParams& p, int64_t* src_row, int64_t* box_src, int64_t* grp_src,
                          cudaStream_t st) {
    if (p.n_tokens <= 0) return CR_OK;
    const int64_t n_grp = 16 * ((p.n_tokens + 127) / 128);
    const int64_t n = p.n_tokens > n_grp ? p.n_tokens : n_grp;
    const int64_t grid = (n + 255) / 256;
    return launch_pdl(src_rows_kernel, dim3(static_cast<unsigned>(grid)), dim3(256), 0, st, p, src_row,
                      box_src, grp_src);
}

cr_status launch_gather(const GatherParams& p, cudaStream_t st) {
    if (p.n_tokens <= 0) return CR_OK;
    if (p.kv_row_bytes == 0) {
        // no cache rows: every row's embedding copy in flight at once (8 rows per block)
        const int64_t grid = (p.n_tokens + 7) / 8;
        return launch_pdl(gather_emb_kernel, dim3(static_cast<unsigned>(grid)), dim3(256), 0, st, p);
    }
    int64_t grid = static_cast<int64_t>(num_sms()) * 4;
    if (grid > p.n_tokens) grid = p.n_tokens;
    return launch_pdl(gather_kernel, dim3(static_cast<unsigned>(grid)), dim3(512), 0, st, p);
}

cr_status launch_layernorm(const float* x, const float* add, int64_t ld_add, float* x_out,
                           const float* g, const float* b, float eps, int64_t M, int64_t D,
                           uint16_t* u, cudaStream_t st) {
    if (M <= 0) return CR_OK;
    switch (D) {
#define CR_LN_CASE(V)                                                                          \
    case V * 128: {                                                                            \
        constexpr int W = (V % 2 == 0) ? 2 : 1;                                                \
        const int grid = static_cast<int>((M + 8 / W - 1) / (8 / W));                          \
        return launch_pdl(layernorm_kernel<V, W>, dim3(grid), dim3(256), 0, st, x, add, ld_add, \
                          x_out, g, b, eps, M, u);                                             \
    }
        CR_LN_CASE(1)
        CR_LN_CASE(2)
        CR_LN_CASE(3)
        CR_LN_CASE(4)
        CR_LN_CASE(5)
        CR_LN_CASE(6)
        CR_LN_CASE(7)
        CR_LN_CASE(8)
#undef CR_LN_CASE
        default:
            return CR_ERR_UNSUPPORTED;
    }
}

cr_status launch_split_bf16(const float* x, int64_t rows, int64_t cols, uint16_t* out,
                            cudaStream_t st) {
    if (rows <= 0) return CR_OK;
    if ((cols % 8) != 0) return CR_ERR_UNSUPPORTED;
    const int64_t n8 = rows * (cols / 8);
    int64_t blocks = (n8 + 255) / 256;
    if (blocks > 8 * 1024) blocks = 8 * 1024;
    return launch_pdl(split_bf16_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, x,
                      rows, cols, out);
}

cr_status launch_to_bf16(const float* x, int64_t n, uint16_t* y, cudaStream_t st) {
    if (n <= 0) return CR_OK;
    int64_t blocks = (n + 255) / 256;
    if (blocks > static_cast<int64_t>(num_sms()) * 16) blocks = static_cast<int64_t>(num_sms()) * 16;
    return launch_pdl(to_bf16_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, x, n, y);
}

// One CTA waiting on a pipeline barrier that nothing arrives on, through the
// same bounded wait every kernel uses: after CR_WAIT_TIMEOUT_NS the wait gives
// up, records a timeout at site 900 in the status word and the kernel returns.
// A check of the failure reporting that neither hangs nor faults the GPU.
namespace {
__global__ void wait_selftest_kernel(unsigned* status) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const WaitCtx wc{&abort_flag, status};
        mbar_wait(&bar, 0, wc, 900);
    }
}
}  // namespace

cr_status launch_wait_selftest(unsigned* status, cudaStream_t st) {
    wait_selftest_kernel<<<1, 32, 0, st>>>(status);
    return cuda_check(cudaGetLastError());
}

}  // namespace cr
