// Backward of the Repair Blocks' masked attention (the mask modes of the
// forward, Sec. 4.1 and App. F), for the training step (Sec. 4.2).  With the
// forward's log-sum-exp per row (lse2, log2 units, scale folded in),
// D_q = sum_d dO[q, d] O[q, d] and c = log2(e) / sqrt(d):
//   P = 2^(s c - lse2) on the visible keys (0 elsewhere), dP = dO V^T,
//   dS = P (dP - D),  dV = P^T dO,  dK = dS^T Q / sqrt(d),  dQ = dS K / sqrt(d).
// Two kernels, each a tcgen05 pipeline like the forward's:
//   attn_bwd_kernel<D, true>   one CTA per (request, 128-key tile, head): walks
//       the query tiles that see any of its keys; S^T = K Q^T and dP^T = V dO^T
//       into TMEM; the elementwise warps (one key row per thread) write P^T and
//       dS^T back as bf16; dV += P^T dO and dK += dS^T Q accumulate in TMEM (the
//       TS form: A from TMEM, B = the query tile's rows, MN-major) and are
//       written once, so no atomics.
//   attn_bwd_kernel<D, false>  one CTA per (request, 128-query tile, head):
//       walks the key tiles it sees (as the forward); S = Q K^T, dP = dO V^T,
//       dS into TMEM, dQ += dS K.
// Warp 0 loads by TMA (the CTA's own two tiles once, the walked tiles' pairs
// into a 2-stage ring), warp 1 issues the MMAs and owns TMEM, warps 4-7 and
// 8-11 do the exponentials on the same rows (TMEM lanes), the first group the
// low 64 columns of each tile and the second the high 64, 32 at a time, so two
// warps share each SM sub-partition.  Every wait is bounded.
#include <cuda_bf16.h>

#include "cr_internal.h"
#include "cr_ptx.cuh"

namespace cr {
namespace {

template <int D>
struct BwdCfg {
    static constexpr uint32_t kRowBytes = D * 2;
    static constexpr uint32_t kAtomBytes = 8 * kRowBytes;
    static constexpr uint32_t kTileBytes = 128 * kRowBytes;
    static constexpr uint32_t kSwz = (D == 64) ? SWZ_128B : SWZ_64B;
    static constexpr int kStages = 2;
    static constexpr uint32_t kFixOff = 0;                          // own tiles A0, A1
    static constexpr uint32_t kRingOff = 2 * kTileBytes;            // walked tiles B0, B1 per stage
    static constexpr uint32_t kVecOff = kRingOff + kStages * 2 * kTileBytes;   // [2][4][128] fp32
    static constexpr uint32_t kBarOff = kVecOff + 2 * 4 * 128 * 4;
    static constexpr uint32_t kSmemBytes = 1024 + kBarOff + 256;
    static constexpr uint32_t kTmemS = 0, kTmemDP = 128, kTmemAcc0 = 256, kTmemAcc1 = 320;
    static constexpr uint32_t kTmemP = 384, kTmemDS = 448;
};

constexpr int kBwdThreads = 384;

__device__ __forceinline__ int bwd_hi(const AttnBwdParams& p, int rs, int len, int q) {
    if (p.mask_mode == CR_MASK_TOKEN_CAUSAL) return q + 1;
    if (p.mask_mode == CR_MASK_BIDIRECTIONAL) return len;
    return __ldg(p.chunk_end + rs + q);
}
__device__ __forceinline__ int bwd_lo(const AttnBwdParams& p, int rs, int q) {
    return p.mask_mode == CR_MASK_BLOCK_DIAGONAL ? __ldg(p.chunk_start + rs + q) : 0;
}

template <int D, bool KV>
__global__ void __launch_bounds__(kBwdThreads, 1)
    attn_bwd_kernel(const __grid_constant__ CUtensorMap tmQKV, const __grid_constant__ CUtensorMap tmDO,
                    const __grid_constant__ AttnBwdParams p) {
    using Cfg = BwdCfg<D>;
    constexpr int NS = Cfg::kStages;
    constexpr uint32_t IDESC_S = idesc_bf16(128, 128, false, false);
    constexpr uint32_t IDESC_PV = idesc_bf16(128, D, false, true);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    float* vec = reinterpret_cast<float*>(smem + Cfg::kVecOff);   // [buf][(lse, D) x 128, hi, lo]
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg::kBarOff);
    uint64_t* fix_full = bars;
    uint64_t* kv_full = bars + 1;
    uint64_t* kv_empty = kv_full + NS;
    uint64_t* s_full = kv_empty + NS;
    uint64_t* s_free = s_full + 1;
    uint64_t* p_full = s_free + 1;
    uint64_t* pv_done = p_full + 1;
    uint64_t* drain = pv_done + 1;
    uint64_t* vec_full = drain + 1;   // [2]: a walked tile's vectors in smem (KV kernel)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(vec_full + 2);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    // ---- work item: (request, own tile, head)
    const int head = blockIdx.x % p.n_heads;
    const int item = static_cast<int>(blockIdx.x / p.n_heads);
    int req = 0;
    while (req + 1 < p.n_req && p.tile_prefix[req + 1] <= item) ++req;
    const int t0 = (item - p.tile_prefix[req]) * 128;   // own tile's first row (request-local)
    const int rs = p.req_start[req];
    const int len = p.req_start[req + 1] - rs;
    const int total = p.req_start[p.n_req];

    const uint32_t warp = warp_id(), lane = lane_id();
    pdl_launch_dependents();
    if (threadIdx.x == 0) {
        mbar_init(fix_full, 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
        mbar_init(s_full, 1);
        mbar_init(s_free, 8);
        mbar_init(p_full, 8);
        mbar_init(pv_done, 1);
        mbar_init(drain, 1);
        mbar_init(&vec_full[0], 256);
        mbar_init(&vec_full[1], 256);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    pdl_wait();   // qkv, dO, lse, D and the chunk map come from earlier kernels

    // walked tiles [w0, w0 + nw) of 128 rows each (request-local)
    int w0, nw;
    if constexpr (KV) {
        // queries that see a key of [t0, t0 + 128): hi(q) > t0 and lo(q) < t0 + 128
        const int klast = min(t0 + 127, len - 1);
        int qa, qb;
        if (p.mask_mode == CR_MASK_TOKEN_CAUSAL) {
            qa = t0;
            qb = len;
        } else if (p.mask_mode == CR_MASK_BIDIRECTIONAL) {
            qa = 0;
            qb = len;
        } else if (p.mask_mode == CR_MASK_BLOCK_DIAGONAL) {
            qa = __ldg(p.chunk_start + rs + t0);
            qb = __ldg(p.chunk_end + rs + klast);
        } else {   // block-causal: from the start of t0's chunk to the end
            qa = __ldg(p.chunk_start + rs + t0);
            qb = len;
        }
        w0 = qa / 128;
        nw = qb > qa ? (qb + 127) / 128 - w0 : 0;
    } else {
        const int last = min(t0 + 127, len - 1);
        w0 = bwd_lo(p, rs, t0) / 128;
        nw = (bwd_hi(p, rs, len, last) + 127) / 128 - w0;
    }
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx wc{abort_flag, p.status};

    if (warp == 0) {
        // ---------------------------------------------------- TMA producer
        if (elect_one()) {
            tma_prefetch(&tmQKV);
            tma_prefetch(&tmDO);
            mbar_expect_tx(fix_full, 2 * Cfg::kTileBytes);
            if constexpr (KV) {   // own tiles: K, V of the key tile
                tma_load_2d(smem + Cfg::kFixOff, &tmQKV, fix_full, p.d_b + head * D, rs + t0);
                tma_load_2d(smem + Cfg::kFixOff + Cfg::kTileBytes, &tmQKV, fix_full, 2 * p.d_b + head * D,
                            rs + t0);
            } else {              // own tiles: Q, dO of the query tile
                tma_load_2d(smem + Cfg::kFixOff, &tmQKV, fix_full, head * D, rs + t0);
                tma_load_2d(smem + Cfg::kFixOff + Cfg::kTileBytes, &tmDO, fix_full, head * D, rs + t0);
            }
        }
        __syncwarp();
        bool ok = true;
        for (int j = 0; j < nw; ++j) {
            const int st = j % NS;
            if (!(ok = mbar_wait_warp(&kv_empty[st], (static_cast<uint32_t>(j / NS) & 1u) ^ 1u, wc, 131))) break;
            uint8_t* b = smem + Cfg::kRingOff + st * 2 * Cfg::kTileBytes;
            const int row = rs + (w0 + j) * 128;
            if (elect_one()) {
                mbar_expect_tx(&kv_full[st], 2 * Cfg::kTileBytes);
                if constexpr (KV) {   // walked: Q, dO of a query tile
                    tma_load_2d(b, &tmQKV, &kv_full[st], head * D, row);
                    tma_load_2d(b + Cfg::kTileBytes, &tmDO, &kv_full[st], head * D, row);
                } else {              // walked: K, V of a key tile
                    tma_load_2d(b, &tmQKV, &kv_full[st], p.d_b + head * D, row);
                    tma_load_2d(b + Cfg::kTileBytes, &tmQKV, &kv_full[st], 2 * p.d_b + head * D, row);
                }
            }
            __syncwarp();
        }
        if (!ok) {
            const uint64_t tw = globaltimer();
            while (globaltimer() - tw < 50000ull) {
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        constexpr uint64_t kStageStep = (2 * Cfg::kTileBytes) >> 4;
        constexpr uint64_t kRow16 = (16 * Cfg::kRowBytes) >> 4;
        const uint32_t a0 = smem_u32(smem + Cfg::kFixOff), a1 = a0 + Cfg::kTileBytes;
        const uint32_t b0 = smem_u32(smem + Cfg::kRingOff), b1 = b0 + Cfg::kTileBytes;
        // K-major views (S-like products) and MN-major views (the TS products' B)
        const uint64_t dA0 = smem_desc(a0, 16, Cfg::kAtomBytes, Cfg::kSwz);
        const uint64_t dA1 = smem_desc(a1, 16, Cfg::kAtomBytes, Cfg::kSwz);
        const uint64_t dB0k = smem_desc(b0, 16, Cfg::kAtomBytes, Cfg::kSwz);
        const uint64_t dB1k = smem_desc(b1, 16, Cfg::kAtomBytes, Cfg::kSwz);
        const uint64_t dB0m = smem_desc(b0, Cfg::kTileBytes, Cfg::kAtomBytes, Cfg::kSwz);
        const uint64_t dB1m = smem_desc(b1, Cfg::kTileBytes, Cfg::kAtomBytes, Cfg::kSwz);
        const uint32_t tS = tmem_base + Cfg::kTmemS, tDP = tmem_base + Cfg::kTmemDP;
        const uint32_t tAcc0 = tmem_base + Cfg::kTmemAcc0, tAcc1 = tmem_base + Cfg::kTmemAcc1;
        const uint32_t tP = tmem_base + Cfg::kTmemP, tDS = tmem_base + Cfg::kTmemDS;
        bool ok = mbar_wait_warp(fix_full, 0, wc, 231);
        if (ok) tc_fence_after();
        for (int j = 0; j < nw && ok; ++j) {
            const int st = j % NS;
            const uint64_t so = static_cast<uint64_t>(st) * kStageStep;
            if (!(ok = mbar_wait_warp(&kv_full[st], static_cast<uint32_t>(j / NS) & 1u, wc, 232))) break;
            tc_fence_after();
            if (j > 0) {
                if (!(ok = mbar_wait_warp(s_free, static_cast<uint32_t>(j - 1) & 1u, wc, 233))) break;
                tc_fence_after();
            }
            // KV: S^T = K Q^T, dP^T = V dO^T;  Q: S = Q K^T, dP = dO V^T  (A = own tile, B = walked)
            if (elect_one()) {
#pragma unroll
                for (int k = 0; k < D / 16; ++k)
                    mma_bf16_ss(tS, dA0 + 2 * k, dB0k + so + 2 * k, IDESC_S, k != 0 ? 1u : 0u);
#pragma unroll
                for (int k = 0; k < D / 16; ++k)
                    mma_bf16_ss(tDP, dA1 + 2 * k, dB1k + so + 2 * k, IDESC_S, k != 0 ? 1u : 0u);
                mma_commit(s_full);
            }
            __syncwarp();
            if (!(ok = mbar_wait_warp(p_full, static_cast<uint32_t>(j) & 1u, wc, 234))) break;
            tc_fence_after();
            if (elect_one()) {
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t acc = (j > 0 || kk != 0) ? 1u : 0u;
                    if constexpr (KV) {
                        // dV += P^T dO (B = dO rows of the query tile), dK += dS^T Q
                        mma_bf16_ts(tAcc0, tP + kk * 8, dB1m + so + kk * kRow16, IDESC_PV, acc);
                        mma_bf16_ts(tAcc1, tDS + kk * 8, dB0m + so + kk * kRow16, IDESC_PV, acc);
                    } else {
                        // dQ += dS K (B = K rows of the key tile)
                        mma_bf16_ts(tAcc0, tDS + kk * 8, dB0m + so + kk * kRow16, IDESC_PV, acc);
                    }
                }
                mma_commit(pv_done);
                mma_commit(&kv_empty[st]);
            }
            __syncwarp();
        }
        if (elect_one()) mma_commit(drain);
        __syncwarp();
        mbar_wait_warp(drain, 0, wc, 237);
    } else if (warp >= 4) {
        // ---------------------------------------------------- elementwise warps
        const uint32_t quad = warp & 3u;
        const int eg = (static_cast<int>(warp) - 4) >> 2;   // column half 0 / 1
        const int r = static_cast<int>(quad * 32 + lane);
        const int own = t0 + r;                  // this thread's row of the own tile
        const bool own_ok = own < len;
        const uint32_t lo16 = (quad * 32u) << 16;
        const uint32_t tS = tmem_base + lo16 + Cfg::kTmemS, tDP = tmem_base + lo16 + Cfg::kTmemDP;
        const uint32_t tP = tmem_base + lo16 + Cfg::kTmemP, tDS = tmem_base + lo16 + Cfg::kTmemDS;
        const float cl = p.scale_log2;
        // Q kernel: the row's own log-sum-exp, D and visible keys
        float my_lse = 0.0f, my_d = 0.0f;
        int my_hi = 0, my_lo = 0;
        if constexpr (!KV) {
            if (own_ok) {
                my_lse = __ldg(p.lse + static_cast<int64_t>(head) * total + rs + own);
                my_d = __ldg(p.dvec + static_cast<int64_t>(head) * total + rs + own);
                my_hi = bwd_hi(p, rs, len, own);
                my_lo = bwd_lo(p, rs, own);
            }
        }
        bool ok = true;
        for (int j = 0; j < nw && ok; ++j) {
            const int wrow0 = (w0 + j) * 128;    // walked tile's first row (request-local)
            float* vb = vec + (j & 1) * 4 * 128;
            if constexpr (KV) {
                // the walked query tile's lse, D and visible-key bounds, one per
                // thread of the first group; both groups arrive, so a buffer is
                // rewritten (two tiles later) only after both have passed the tile
                // in between
                if (eg == 0) {
                    const int q = wrow0 + r;
                    const bool qv = q < len;
                    reinterpret_cast<float2*>(vb)[r] =
                        qv ? make_float2(__ldg(p.lse + static_cast<int64_t>(head) * total + rs + q),
                                         __ldg(p.dvec + static_cast<int64_t>(head) * total + rs + q))
                           : make_float2(0.0f, 0.0f);
                    vb[256 + r] = __int_as_float(qv ? bwd_hi(p, rs, len, q) : 0);
                    vb[384 + r] = __int_as_float(qv ? bwd_lo(p, rs, q) : 0);
                }
                mbar_arrive(&vec_full[j & 1]);
                ok = mbar_wait(&vec_full[j & 1], static_cast<uint32_t>(j >> 1) & 1u, wc, 330);
                if (!__all_sync(0xffffffffu, ok)) {
                    ok = false;
                    break;
                }
            }
            ok = mbar_wait(s_full, static_cast<uint32_t>(j) & 1u, wc, 331);
            if (!__all_sync(0xffffffffu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            // KV: does every query of the walked tile see this key?  (hi and lo never
            // decrease along the queries, so the first hi and the last lo decide)
            bool full = false;
            if constexpr (KV)
                full = own_ok && wrow0 + 127 < len && own < __float_as_int(vb[256]) &&
                       own >= __float_as_int(vb[384 + 127]);
            for (int c0 = eg * 64; c0 < eg * 64 + 64; c0 += 32) {
                float s[32], dp[32];
                tmem_ld32(tS + c0, s);
                tmem_ld32(tDP + c0, dp);
                tmem_wait_ld();
                if (c0 == eg * 64 + 32) {   // this half of S and dP read: the next tile's MMAs may overwrite them
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(s_free);
                }
                float pv[32], dsv[32];
                if (KV && full) {
                    const float2* ld = reinterpret_cast<const float2*>(vb) + c0;
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const float2 e = ld[i];
                        const float pr = ex2(fmaf(s[i], cl, -e.x));
                        pv[i] = pr;
                        dsv[i] = pr * (dp[i] - e.y);
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        bool vis;
                        float lse, dd;
                        if constexpr (KV) {   // this thread's key against query column c0 + i
                            const int qi = c0 + i;
                            vis = own_ok && own < __float_as_int(vb[256 + qi]) &&
                                  own >= __float_as_int(vb[384 + qi]);
                            const float2 e = reinterpret_cast<const float2*>(vb)[qi];
                            lse = e.x;
                            dd = e.y;
                        } else {              // this thread's query against key column c0 + i
                            const int k = wrow0 + c0 + i;
                            vis = own_ok && k < my_hi && k >= my_lo;
                            lse = my_lse;
                            dd = my_d;
                        }
                        const float pr = vis ? ex2(fmaf(s[i], cl, -lse)) : 0.0f;
                        pv[i] = pr;
                        dsv[i] = pr * (dp[i] - dd);
                    }
                }
                uint32_t pk[16], dk[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    pk[i] = pack_bf16x2(pv[2 * i], pv[2 * i + 1]);
                    dk[i] = pack_bf16x2(dsv[2 * i], dsv[2 * i + 1]);
                }
                if (c0 == eg * 64 && j > 0) {   // the previous tile's TS products read P and dS
                    ok = mbar_wait(pv_done, static_cast<uint32_t>(j - 1) & 1u, wc, 332);
                    if (!__all_sync(0xffffffffu, ok)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                }
                float pf[16], df[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    pf[i] = __uint_as_float(pk[i]);
                    df[i] = __uint_as_float(dk[i]);
                }
                if constexpr (KV) tmem_st16(tP + c0 / 2, pf);
                tmem_st16(tDS + c0 / 2, df);
            }
            if (!ok) break;
            tmem_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(p_full);
        }
        // results: dV, dK (KV) or dQ, one row per thread, into dqkv [N, 3 d_b] fp32
        if (ok && nw > 0) {
            ok = mbar_wait(pv_done, static_cast<uint32_t>(nw - 1) & 1u, wc, 334);
            ok = __all_sync(0xffffffffu, ok);
            if (ok) tc_fence_after();
        }
        if (ok) {
            float* row = p.dqkv + static_cast<int64_t>(rs + own) * 3 * p.d_b;
#pragma unroll
            for (int a = 0; a < (KV ? 2 : 1); ++a) {
                // KV: acc0 = dV (column block 2 d_b), acc1 = dK (d_b, scaled); Q: acc0 = dQ (0, scaled)
                const uint32_t ta = tmem_base + lo16 + (a == 0 ? Cfg::kTmemAcc0 : Cfg::kTmemAcc1);
                const float f = (KV && a == 0) ? 1.0f : p.scale;
                float* dst = row + (KV ? (a == 0 ? 2 * p.d_b : p.d_b) : 0) + head * D;
#pragma unroll
                for (int c = eg * (D / 2); c < (eg + 1) * (D / 2); c += 16) {
                    float v[16];
                    if (nw > 0) {
                        tmem_ld16(ta + c, v);
                        tmem_wait_ld();
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) v[i] = 0.0f;
                    }
                    if (own_ok) {
                        float4* d4 = reinterpret_cast<float4*>(dst + c);
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            d4[i] = make_float4(v[4 * i] * f, v[4 * i + 1] * f, v[4 * i + 2] * f, v[4 * i + 3] * f);
                    }
                }
            }
        }
        tc_fence_before();
    }
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, 512);
    }
}

// D[h][t] = sum_d dO[t, h d + d] O[t, h d + d]: one thread per (token, head)
__global__ void __launch_bounds__(256)
    attn_bwd_dvec_kernel(const float* __restrict__ dO, const uint16_t* __restrict__ O, int64_t N, int db, int hd,
                         float* __restrict__ dvec) {
    pdl_launch_dependents();
    pdl_wait();
    const int heads = db / hd;
    const int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
    if (i >= N * heads) return;
    const int64_t t = i / heads;
    const int h = static_cast<int>(i - t * heads);
    const float* a = dO + t * db + h * hd;
    const uint16_t* o = O + t * db + h * hd;
    float s = 0.0f;
    for (int k = 0; k < hd; k += 8) {
        const uint4 w = *reinterpret_cast<const uint4*>(o + k);
        const float4 x0 = *reinterpret_cast<const float4*>(a + k);
        const float4 x1 = *reinterpret_cast<const float4*>(a + k + 4);
        s = fmaf(x0.x, __uint_as_float(w.x << 16), s);
        s = fmaf(x0.y, __uint_as_float(w.x & 0xFFFF0000u), s);
        s = fmaf(x0.z, __uint_as_float(w.y << 16), s);
        s = fmaf(x0.w, __uint_as_float(w.y & 0xFFFF0000u), s);
        s = fmaf(x1.x, __uint_as_float(w.z << 16), s);
        s = fmaf(x1.y, __uint_as_float(w.z & 0xFFFF0000u), s);
        s = fmaf(x1.z, __uint_as_float(w.w << 16), s);
        s = fmaf(x1.w, __uint_as_float(w.w & 0xFFFF0000u), s);
    }
    dvec[static_cast<int64_t>(h) * N + t] = s;
}

template <int D>
cr_status launch_bwd_d(const CUtensorMap& tq, const CUtensorMap& td, const AttnBwdParams& p, cudaStream_t st) {
    using Cfg = BwdCfg<D>;
    static unsigned long long attr_kv = 0, attr_q = 0;
    cr_status s = ensure_smem_attr(attn_bwd_kernel<D, true>, static_cast<int>(Cfg::kSmemBytes), &attr_kv);
    if (s == CR_OK) s = ensure_smem_attr(attn_bwd_kernel<D, false>, static_cast<int>(Cfg::kSmemBytes), &attr_q);
    if (s != CR_OK) return s;
    const dim3 grid(static_cast<unsigned>(p.n_items * p.n_heads));
    s = launch_pdl(attn_bwd_kernel<D, true>, grid, dim3(kBwdThreads), Cfg::kSmemBytes, st, tq, td, p);
    if (s != CR_OK) return s;
    return launch_pdl(attn_bwd_kernel<D, false>, grid, dim3(kBwdThreads), Cfg::kSmemBytes, st, tq, td, p);
}

}  // namespace

cr_status launch_attention_backward(const uint16_t* qkv, const uint16_t* dO16, const float* dO, const uint16_t* O,
                                    int64_t n_tokens, int head_dim, AttnBwdParams& p, float* dvec, cudaStream_t st) {
    if (head_dim != 32 && head_dim != 64) return CR_ERR_UNSUPPORTED;
    if (p.n_items <= 0) return CR_OK;
    const int64_t pairs = n_tokens * (p.d_b / head_dim);
    cr_status s = launch_pdl(attn_bwd_dvec_kernel, dim3(static_cast<unsigned>((pairs + 255) / 256)), dim3(256), 0,
                             st, dO, O, n_tokens, p.d_b, head_dim, dvec);
    if (s != CR_OK) return s;
    p.dvec = dvec;
    CUtensorMap tq, td;
    const CUtensorMapSwizzle sw = head_dim == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    if (!make_tmap_2d(&tq, qkv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3ull * p.d_b, n_tokens, 3ull * p.d_b * 2,
                      head_dim, 128, sw))
        return CR_ERR_INVALID_ARG;
    if (!make_tmap_2d(&td, dO16, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, static_cast<uint64_t>(p.d_b), n_tokens,
                      static_cast<uint64_t>(p.d_b) * 2, head_dim, 128, sw))
        return CR_ERR_INVALID_ARG;
    return head_dim == 64 ? launch_bwd_d<64>(tq, td, p, st) : launch_bwd_d<32>(tq, td, p, st);
}

}  // namespace cr
