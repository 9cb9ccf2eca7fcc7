// Chunk-block-causal attention of the Repair Blocks (Sec. 4.1):
//   o_i = sum_{j : c(j) <= c(i)} softmax_j(q_i . k_j / sqrt(d)) v_j
// inside each request.  Chunk ids are non-decreasing along a request, so the
// keys visible to query i are exactly j < chunk_end[i]: a prefix.  A query
// tile [q0, q0+128) therefore needs key tiles 0 .. ceil(max_i chunk_end / 128)
// and nothing past that; those tiles are never loaded or multiplied.  Inside
// the last tiles a per-row compare against chunk_end masks the rest.
//
// CTA = (request, 128-query tile, head).  Warp roles:
//   warp 0      TMA: Q once, then K_j and V_j per key tile into a 3-deep ring
//   warp 1      TMEM owner; one lane issues S_j = Q K_j^T (M=128, N=128,
//               K=d, into one of two 128-column S buffers), and after the
//               softmax has written P_j, PV_j = P_j V_j (M=128, N=d, K=128,
//               V read MN-major) into one of two d-column buffers
//   warps 2..5  one query row per thread: masked online softmax on S_j read
//               from TMEM, P_j (bf16) written to shared memory in the
//               128B-swizzled K-major layout the MMA reads, O kept in
//               registers and updated as O = O * alpha_j + PV_j.
// S_{j+1} is issued before waiting for P_j, so the tensor core works on the
// next score tile while the softmax of the current one runs.
#include <cuda_bf16.h>

#include "cr_internal.h"
#include "cr_ptx.cuh"

namespace cr {
namespace {

template <int D>
struct AttnCfg {
    static constexpr uint32_t kRowBytes = D * 2;            // one K/V/Q row
    static constexpr uint32_t kAtomBytes = 8 * kRowBytes;    // swizzle atom (8 rows)
    static constexpr uint32_t kTileBytes = 128 * kRowBytes;
    static constexpr uint32_t kSwz = (D == 64) ? SWZ_128B : SWZ_64B;
    static constexpr int kStages = 3;
    static constexpr uint32_t kPBytes = 128 * 128 * 2;
    static constexpr uint32_t kQOff = 0;
    static constexpr uint32_t kKVOff = kTileBytes;                       // K then V per stage
    static constexpr uint32_t kPOff = kKVOff + kStages * 2 * kTileBytes;  // 2 P buffers
    static constexpr uint32_t kBarOff = kPOff + 2 * kPBytes;
    static constexpr uint32_t kSmemBytes = 1024 + kBarOff + 256;
    static constexpr uint32_t kTmemS = 0;      // two 128-column score buffers
    static constexpr uint32_t kTmemPV = 256;   // two D-column PV buffers
};

// Byte offset of 16 consecutive keys (c multiple of 16) of row r inside a
// [128 x 128] bf16 P tile held as two 64-column, 128B-swizzled K-major atoms.
__device__ __forceinline__ void p_offsets(int r, int c, uint32_t* o0, uint32_t* o1) {
    const uint32_t base = (c >> 6) * 16384 + r * 128;
    const int ch = (c & 63) >> 3;
    *o0 = base + ((ch ^ (r & 7)) << 4);
    *o1 = base + (((ch + 1) ^ (r & 7)) << 4);
}

template <int D>
__global__ void __launch_bounds__(192, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQKV, const __grid_constant__ AttnParams p) {
    using Cfg = AttnCfg<D>;
    constexpr int NS = Cfg::kStages;
    constexpr uint32_t IDESC_S = idesc_bf16(128, 128, false, false);
    constexpr uint32_t IDESC_PV = idesc_bf16(128, D, false, true);
    const float NEG_INF = -__int_as_float(0x7f800000);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg::kBarOff);
    uint64_t* q_full = bars;
    uint64_t* k_full = bars + 1;
    uint64_t* v_full = k_full + NS;
    uint64_t* kv_empty = v_full + NS;
    uint64_t* s_full = kv_empty + NS;
    uint64_t* p_full = s_full + 2;
    uint64_t* pv_full = p_full + 2;
    uint64_t* drain = pv_full + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    // ---- work item: heaviest (last) query tiles first
    const int head = blockIdx.x % p.n_heads;
    const int item = p.n_items - 1 - static_cast<int>(blockIdx.x / p.n_heads);
    int req = 0;
    while (req + 1 < p.n_req && p.tile_prefix[req + 1] <= item) ++req;
    const int q0 = (item - p.tile_prefix[req]) * 128;
    const int rs = p.req_start[req];
    const int len = p.req_start[req + 1] - rs;
    const int last = min(q0 + 127, len - 1);
    const int kv_extent = __ldg(p.chunk_end + rs + last);      // keys visible to the tile
    const int n_kv = (kv_extent + 127) / 128;

    const uint32_t warp = warp_id(), lane = lane_id();
    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&s_full[s], 1);
            mbar_init(&p_full[s], 128);
            mbar_init(&pv_full[s], 1);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx wc{abort_flag, p.status};

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch(&tmQKV);
            mbar_expect_tx(q_full, Cfg::kTileBytes);
            tma_load_2d(smem + Cfg::kQOff, &tmQKV, q_full, head * D, rs + q0);
            bool ok = true;
            for (int j = 0; j < n_kv; ++j) {
                const int st = j % NS;
                const uint32_t ph = static_cast<uint32_t>(j / NS) & 1u;
                if (!(ok = mbar_wait(&kv_empty[st], ph ^ 1u, wc, 121))) break;
                uint8_t* kt = smem + Cfg::kKVOff + st * 2 * Cfg::kTileBytes;
                mbar_expect_tx(&k_full[st], Cfg::kTileBytes);
                tma_load_2d(kt, &tmQKV, &k_full[st], p.d_b + head * D, rs + j * 128);
                mbar_expect_tx(&v_full[st], Cfg::kTileBytes);
                tma_load_2d(kt + Cfg::kTileBytes, &tmQKV, &v_full[st], 2 * p.d_b + head * D,
                            rs + j * 128);
            }
            if (!ok) {
                const uint64_t t0 = globaltimer();
                while (globaltimer() - t0 < 50000ull) {
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t sq = smem_u32(smem + Cfg::kQOff);
            auto issue_s = [&](int j) -> bool {
                const int st = j % NS;
                const uint32_t ph = static_cast<uint32_t>(j / NS) & 1u;
                if (!mbar_wait(&k_full[st], ph, wc, 222)) return false;
                tc_fence_after();
                const uint32_t sk = smem_u32(smem + Cfg::kKVOff + st * 2 * Cfg::kTileBytes);
                const uint32_t d = tmem_base + Cfg::kTmemS + (j & 1) * 128;
#pragma unroll
                for (int k = 0; k < D / 16; ++k)
                    mma_bf16_ss(d, smem_desc(sq + k * 32, 16, Cfg::kAtomBytes, Cfg::kSwz),
                                smem_desc(sk + k * 32, 16, Cfg::kAtomBytes, Cfg::kSwz), IDESC_S,
                                k != 0 ? 1u : 0u);
                mma_commit(&s_full[j & 1]);
                return true;
            };
            bool ok = mbar_wait(q_full, 0, wc, 221);
            if (ok) {
                tc_fence_after();
                ok = issue_s(0);
            }
            for (int j = 0; j < n_kv && ok; ++j) {
                if (j + 1 < n_kv && !(ok = issue_s(j + 1))) break;
                const int st = j % NS;
                const uint32_t ph = static_cast<uint32_t>(j / NS) & 1u;
                if (!(ok = mbar_wait(&p_full[j & 1], static_cast<uint32_t>(j >> 1) & 1u, wc, 223)))
                    break;
                if (!(ok = mbar_wait(&v_full[st], ph, wc, 224))) break;
                tc_fence_after();
                const uint32_t sp = smem_u32(smem + Cfg::kPOff + (j & 1) * Cfg::kPBytes);
                const uint32_t sv =
                    smem_u32(smem + Cfg::kKVOff + st * 2 * Cfg::kTileBytes + Cfg::kTileBytes);
                const uint32_t d = tmem_base + Cfg::kTmemPV + (j & 1) * D;
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint64_t da =
                        smem_desc(sp + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024, SWZ_128B);
                    // V: rows = keys (K dimension), D contiguous (MN-major);
                    // 16 keys = 2 swizzle atoms of 8 rows.
                    const uint64_t db = smem_desc(sv + kk * 16 * Cfg::kRowBytes, Cfg::kTileBytes,
                                                  Cfg::kAtomBytes, Cfg::kSwz);
                    mma_bf16_ss(d, da, db, IDESC_PV, kk != 0 ? 1u : 0u);
                }
                mma_commit(&pv_full[j & 1]);
                mma_commit(&kv_empty[st]);
            }
            mma_commit(drain);
            mbar_wait(drain, 0, wc, 225);
        }
    } else {
        // ---------------------------------------------------- softmax (warps 2..5)
        const uint32_t quad = warp & 3u;
        const int r = static_cast<int>(quad * 32 + lane);
        const int qrow = q0 + r;
        const bool valid = qrow < len;
        const int cend = valid ? __ldg(p.chunk_end + rs + qrow) : 1;
        const uint32_t lane_off = (quad * 32u) << 16;
        float m = NEG_INF, l = 0.0f;
        float o[D];
#pragma unroll
        for (int i = 0; i < D; ++i) o[i] = 0.0f;
        bool ok = true;
        for (int j = 0; j < n_kv; ++j) {
            ok = mbar_wait(&s_full[j & 1], static_cast<uint32_t>(j >> 1) & 1u, wc, 321);
            if (!__all_sync(0xffffffffu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const int k0 = j * 128;
            const uint32_t ts = tmem_base + lane_off + Cfg::kTmemS + (j & 1) * 128;
            // pass 1: row max of the scaled, masked scores
            float mx = NEG_INF;
            for (int c = 0; c < 128; c += 16) {
                float v[16];
                __syncwarp();
                tmem_ld16(ts + c, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    if (k0 + c + i < cend) mx = fmaxf(mx, v[i] * p.scale_log2);
            }
            const float m_new = fmaxf(m, mx);
            const float alpha = exp2f(m - m_new);
            // pass 2: probabilities -> P (bf16, swizzled K-major), row sum
            float rsum = 0.0f;
            uint8_t* pt = smem + Cfg::kPOff + (j & 1) * Cfg::kPBytes;
            for (int c = 0; c < 128; c += 16) {
                float v[16];
                __syncwarp();
                tmem_ld16(ts + c, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float e = (k0 + c + i < cend) ? exp2f(v[i] * p.scale_log2 - m_new) : 0.0f;
                    v[i] = e;
                    rsum += e;
                }
                uint32_t o0, o1;
                p_offsets(r, c, &o0, &o1);
                *reinterpret_cast<uint4*>(pt + o0) =
                    make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                               pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
                *reinterpret_cast<uint4*>(pt + o1) =
                    make_uint4(pack_bf16x2(v[8], v[9]), pack_bf16x2(v[10], v[11]),
                               pack_bf16x2(v[12], v[13]), pack_bf16x2(v[14], v[15]));
            }
            l = l * alpha + rsum;
            m = m_new;
            fence_async_smem();
            tc_fence_before();
            mbar_arrive(&p_full[j & 1]);
            ok = mbar_wait(&pv_full[j & 1], static_cast<uint32_t>(j >> 1) & 1u, wc, 322);
            if (!__all_sync(0xffffffffu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t tp = tmem_base + lane_off + Cfg::kTmemPV + (j & 1) * D;
#pragma unroll
            for (int c = 0; c < D; c += 16) {
                float v[16];
                __syncwarp();
                tmem_ld16(tp + c, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i) o[c + i] = fmaf(o[c + i], alpha, v[i]);
            }
        }
        tc_fence_before();
        if (ok && valid) {
            const float inv = 1.0f / l;
            uint16_t* dst = p.out + static_cast<int64_t>(rs + qrow) * p.d_b + head * D;
#pragma unroll
            for (int c = 0; c < D; c += 8) {
                *reinterpret_cast<uint4*>(dst + c) =
                    make_uint4(pack_bf16x2(o[c] * inv, o[c + 1] * inv),
                               pack_bf16x2(o[c + 2] * inv, o[c + 3] * inv),
                               pack_bf16x2(o[c + 4] * inv, o[c + 5] * inv),
                               pack_bf16x2(o[c + 6] * inv, o[c + 7] * inv));
            }
        }
    }
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, 512);
    }
}

template <int D>
cr_status launch_d(const CUtensorMap& tm, const AttnParams& p, cudaStream_t st) {
    using Cfg = AttnCfg<D>;
    auto kern = attn_kernel<D>;
    static unsigned long long attr_done = 0;   // one per template instantiation
    const cr_status sa = ensure_smem_attr(kern, static_cast<int>(Cfg::kSmemBytes), &attr_done);
    if (sa != CR_OK) return sa;
    const int grid = p.n_items * p.n_heads;
    kern<<<grid, 192, Cfg::kSmemBytes, st>>>(tm, p);
    return cuda_check(cudaGetLastError());
}

}  // namespace

cr_status launch_attention(const uint16_t* qkv, int64_t n_tokens, int head_dim,
                           const AttnParams& p, cudaStream_t st) {
    if (head_dim != 32 && head_dim != 64) return CR_ERR_UNSUPPORTED;
    if (p.n_items <= 0) return CR_OK;
    CUtensorMap tm;
    if (!make_tmap_2d(&tm, qkv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3ull * p.d_b, n_tokens,
                      3ull * p.d_b * 2, head_dim, 128,
                      head_dim == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B))
        return CR_ERR_INVALID_ARG;
    return head_dim == 64 ? launch_d<64>(tm, p, st) : launch_d<32>(tm, p, st);
}

}  // namespace cr
