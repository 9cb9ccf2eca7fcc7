// Chunk-block-causal attention of the Repair Blocks (Sec. 4.1):
//   o_i = sum_{j : c(j) <= c(i)} softmax_j(q_i . k_j / sqrt(d)) v_j
// inside each request.  Chunk ids are non-decreasing along a request, so the
// keys visible to query i are exactly j < chunk_end[i]: a prefix.  A query
// tile therefore needs key tiles 0 .. ceil(max_i chunk_end / 128) - 1 and
// nothing past that; those tiles are never loaded or multiplied.  Rows whose
// chunk ends inside a key tile mask the rest of it; fully visible tiles do no
// masking work at all.
//
// CTA = (request, head, two consecutive 128-query tiles).  10 warps:
//   warp 0      TMA: both Q tiles once, then K_j and V_j per key tile into a
//               5-deep ring shared by the two query tiles
//   warp 1      TMEM owner; one lane issues, per key tile j and query tile w,
//               S_w,j = Q_w K_j^T (M=128, N=128, K=d) into S_w, and, once
//               softmax w has written P_w,j, O_w += P_w,j V_j (M=128, N=d,
//               K=128, V read MN-major) accumulating in TMEM
//   warps 2..5  softmax group 0 (query tile 0), one row per thread
//   warps 6..9  softmax group 1 (query tile 1)
// The two groups ping-pong on the tensor core.  Per key tile a group reads its
// S row from TMEM twice, 64 columns at a time (the (masked) row max, then the
// exponentials; 320 threads leave 168 registers each), and writes
// P = 2^(s*scale*log2e - m) as bf16 pairs into its own TMEM columns, from
// where the PV MMA reads it as the A operand (TMEM holds S_0, S_1, O_0, O_1,
// P_0, P_1: 512 columns).  The reference m is the row's running max,
// updated lazily: only when a tile raises it by more than 2^8 does the group
// rescale its O row in TMEM (and the row sum l).  Any reference m gives the same
// softmax (it cancels in O / l), and keeping it at most 8 below the true
// running max keeps P <= 2^8, so this is exact up to rounding.
// O_w is read back and divided by l after the last tile.
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
    static constexpr int kStages = 5;
    static constexpr uint32_t kQOff = 0;                                  // Q0, Q1
    static constexpr uint32_t kKVOff = 2 * kTileBytes;                    // K, V per stage
    static constexpr uint32_t kBarOff = kKVOff + kStages * 2 * kTileBytes;
    static constexpr uint32_t kSmemBytes = 1024 + kBarOff + 256;
    static constexpr uint32_t kTmemS = 0;      // S_w at w * 128 (fp32)
    static constexpr uint32_t kTmemO = 256;    // O_w at 256 + w * D (fp32)
    static constexpr uint32_t kTmemP = 384;    // P_w at 384 + w * 64 (bf16 pairs)
};

constexpr int kThreads = 320;
constexpr float kRescaleLog2 = 8.0f;   // lazy-rescale threshold (log2 units)

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
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
    uint64_t* s_full = kv_empty + NS;     // [2]
    uint64_t* p_full = s_full + 2;        // [2]
    uint64_t* o_done = p_full + 2;        // [2]
    uint64_t* drain = o_done + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    // ---- work item: (request, pair of query tiles, head); heaviest pairs first
    const int head = blockIdx.x % p.n_heads;
    const int item = p.n_items - 1 - static_cast<int>(blockIdx.x / p.n_heads);
    int req = 0;
    while (req + 1 < p.n_req && p.tile_prefix[req + 1] <= item) ++req;
    const int q0 = (item - p.tile_prefix[req]) * 256;
    const int rs = p.req_start[req];
    const int len = p.req_start[req + 1] - rs;
    int n_kv[2];
#pragma unroll
    for (int w = 0; w < 2; ++w) {
        const int first = q0 + 128 * w;
        n_kv[w] = first < len ? (__ldg(p.chunk_end + rs + min(first + 127, len - 1)) + 127) / 128 : 0;
    }
    const int n_max = max(n_kv[0], n_kv[1]);

    const uint32_t warp = warp_id(), lane = lane_id();
    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
        for (int w = 0; w < 2; ++w) {
            mbar_init(&s_full[w], 1);
            mbar_init(&p_full[w], 128);
            mbar_init(&o_done[w], 1);
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
            // ---------------------------------------------------- TMA producer
            tma_prefetch(&tmQKV);
            mbar_expect_tx(q_full, 2 * Cfg::kTileBytes);
            tma_load_2d(smem + Cfg::kQOff, &tmQKV, q_full, head * D, rs + q0);
            tma_load_2d(smem + Cfg::kQOff + Cfg::kTileBytes, &tmQKV, q_full, head * D,
                        rs + q0 + 128);
            bool ok = true;
            for (int j = 0; j < n_max; ++j) {
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
            // ---------------------------------------------------- MMA issuer
            // Per query tile w the order is S_0, [P_0] PV_0, S_1, [P_1] PV_1, ...
            // so the commit after S_j+1 also covers PV_j: when the softmax group
            // sees S_j+1 its O row is current and its P buffer is free.
            const uint32_t sq0 = smem_u32(smem + Cfg::kQOff);
            auto issue_s = [&](int w, int j) -> bool {
                const int st = j % NS;
                if (!mbar_wait(&k_full[st], static_cast<uint32_t>(j / NS) & 1u, wc, 222)) return false;
                tc_fence_after();
                const uint32_t sq = sq0 + w * Cfg::kTileBytes;
                const uint32_t sk = smem_u32(smem + Cfg::kKVOff + st * 2 * Cfg::kTileBytes);
                const uint32_t d = tmem_base + Cfg::kTmemS + w * 128;
#pragma unroll
                for (int k = 0; k < D / 16; ++k)
                    mma_bf16_ss(d, smem_desc(sq + k * 32, 16, Cfg::kAtomBytes, Cfg::kSwz),
                                smem_desc(sk + k * 32, 16, Cfg::kAtomBytes, Cfg::kSwz), IDESC_S,
                                k != 0 ? 1u : 0u);
                mma_commit(&s_full[w]);
                return true;
            };
            auto issue_pv = [&](int w, int j) -> bool {
                const int st = j % NS;
                if (!mbar_wait(&p_full[w], static_cast<uint32_t>(j) & 1u, wc, 224)) return false;
                if (!mbar_wait(&v_full[st], static_cast<uint32_t>(j / NS) & 1u, wc, 225)) return false;
                tc_fence_after();
                const uint32_t sv =
                    smem_u32(smem + Cfg::kKVOff + st * 2 * Cfg::kTileBytes + Cfg::kTileBytes);
                const uint32_t d = tmem_base + Cfg::kTmemO + w * D;
                const uint32_t pa = tmem_base + Cfg::kTmemP + w * 64;
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    // P from TMEM (16 keys = 8 columns); V: rows = keys (the K
                    // dimension), d contiguous (MN-major); 16 keys = two 8-row atoms.
                    const uint64_t db = smem_desc(sv + kk * 16 * Cfg::kRowBytes, Cfg::kTileBytes,
                                                  Cfg::kAtomBytes, Cfg::kSwz);
                    mma_bf16_ts(d, pa + kk * 8, db, IDESC_PV, (j > 0 || kk != 0) ? 1u : 0u);
                }
                return true;
            };
            bool ok = mbar_wait(q_full, 0, wc, 221);
            if (ok) tc_fence_after();
            for (int w = 0; w < 2 && ok; ++w)
                if (n_kv[w] > 0) ok = issue_s(w, 0);
            for (int j = 0; j < n_max && ok; ++j) {
                for (int w = 0; w < 2 && ok; ++w) {
                    if (j >= n_kv[w]) continue;
                    if (!(ok = issue_pv(w, j))) break;
                    if (j + 1 < n_kv[w])
                        ok = issue_s(w, j + 1);
                    else
                        mma_commit(&o_done[w]);
                }
                if (ok) mma_commit(&kv_empty[j % NS]);
            }
            mma_commit(drain);
            mbar_wait(drain, 0, wc, 227);
        }
    } else {
        // ---------------------------------------------------- softmax groups
        const int w = (warp >= 6) ? 1 : 0;
        const uint32_t quad = warp & 3u;
        const int r = static_cast<int>(quad * 32 + lane);
        const int qrow = q0 + 128 * w + r;
        const bool valid = qrow < len;
        const int cend = valid ? __ldg(p.chunk_end + rs + qrow) : 1;
        const uint32_t lane_off = (quad * 32u) << 16;
        const uint32_t ts = tmem_base + lane_off + Cfg::kTmemS + w * 128;
        const uint32_t to = tmem_base + lane_off + Cfg::kTmemO + w * D;
        const float sc = p.scale_log2;
        const int n = n_kv[w];
        const uint32_t tp = tmem_base + lane_off + Cfg::kTmemP + w * 64;
        float m = NEG_INF, l = 0.0f;

        bool ok = true;
        for (int j = 0; j < n; ++j) {
            ok = mbar_wait(&s_full[w], static_cast<uint32_t>(j) & 1u, wc, 321);
            if (!__all_sync(0xffffffffu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const int k0 = j * 128;
            const bool full_tile = k0 + 128 <= cend;     // all 128 keys visible to this row
            // pass 1: row max of the (masked) scores, 64 columns at a time, in
            // eight independent chains
            float mxv[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) mxv[q] = NEG_INF;
#pragma unroll
            for (int h = 0; h < 128; h += 64) {
                float s[64];
                __syncwarp();
                tmem_ld32(ts + h, s);
                tmem_ld32(ts + h + 32, s + 32);
                tmem_wait_ld();
                if (full_tile) {
#pragma unroll
                    for (int i = 0; i < 64; ++i) mxv[i & 7] = fmaxf(mxv[i & 7], s[i]);
                } else {
#pragma unroll
                    for (int i = 0; i < 64; ++i)
                        if (k0 + h + i < cend) mxv[i & 7] = fmaxf(mxv[i & 7], s[i]);
                }
            }
            float mx = fmaxf(fmaxf(fmaxf(mxv[0], mxv[1]), fmaxf(mxv[2], mxv[3])),
                             fmaxf(fmaxf(mxv[4], mxv[5]), fmaxf(mxv[6], mxv[7])));
            mx *= sc;
            // lazily move the reference max: on the first tile, or when this
            // tile would push P above 2^8 somewhere in the warp
            const bool raise = (j == 0) || (mx > m + kRescaleLog2);
            if (__any_sync(0xffffffffu, raise)) {
                const float m_new = fmaxf(m, mx);
                if (j > 0) {
                    // O holds sum_{k<j} P_k V_k (complete: S_j was issued after PV_{j-1})
                    const float alpha = ex2(m - m_new);
#pragma unroll
                    for (int c = 0; c < D; c += 16) {
                        float o[16];
                        tmem_ld16(to + c, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 16; ++i) o[i] *= alpha;
                        tmem_st16(to + c, o);
                    }
                    tmem_wait_st();
                    l *= alpha;
                }
                m = m_new;
            }
            // pass 2: P = 2^(s*sc - m) -> bf16, swizzled K-major, and the row sum.
            // Fully visible tiles (all tiles of chunk-aligned maps) take a loop
            // with no per-element masking.
            float rs8[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) rs8[q] = 0.0f;
            const int lim = full_tile ? 128 : cend - k0;   // keys < lim are visible
#pragma unroll
            for (int h = 0; h < 128; h += 64) {
                float s[64];
                __syncwarp();
                tmem_ld32(ts + h, s);
                tmem_ld32(ts + h + 32, s + 32);
                tmem_wait_ld();
                if (!full_tile) {
#pragma unroll
                    for (int i = 0; i < 64; ++i) s[i] = (h + i < lim) ? s[i] : NEG_INF;
                }
                uint32_t pk[32];
#pragma unroll
                for (int i = 0; i < 64; i += 2) {
                    const float e0 = ex2(fmaf(s[i], sc, -m));
                    const float e1 = ex2(fmaf(s[i + 1], sc, -m));
                    rs8[(i >> 1) & 7] += e0 + e1;
                    pk[i >> 1] = pack_bf16x2(e0, e1);
                }
                tmem_st32u(tp + h / 2, pk);
            }
            l += ((rs8[0] + rs8[1]) + (rs8[2] + rs8[3])) + ((rs8[4] + rs8[5]) + (rs8[6] + rs8[7]));
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(&p_full[w]);
        }
        if (ok && n > 0) {
            ok = mbar_wait(&o_done[w], 0, wc, 322);
            ok = __all_sync(0xffffffffu, ok);
        }
        if (ok && n > 0) {
            tc_fence_after();
            const float inv = 1.0f / l;
            uint16_t* dst = p.out + static_cast<int64_t>(rs + qrow) * p.d_b + head * D;
#pragma unroll
            for (int c = 0; c < D; c += 16) {
                float o[16];
                tmem_ld16(to + c, o);
                tmem_wait_ld();
                if (valid) {
                    uint4* d4 = reinterpret_cast<uint4*>(dst + c);
                    d4[0] = make_uint4(pack_bf16x2(o[0] * inv, o[1] * inv), pack_bf16x2(o[2] * inv, o[3] * inv),
                                       pack_bf16x2(o[4] * inv, o[5] * inv), pack_bf16x2(o[6] * inv, o[7] * inv));
                    d4[1] = make_uint4(pack_bf16x2(o[8] * inv, o[9] * inv),
                                       pack_bf16x2(o[10] * inv, o[11] * inv),
                                       pack_bf16x2(o[12] * inv, o[13] * inv),
                                       pack_bf16x2(o[14] * inv, o[15] * inv));
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

template <int D>
cr_status launch_d(const CUtensorMap& tm, const AttnParams& p, cudaStream_t st) {
    using Cfg = AttnCfg<D>;
    auto kern = attn_kernel<D>;
    static unsigned long long attr_done = 0;   // one per template instantiation
    const cr_status sa = ensure_smem_attr(kern, static_cast<int>(Cfg::kSmemBytes), &attr_done);
    if (sa != CR_OK) return sa;
    const int grid = p.n_items * p.n_heads;
    kern<<<grid, kThreads, Cfg::kSmemBytes, st>>>(tm, p);
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
