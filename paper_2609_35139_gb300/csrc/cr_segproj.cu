// StaleEncoder stage 1 (Sec. 4.1): every one of the S = 2 L H_KV segments of
// a token has its own d_h -> d_seg linear, applied to the cache divided by
// sigma_stale.  Per token this reads D_KV cache values and does 2 D_KV d_seg
// flops, i.e. 16 flop/byte at d_seg = 16: the kernel is bound by HBM, and the
// tensor cores only have to keep up with the stream of cache tiles.
//
// Work item: 128 tokens x G = 16 consecutive segments.  Warp 0 streams, per
// segment, the [128 x d_h] cache slice (TMA, 128B swizzle) and the segment's
// [16 x d_h] weight rows through a ring of shared-memory stages.  The weights
// W_seg / sigma_stale come as two bf16 terms (hi + lo, folded once per call),
// so the folded weight carries about 16 significant bits, not 8; warp 1
// issues, per segment, one M=128, N=16 MMA chain over both terms into the
// segment's own 16 TMEM columns (two 256-column buffers).  The MMAs are idle
// most of the time either way: the doubled chain costs no time.  Warps 2..5
// add the bias and store d_seg values per segment, as bf16 (y) and, when
// asked, as the bf16 remainder y - bf16(y) too (y_lo), so that the next
// linear can take y to about 16 bits.  For d_seg = 8 the weight box still
// spans 16 rows (the next segment's rows, or TMA zero fill past the end);
// those 8 extra output columns are computed and discarded.
//
// Pool variant (kPool): the same projection reads its cache tiles straight
// from the chunk pool, each 128-row tile inside one selected chunk, and warp 6
// stores every tile it has loaded into the assembled cache (TMA store from the
// same shared-memory stage, or plain stores for a chunk's last, shorter tile).
// The assembly of Sec. 4.1 then costs one read and one write of the cache
// instead of two reads and a write.  Rows of a shorter tile past its chunk
// end are loaded (the pool's next rows, or zero fill) but neither projected
// into y nor stored.
#include <type_traits>
#include "cr_internal.h"
#include "cr_ptx.cuh"

namespace cr {
namespace {

constexpr int SP_G = 16;          // segments per work item
constexpr int SP_N = 16;          // MMA N (>= d_seg)

template <int DH>
struct SegCfg {
    static constexpr int kBoxes = DH / 64;                 // 64-column swizzle boxes per slice
    static constexpr uint32_t kABytes = 128 * DH * 2;
    static constexpr uint32_t kBBytes = SP_N * DH * 2;         // one weight term
    static constexpr uint32_t kStageBytes = kABytes + 2 * kBBytes;
    static constexpr int kStages = (DH == 128) ? 5 : 8;
    static constexpr uint32_t kSmemBytes = 1024 + kStages * kStageBytes + 256;
};

// W_seg / sigma_stale per input coordinate as two bf16 terms: out[i] = hi =
// rn(w / sigma), out[n + i] = lo = rn(w / sigma - hi); eight weights (16 bytes)
// per thread.  n and d_h are multiples of 8.
__global__ void fold_sigma_kernel(const uint16_t* __restrict__ w, const float* __restrict__ sigma,
                                  int64_t n, int d_seg, int dh, uint16_t* __restrict__ out) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t n8 = n >> 3;
    for (int64_t i8 = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i8 < n8;
         i8 += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t i = i8 << 3;
        const int64_t d = i % dh;
        const int64_t s = i / (static_cast<int64_t>(d_seg) * dh);
        const uint4 wv = __ldg(reinterpret_cast<const uint4*>(w) + i8);
        const float4* sp = reinterpret_cast<const float4*>(sigma + s * dh + d);
        const float4 s0 = __ldg(sp), s1 = __ldg(sp + 1);
        const uint32_t in[4] = {wv.x, wv.y, wv.z, wv.w};
        const float sg[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
        uint32_t oh[4], ol[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float a = __uint_as_float(in[k] << 16) / sg[2 * k];
            const float b = __uint_as_float(in[k] & 0xFFFF0000u) / sg[2 * k + 1];
            split_bf16x2(a, b, &oh[k], &ol[k]);
        }
        reinterpret_cast<uint4*>(out)[i8] = make_uint4(oh[0], oh[1], oh[2], oh[3]);
        reinterpret_cast<uint4*>(out + n)[i8] = make_uint4(ol[0], ol[1], ol[2], ol[3]);
    }
}

struct NoTiles {};

// Rows of M tile mt: its first source row, first output row and row count.
struct TileRows {
    int64_t src;
    int32_t dst;
    int32_t rows;
};
__device__ __forceinline__ TileRows tile_rows(const NoTiles&, const SegParams& p, int mt) {
    const int r0 = mt * 128;
    return TileRows{r0, r0, min(128, p.M - r0)};
}
__device__ __forceinline__ TileRows tile_rows(const SegTiles& tm, const SegParams&, int mt) {
    int lo = 0, hi = tm.n_seg - 1;   // last chunk whose first tile is <= mt
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (tm.tile_prefix[mid] <= mt)
            lo = mid;
        else
            hi = mid - 1;
    }
    const int k = (mt - tm.tile_prefix[lo]) * 128;
    return TileRows{tm.src_row[lo] + k, tm.dst_row[lo] + k, min(128, tm.len[lo] - k)};
}


template <int DH, bool kPool>
__global__ void __launch_bounds__(224, 1)
    segproj_kernel(const __grid_constant__ CUtensorMap tmKV, const __grid_constant__ CUtensorMap tmW,
                   const __grid_constant__ CUtensorMap tmOut, const __grid_constant__ SegParams p,
                   const __grid_constant__ std::conditional_t<kPool, SegTiles, NoTiles> tiles) {
    using Cfg = SegCfg<DH>;
    constexpr int STAGES = Cfg::kStages;
    constexpr uint32_t IDESC = idesc_bf16(128, SP_N, false, false);
    constexpr uint32_t TMEM_COLS = 512;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * Cfg::kStageBytes);
    uint64_t* full = bars;
    uint64_t* empty = bars + STAGES;
    uint64_t* tfull = bars + 2 * STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    const uint32_t warp = warp_id(), lane = lane_id();
    pdl_launch_dependents();
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kPool ? 2 : 1);   // the MMA's commit (+ the tile store)
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&tfull[s], 1);
            mbar_init(&tempty[s], 4);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    pdl_wait();   // the cache and the folded weights come from earlier kernels
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx wc{abort_flag, p.status};
    const int total = p.num_m * p.num_g;

    // Producer and MMA issuer run as converged warps; one elected lane issues.
    if (warp == 0) {
        if (elect_one()) {
            tma_prefetch(&tmKV);
            tma_prefetch(&tmW);
        }
        __syncwarp();
        uint32_t stage = 0, phase = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
            const int src0 = static_cast<int>(tile_rows(tiles, p, t % p.num_m).src);
            const int s0 = (t / p.num_m) * SP_G;
            const int ns = min(SP_G, p.S - s0);
            for (int g = 0; g < ns; ++g) {
                if (!(ok = mbar_wait_warp(&empty[stage], phase ^ 1u, wc, 111))) break;
                uint8_t* sa = smem + stage * Cfg::kStageBytes;
                uint8_t* sb = sa + Cfg::kABytes;
                const int seg = s0 + g;
                if (elect_one()) {
                    mbar_expect_tx(&full[stage], Cfg::kStageBytes);
#pragma unroll
                    for (int b = 0; b < Cfg::kBoxes; ++b) {
                        tma_load_2d(sa + b * 16384, &tmKV, &full[stage], seg * DH + b * 64, src0);
                        // hi term rows [0, S d_seg), lo term rows [S d_seg, 2 S d_seg)
                        tma_load_2d(sb + b * (SP_N * 128), &tmW, &full[stage], b * 64,
                                    seg * p.d_seg);
                        tma_load_2d(sb + Cfg::kBBytes + b * (SP_N * 128), &tmW, &full[stage], b * 64,
                                    (p.S + seg) * p.d_seg);
                    }
                }
                __syncwarp();
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
        }
        if (!ok) {
            const uint64_t t0 = globaltimer();
            while (globaltimer() - t0 < 50000ull) {
            }
        }
    } else if (warp == 1) {
        // a K=16 step adds 32 bytes (2 units of 16 B) to a descriptor's start
        const uint64_t da0 = smem_desc(smem_u32(smem), 16, 1024, SWZ_128B);
        constexpr uint64_t kStageStep = Cfg::kStageBytes >> 4;
        uint32_t stage = 0, phase = 0, acc = 0, acc_phase = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
            const int s0 = (t / p.num_m) * SP_G;
            const int ns = min(SP_G, p.S - s0);
            if (!(ok = mbar_wait_warp(&tempty[acc], acc_phase ^ 1u, wc, 211))) break;
            tc_fence_after();
            for (int g = 0; g < ns; ++g) {
                if (!(ok = mbar_wait_warp(&full[stage], phase, wc, 212))) break;
                tc_fence_after();
                const uint32_t d = tmem_base + acc * 256 + g * SP_N;
                const uint64_t da = da0 + stage * kStageStep;
                const uint64_t db = da + (Cfg::kABytes >> 4);
                if (elect_one()) {
#pragma unroll
                    for (int b = 0; b < Cfg::kBoxes; ++b) {
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint64_t a = da + b * (16384 >> 4) + 2 * k;
                            const uint64_t w = db + b * ((SP_N * 128) >> 4) + 2 * k;
                            mma_bf16_ss(d, a, w, IDESC, (b | k) != 0 ? 1u : 0u);
                            mma_bf16_ss(d, a, w + (Cfg::kBBytes >> 4), IDESC, 1u);
                        }
                    }
                    mma_commit(&empty[stage]);
                }
                __syncwarp();
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            if (elect_one()) mma_commit(&tfull[acc]);
            __syncwarp();
            acc ^= 1u;
            if (acc == 0) acc_phase ^= 1u;
        }
        if (elect_one()) mma_commit(drain);
        __syncwarp();
        mbar_wait_warp(drain, 0, wc, 213);
    } else if (warp == 6) {
        if constexpr (kPool) {
            // tile store: a whole tile goes out by TMA from the stage it was
            // loaded into, and the stage is released once the store has read
            // it (two younger stores stay in flight: q0, q1 are the stages whose
            // stores may still be reading, oldest first); a chunk's shorter
            // last tile is copied row by row with plain stores
            uint32_t stage = 0, phase = 0, q0 = 0, q1 = 0;
            int npend = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
                const TileRows tr = tile_rows(tiles, p, t % p.num_m);
                const int s0 = (t / p.num_m) * SP_G;
                const int ns = min(SP_G, p.S - s0);
                for (int g = 0; g < ns; ++g) {
                    if (!(ok = mbar_wait_warp(&full[stage], phase, wc, 114))) break;
                    const uint8_t* sa = smem + stage * Cfg::kStageBytes;
                    const int col = (s0 + g) * DH;
                    if (!p.kv_out) {
                        // no assembled cache asked for: the projection alone reads the stage
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&empty[stage]);
                    } else if (tr.rows == 128) {
                        if (lane == 0) {
                            fence_async_smem();
#pragma unroll
                            for (int b = 0; b < Cfg::kBoxes; ++b)
                                tma_store_2d(&tmOut, sa + b * 16384, col + b * 64, tr.dst);
                            tma_store_commit();
                        }
                        if (npend == 2) {
                            // q0's store is done reading once at most two groups remain
                            if (lane == 0) tma_store_wait_read<2>();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(&empty[q0]);
                            q0 = q1;
                            q1 = stage;
                        } else if (npend == 1) {
                            q1 = stage;
                            npend = 2;
                        } else {
                            q0 = stage;
                            npend = 1;
                        }
                    } else {
                        // release the held stages first: a held stage may be at most
                        // two uses old, or the producer, which refills in ring order,
                        // would wait for it while this warp waits for the producer
                        if (npend > 0) {
                            if (lane == 0) tma_store_wait_read<0>();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(&empty[q0]);
                            if (lane == 0 && npend > 1) mbar_arrive(&empty[q1]);
                            npend = 0;
                        }
                        // 16-byte chunk c of row r sits at r*128 + ((c ^ (r & 7)) << 4)
                        // in each 128B-swizzled box of 64 columns
                        const int n16 = tr.rows * 8;
                        for (int b = 0; b < Cfg::kBoxes; ++b) {
                            for (int i = static_cast<int>(lane); i < n16; i += 32) {
                                const int r = i >> 3, c = i & 7;
                                const uint4 v = *reinterpret_cast<const uint4*>(
                                    sa + b * 16384 + r * 128 + ((c ^ (r & 7)) << 4));
                                *reinterpret_cast<uint4*>(p.kv_out + static_cast<int64_t>(tr.dst + r) * p.ld_out +
                                                          col + b * 64 + c * 8) = v;
                            }
                        }
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&empty[stage]);
                    }
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            // every store has finished reading (and, before exit, writing)
            if (lane == 0) tma_store_wait_read<0>();
            __syncwarp();
            if (lane == 0 && npend > 0) mbar_arrive(&empty[q0]);
            if (lane == 0 && npend > 1) mbar_arrive(&empty[q1]);
            if (lane == 0) tma_store_wait0();
            __syncwarp();
        }
    } else {
        const uint32_t quad = warp & 3u;
        const int r = static_cast<int>(quad * 32 + lane);
        const int64_t ldy = p.ldy;
        uint32_t acc = 0, acc_phase = 0;
        for (int t = blockIdx.x; t < total; t += gridDim.x) {
            const TileRows tr = tile_rows(tiles, p, t % p.num_m);
            const int s0 = (t / p.num_m) * SP_G;
            const int ns = min(SP_G, p.S - s0);
            const bool ok = mbar_wait(&tfull[acc], acc_phase, wc, 311);
            if (!__all_sync(0xffffffffu, ok)) break;
            tc_fence_after();
            const int row = tr.dst + r;
            const uint32_t taddr = tmem_base + ((quad * 32u) << 16) + acc * 256;
            uint16_t* yrow = p.y + static_cast<int64_t>(row) * ldy;
            uint16_t* ylrow = p.y_lo ? p.y_lo + static_cast<int64_t>(row) * ldy : nullptr;
            for (int g = 0; g < ns; ++g) {
                float v[16];
                __syncwarp();
                tmem_ld16(taddr + g * SP_N, v);
                tmem_wait_ld();
                const int seg = s0 + g;
                const float* bs = p.b_seg + seg * p.d_seg;
                if (r < tr.rows) {
                    uint32_t w[8], wl[8];
                    const int dm = p.d_seg - 1;   // d_seg is 8 or 16; columns >= d_seg are dropped
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        split_bf16x2(v[2 * i] + __ldg(bs + ((2 * i) & dm)),
                                     v[2 * i + 1] + __ldg(bs + ((2 * i + 1) & dm)), &w[i], &wl[i]);
                    uint4* dst = reinterpret_cast<uint4*>(yrow + seg * p.d_seg);
                    dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
                    if (p.d_seg == 16) dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
                    if (ylrow) {
                        uint4* dl = reinterpret_cast<uint4*>(ylrow + seg * p.d_seg);
                        dl[0] = make_uint4(wl[0], wl[1], wl[2], wl[3]);
                        if (p.d_seg == 16) dl[1] = make_uint4(wl[4], wl[5], wl[6], wl[7]);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
            acc ^= 1u;
            if (acc == 0) acc_phase ^= 1u;
        }
    }
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, TMEM_COLS);
    }
}

template <int DH, bool kPool, class Tiles>
cr_status launch_dh(const CUtensorMap& tk, const CUtensorMap& tw, const CUtensorMap& to,
                    const SegParams& p, const Tiles& tiles, cudaStream_t st) {
    using Cfg = SegCfg<DH>;
    auto kern = segproj_kernel<DH, kPool>;
    static unsigned long long attr_done = 0;   // one per template instantiation
    const cr_status sa = ensure_smem_attr(kern, static_cast<int>(Cfg::kSmemBytes), &attr_done);
    if (sa != CR_OK) return sa;
    const int items = p.num_m * p.num_g;
    const int grid = items < num_sms() ? items : num_sms();
    return launch_pdl(kern, dim3(grid), dim3(kPool ? 224 : 192), Cfg::kSmemBytes, st, tk, tw, to, p,
                      tiles);
}

}  // namespace

cr_status launch_fold_sigma(const uint16_t* w_seg, const float* sigma, int S, int d_seg,
                            int head_dim, uint16_t* wfold, cudaStream_t st) {
    const int64_t n = static_cast<int64_t>(S) * d_seg * head_dim;
    const int threads = 256;
    int64_t blocks = (n / 8 + threads - 1) / threads;
    if (blocks > 4 * 1024) blocks = 4 * 1024;
    return launch_pdl(fold_sigma_kernel, dim3(static_cast<unsigned>(blocks)), dim3(threads), 0, st,
                      w_seg, sigma, n, d_seg, head_dim, wfold);
}

cr_status launch_segproj(const uint16_t* kv, int64_t ld_kv, const uint16_t* wfold, int head_dim,
                         SegParams p, cudaStream_t st) {
    if (head_dim != 64 && head_dim != 128) return CR_ERR_UNSUPPORTED;
    if (p.d_seg != 8 && p.d_seg != 16) return CR_ERR_UNSUPPORTED;
    p.num_m = (p.M + 127) / 128;
    p.num_g = (p.S + SP_G - 1) / SP_G;
    CUtensorMap tk, tw;
    const uint64_t dkv = static_cast<uint64_t>(p.S) * head_dim;
    if (!make_tmap_2d(&tk, kv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dkv, p.M, ld_kv * 2, 64, 128,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    if (!make_tmap_2d(&tw, wfold, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, head_dim,
                      2 * static_cast<uint64_t>(p.S) * p.d_seg, head_dim * 2, 64, SP_N,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    const NoTiles none{};
    return head_dim == 128 ? launch_dh<128, false>(tk, tw, tk, p, none, st)
                           : launch_dh<64, false>(tk, tw, tk, p, none, st);
}

cr_status launch_segproj_pool(const uint16_t* kv_pool, int64_t n_pool_tokens, uint16_t* kv_out,
                              const uint16_t* wfold, int head_dim, SegParams p,
                              const SegTiles& tiles, cudaStream_t st) {
    if (head_dim != 64 && head_dim != 128) return CR_ERR_UNSUPPORTED;
    if (p.d_seg != 8 && p.d_seg != 16) return CR_ERR_UNSUPPORTED;
    if (tiles.n_seg < 1 || tiles.n_seg > kMaxSegs || n_pool_tokens > INT32_MAX) return CR_ERR_INVALID_ARG;
    p.num_m = tiles.tile_prefix[tiles.n_seg];
    p.num_g = (p.S + SP_G - 1) / SP_G;
    const uint64_t dkv = static_cast<uint64_t>(p.S) * head_dim;
    p.kv_out = kv_out;
    p.ld_out = static_cast<int64_t>(dkv);
    CUtensorMap tk, tw, to;
    if (!make_tmap_2d(&tk, kv_pool, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, dkv, n_pool_tokens, dkv * 2, 64,
                      128, CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    if (!make_tmap_2d(&tw, wfold, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, head_dim,
                      2 * static_cast<uint64_t>(p.S) * p.d_seg, head_dim * 2, 64, SP_N,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    // without an assembled cache the output map is never used (the pool's stands in)
    if (!make_tmap_2d(&to, kv_out ? static_cast<const void*>(kv_out) : kv_pool, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                      dkv, kv_out ? static_cast<uint64_t>(p.M) : static_cast<uint64_t>(n_pool_tokens), dkv * 2,
                      64, 128, CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    return head_dim == 128 ? launch_dh<128, true>(tk, tw, to, p, tiles, st)
                           : launch_dh<64, true>(tk, tw, to, p, tiles, st);
}

}  // namespace cr
