// Chunk-block-causal attention of the Repair Blocks (Sec. 4.1):
//   o_i = sum_{j : c(j) <= c(i)} softmax_j(q_i . k_j / sqrt(d)) v_j
// inside each request.  Chunk ids are non-decreasing along a request, so the
// keys visible to query i are exactly j < chunk_end[i]: a prefix.  The
// attention-topology ablations of App. F keep that shape: with A1 (token-
// causal) the keys are j <= i, with A2 (bidirectional) the whole request, with
// A3 (block-diagonal) j in [chunk_start[i], chunk_end[i]).  In every mode the
// visible keys of row i are one interval [lo(i), hi(i)) whose ends never
// decrease with i, so a query tile needs key tiles
// floor(lo(first row) / 128) .. ceil(hi(last row) / 128) - 1 and nothing
// else; other tiles are never loaded or multiplied.  Rows whose interval ends
// inside a key tile mask the rest of it; fully visible tiles do no masking
// work at all.
//
// CTA = (request, head, two consecutive 128-query tiles w = 0, 1); three
// warpgroups, the first of which gives registers to the other two:
//   warp 0      TMA: both Q tiles once, then K_j and V_j per key tile into a
//               5-deep ring shared by the two query tiles
//   warp 1 + w  MMA issue for query tile w (warp 1 also owns TMEM): per key
//               tile j, S_w,j+1 = Q_w K_j+1^T (M=128, N=128, K=d) as soon as
//               softmax w has read S_w,j into registers, and O_w += P_w,j V_j
//               (M=128, N=d, K=128, P read from TMEM, V MN-major from smem)
//               once softmax w has written P_w,j.  Issue runs in a converged
//               warp with one elected lane, and each query tile has its own
//               issuer: the small MMAs of a d <= 64 head are cheap enough that
//               issue and barrier latency, not the tensor core, set the pace.
//   warps 4..7  softmax group 0 (query tile 0), one row per thread
//   warps 8..11 softmax group 1 (query tile 1)
// Per key tile a softmax thread loads its whole S row (128 fp32) from TMEM in
// one round trip, masks and takes the row max in registers, and writes
// P = 2^(s*scale*log2e - m) as bf16 pairs into its group's TMEM columns, from
// where the PV MMA reads it as the A operand (TMEM holds S_0, S_1, O_0, O_1,
// P_0, P_1: 512 columns).  The two groups overlap each other's exponentials
// with their MMAs.  The reference m is the row's running max, updated
// lazily: only when a tile raises it by more than 2^8 does the group rescale
// its O row in TMEM (and the row sum l).  Any reference m gives the same
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
    static constexpr uint32_t kSmemBytes = 1024 + kBarOff + 320;
    static constexpr uint32_t kTmemS = 0;      // S_w at w * 128 (fp32)
    static constexpr uint32_t kTmemO = 256;    // O_w at 256 + w * D (fp32)
    static constexpr uint32_t kTmemP = 384;    // P_w at 384 + w * 64 (bf16 pairs)
};

// Three warpgroups: control (TMA, two MMA issuers, one idle warp) and two
// softmax groups.
// At launch each thread gets 65536 / 384 = 168 registers (the host checks
// this); the control warpgroup gives up most of its share so that the softmax
// threads can hold a whole S row: 48 * 128 + 2 * 224 * 128 <= 168 * 384 (the
// control warps keep only descriptors, counters and phases).
constexpr int kThreads = 384;
constexpr uint32_t kRegsLaunch = 168;
constexpr uint32_t kRegsCtl = 48;
constexpr uint32_t kRegsSoftmax = 224;
static_assert(kRegsCtl * 128 + 2 * kRegsSoftmax * 128 <= kRegsLaunch * kThreads,
              "register split exceeds the launch allocation");
constexpr float kRescaleLog2 = 8.0f;   // lazy-rescale threshold (log2 units)
// Warp q of softmax group 0 and warp q of group 1 share an SM sub-partition
// (warps 4 + q and 8 + q) and take turns on the exponentials: while one runs
// its exp pass, the other waits for its S and PV MMAs, loads S and takes the
// row max, so the special-function unit stays busy.
constexpr bool kTurns = true;

// Exclusive end and start of the visible keys of request-local row i.
__device__ __forceinline__ int key_hi(const AttnParams& p, int rs, int len, int i) {
    if (p.mask_mode == CR_MASK_TOKEN_CAUSAL) return i + 1;
    if (p.mask_mode == CR_MASK_BIDIRECTIONAL) return len;
    return __ldg(p.chunk_end + rs + i);
}
__device__ __forceinline__ int key_lo(const AttnParams& p, int rs, int i) {
    return p.mask_mode == CR_MASK_BLOCK_DIAGONAL ? __ldg(p.chunk_start + rs + i) : 0;
}

// kLse: also write each row's log-sum-exp (for the training step's backward);
// the inference forward's instantiation has none of that code.
template <int D, bool kLse>
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
    uint64_t* kv_full = bars + 1;
    uint64_t* kv_empty = kv_full + NS;
    uint64_t* s_full = kv_empty + NS;     // [2] S_w,j in TMEM
    uint64_t* s_free = s_full + 2;        // [2] S_w,j read into registers
    uint64_t* p_full = s_free + 2;        // [2][2] half h of P_w,j (64 keys) in TMEM
    uint64_t* pv_done = p_full + 4;       // [2] O_w += P_w,j V_j complete
    uint64_t* drain = pv_done + 2;        // [2]
    uint64_t* turn = drain + 2;           // [2][4]: warp q of group w finished an exp pass
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(turn + 8);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    // ---- work item: (request, pair of query tiles, head); heaviest pairs first
    const int head = blockIdx.x % p.n_heads;
    const int item = p.n_items - 1 - static_cast<int>(blockIdx.x / p.n_heads);
    int req = 0;
    while (req + 1 < p.n_req && p.tile_prefix[req + 1] <= item) ++req;
    const int q0 = (item - p.tile_prefix[req]) * 256;
    const int rs = p.req_start[req];
    const int len = p.req_start[req + 1] - rs;

    const uint32_t warp = warp_id(), lane = lane_id();
    pdl_launch_dependents();
    if (threadIdx.x == 0) {
        mbar_init(q_full, 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 2);   // both issuers release each stage
        }
        for (int w = 0; w < 2; ++w) {
            mbar_init(&s_full[w], 1);
            mbar_init(&s_free[w], 4);
            mbar_init(&p_full[2 * w], 4);
            mbar_init(&p_full[2 * w + 1], 4);
            mbar_init(&pv_done[w], 1);
            mbar_init(&drain[w], 1);
        }
        for (int t = 0; t < 8; ++t) mbar_init(&turn[t], 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    pdl_wait();   // qkv and the chunk map come from earlier kernels
    // Both query tiles start at the key tile of the pair's first visible key,
    // kbase = 128 * floor(lo(q0) / 128): every issuer and softmax group then
    // takes the ring's tiles in order from its first slot use, which keeps
    // each parity wait within one phase of its barrier.  (Under the
    // block-diagonal mask the second tile's rows may start later; their
    // leading key tiles are fully masked and contribute exact zeros.)  Tile j
    // below is key tile kbase / 128 + j; query tile w needs j in [0, n_kv[w]),
    // an empty second tile (past the request's end) none.
    const int kbase = key_lo(p, rs, q0) & ~127;
    int n_kv[2];
#pragma unroll
    for (int w = 0; w < 2; ++w) {
        const int first = q0 + 128 * w;
        n_kv[w] = first < len ? (key_hi(p, rs, len, min(first + 127, len - 1)) - kbase + 127) / 128 : 0;
    }
    const int n_max = max(n_kv[0], n_kv[1]);
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx wc{abort_flag, p.status};

    if (warp < 4) {
        setmaxnreg_dec<kRegsCtl>();
        if (warp == 0) {
            // ---------------------------------------------------- TMA producer
            // (the whole warp runs the loop; one elected lane issues)
            if (elect_one()) {
                tma_prefetch(&tmQKV);
                mbar_expect_tx(q_full, 2 * Cfg::kTileBytes);
                tma_load_2d(smem + Cfg::kQOff, &tmQKV, q_full, head * D, rs + q0);
                tma_load_2d(smem + Cfg::kQOff + Cfg::kTileBytes, &tmQKV, q_full, head * D,
                            rs + q0 + 128);
            }
            __syncwarp();
            bool ok = true;
            for (int j = 0; j < n_max; ++j) {
                const int st = j % NS;
                const uint32_t ph = static_cast<uint32_t>(j / NS) & 1u;
                if (!(ok = mbar_wait_warp(&kv_empty[st], ph ^ 1u, wc, 121))) break;
                uint8_t* kt = smem + Cfg::kKVOff + st * 2 * Cfg::kTileBytes;
                if (elect_one()) {
                    mbar_expect_tx(&kv_full[st], 2 * Cfg::kTileBytes);
                    tma_load_2d(kt, &tmQKV, &kv_full[st], p.d_b + head * D, rs + kbase + j * 128);
                    tma_load_2d(kt + Cfg::kTileBytes, &tmQKV, &kv_full[st], 2 * p.d_b + head * D,
                                rs + kbase + j * 128);
                    // the stage is free once both issuers release it; an issuer
                    // whose query tile ends before tile j is released for here
                    // (its partner's release, after its MMAs, completes the phase)
                    if (j >= n_kv[0]) mbar_arrive(&kv_empty[st]);
                    if (j >= n_kv[1]) mbar_arrive(&kv_empty[st]);
                }
                __syncwarp();
            }
            if (!ok) {
                const uint64_t t0 = globaltimer();
                while (globaltimer() - t0 < 50000ull) {
                }
            }
        } else if (warp == 1 || warp == 2) {
            // ---------------------------------------------------- MMA issuers
            // Warp 1 + w issues for query tile w: per key tile j, S_w,j+1 as
            // soon as softmax w has read S_w,j out of TMEM, then O_w += P_w,j V_j
            // once P_w,j is written.  The whole warp runs the loop and computes
            // the descriptors; one elected lane issues the MMAs and commits.
            const int w = static_cast<int>(warp) - 1;
            constexpr int jl = 0;
            const int n = n_kv[w];
            // Descriptors are built once; a K=16 step adds 32 bytes (2 units of
            // 16 B) to the start address, a stage adds 2 tiles, a V step 16 rows.
            constexpr uint64_t kStageStep = (2 * Cfg::kTileBytes) >> 4;
            const uint64_t dq = smem_desc(smem_u32(smem + Cfg::kQOff + w * Cfg::kTileBytes), 16,
                                          Cfg::kAtomBytes, Cfg::kSwz);
            const uint64_t dk0 = smem_desc(smem_u32(smem + Cfg::kKVOff), 16, Cfg::kAtomBytes, Cfg::kSwz);
            const uint64_t dv0 = smem_desc(smem_u32(smem + Cfg::kKVOff + Cfg::kTileBytes),
                                           Cfg::kTileBytes, Cfg::kAtomBytes, Cfg::kSwz);
            const uint32_t ds = tmem_base + Cfg::kTmemS + w * 128;
            const uint32_t dout = tmem_base + Cfg::kTmemO + w * D;
            const uint32_t pa = tmem_base + Cfg::kTmemP + w * 64;
            int kv_ready = -1;   // key/value tiles 0..kv_ready are known to be in smem
            auto ensure_kv = [&](int j) -> bool {
                if (j <= kv_ready) return true;
                if (!mbar_wait_warp(&kv_full[j % NS], static_cast<uint32_t>(j / NS) & 1u, wc, 222))
                    return false;
                tc_fence_after();
                kv_ready = j;
                return true;
            };
            auto issue_s = [&](int j) -> bool {
                if (!ensure_kv(j)) return false;
                const uint64_t dk = dk0 + static_cast<uint64_t>(j % NS) * kStageStep;
                if (elect_one()) {
#pragma unroll
                    for (int k = 0; k < D / 16; ++k)
                        mma_bf16_ss(ds, dq + 2 * k, dk + 2 * k, IDESC_S, k != 0 ? 1u : 0u);
                    mma_commit(&s_full[w]);
                }
                __syncwarp();
                return true;
            };
            // PV in two halves of 64 keys, each issued as soon as softmax w has
            // written that half of P: the first half's MMAs run while the
            // second half is being exponentiated.
            auto issue_pv = [&](int j) -> bool {
                if (!ensure_kv(j)) return false;
                const uint64_t dv = dv0 + static_cast<uint64_t>(j % NS) * kStageStep;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (!mbar_wait_warp(&p_full[2 * w + h], static_cast<uint32_t>(j - jl) & 1u, wc, 224))
                        return false;
                    tc_fence_after();
                    if (elect_one()) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            // P from TMEM (16 keys = 8 columns); V: rows = keys (the K
                            // dimension), d contiguous (MN-major); 16 keys = two 8-row atoms.
                            const int kk = 4 * h + q;
                            mma_bf16_ts(dout, pa + kk * 8, dv + kk * ((16 * Cfg::kRowBytes) >> 4),
                                        IDESC_PV, (j > jl || kk != 0) ? 1u : 0u);
                        }
                        if (h == 1) mma_commit(&pv_done[w]);
                    }
                    __syncwarp();
                }
                return true;
            };
            bool ok = mbar_wait_warp(q_full, 0, wc, 221);
            if (ok) tc_fence_after();
            // only the tiles of [jl, n): the producer releases the others
            if (ok && n > jl) ok = issue_s(jl);
            for (int j = jl; j < n && ok; ++j) {
                if (j + 1 < n) {
                    ok = mbar_wait_warp(&s_free[w], static_cast<uint32_t>(j - jl) & 1u, wc, 223);
                    if (ok) {
                        tc_fence_after();
                        ok = issue_s(j + 1);
                    }
                }
                if (ok) ok = issue_pv(j);
                if (ok) {
                    if (elect_one()) mma_commit(&kv_empty[j % NS]);
                    __syncwarp();
                }
            }
            if (elect_one()) mma_commit(&drain[w]);
            __syncwarp();
            mbar_wait_warp(&drain[w], 0, wc, 227);
        }
    } else {
        setmaxnreg_inc<kRegsSoftmax>();
        // ---------------------------------------------------- softmax groups
        const int w = (warp >= 8) ? 1 : 0;
        const uint32_t quad = warp & 3u;
        const int r = static_cast<int>(quad * 32 + lane);
        const int qrow = q0 + 128 * w + r;
        const bool valid = qrow < len;
        // visible keys of this row, relative to kbase
        const int cend = (valid ? key_hi(p, rs, len, qrow) : 1) - kbase;
        const int cbeg = (valid ? key_lo(p, rs, qrow) : 0) - kbase;
        const uint32_t lane_off = (quad * 32u) << 16;
        const uint32_t ts = tmem_base + lane_off + Cfg::kTmemS + w * 128;
        const uint32_t to = tmem_base + lane_off + Cfg::kTmemO + w * D;
        const float sc = p.scale_log2;
        constexpr int jl = 0;
        const int n = n_kv[w];
        // exp-pass turns: tile j of group 0 waits for group 1's tile j - 1, tile
        // j of group 1 for group 0's tile j, when the other group has that tile;
        // jt = j - turn_lo is the waited-for pass of the other group
        const int turn_lo = (w == 0) ? 1 : 0;
        const int turn_hi = (w == 0) ? n_kv[1] + 1 : n_kv[0];
        const uint32_t tp = tmem_base + lane_off + Cfg::kTmemP + w * 64;
        float m = NEG_INF, l = 0.0f;

        bool ok = true;
        for (int j = jl; j < n; ++j) {
            const uint32_t it = static_cast<uint32_t>(j - jl);   // tiles done by this group
            ok = mbar_wait(&s_full[w], it & 1u, wc, 321);
            if (!__all_sync(0xffffffffu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            // the whole S row in registers: one TMEM round trip per tile, after
            // which the tensor core may overwrite S with the next tile's scores
            float s[128];
            tmem_ld32(ts, s);
            tmem_ld32(ts + 32, s + 32);
            tmem_ld32(ts + 64, s + 64);
            tmem_ld32(ts + 96, s + 96);
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&s_free[w]);
            const int k0 = j * 128;
            if (k0 + 128 > cend || k0 < cbeg) {
                // keys outside [cbeg, cend) are masked; fully visible tiles skip this
                const int hi = cend - k0, lo = cbeg - k0;
#pragma unroll
                for (int i = 0; i < 128; ++i) s[i] = (i < hi && i >= lo) ? s[i] : NEG_INF;
            }
            // row max of the (masked) scores in eight independent chains
            float mxv[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) mxv[q] = NEG_INF;
#pragma unroll
            for (int i = 0; i < 128; i += 2) mxv[(i >> 1) & 7] = fmax3(mxv[(i >> 1) & 7], s[i], s[i + 1]);
            float mx = fmaxf(fmaxf(fmaxf(mxv[0], mxv[1]), fmaxf(mxv[2], mxv[3])),
                             fmaxf(fmaxf(mxv[4], mxv[5]), fmaxf(mxv[6], mxv[7])));
            mx *= sc;
            // O_w and P_w are free once PV_w,j-1 has completed
            if (j > jl) {
                ok = mbar_wait(&pv_done[w], (it - 1u) & 1u, wc, 322);
                if (!__all_sync(0xffffffffu, ok)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
            }
            // lazily move the reference max: on the first tile, or when this
            // tile would push P above 2^8 somewhere in the warp.  A row whose
            // visible keys start in a later tile (block-diagonal mask) keeps
            // m = -inf until then: its P is 0 (exponent taken against 0) and
            // its first rescale multiplies the zero O and l by 0.
            const bool raise = (j == jl) || (mx > m + kRescaleLog2);
            if (__any_sync(0xffffffffu, raise)) {
                const float m_new = fmaxf(m, mx);
                if (j > jl) {
                    const float alpha = (m == m_new) ? 1.0f : ex2(m - m_new);
#pragma unroll
                    for (int c = 0; c < D; c += 16) {
                        float o[16];
                        tmem_ld16(to + c, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 16; ++i) o[i] *= alpha;
                        tmem_st16(to + c, o);
                    }
                    l *= alpha;
                }
                m = m_new;
            }
            if (kTurns && j >= turn_lo && j < turn_hi) {
                // group 0 goes first on each key tile
                const int jt = j - turn_lo;
                ok = mbar_wait(&turn[(1 - w) * 4 + quad], static_cast<uint32_t>(jt) & 1u, wc, 323);
                if (!__all_sync(0xffffffffu, ok)) {
                    ok = false;
                    break;
                }
            }
            // P = 2^(s*sc - m) -> bf16 pairs in TMEM, and the row sum
            const float m_ref = (m == NEG_INF) ? 0.0f : m;
            float rs8[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) rs8[q] = 0.0f;
#pragma unroll
            for (int h = 0; h < 128; h += 64) {
                uint32_t pk[32];
#pragma unroll
                for (int i = 0; i < 64; i += 2) {
                    float t0, t1;
                    ffma2(t0, t1, s[h + i], s[h + i + 1], sc, sc, -m_ref, -m_ref);
                    const float e0 = ex2(t0);
                    const float e1 = ex2(t1);
                    const int q = (i >> 1) & 3;       // four pairs of running sums
                    fadd2(rs8[2 * q], rs8[2 * q + 1], rs8[2 * q], rs8[2 * q + 1], e0, e1);
                    pk[i >> 1] = pack_bf16x2(e0, e1);
                }
                tmem_st32u(tp + h / 2, pk);
                // hand this half of P to the MMA issuer
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&p_full[2 * w + (h >> 6)]);
            }
            if (kTurns) {
                __syncwarp();
                if (lane == 0) mbar_arrive(&turn[w * 4 + quad]);
            }
            l += ((rs8[0] + rs8[1]) + (rs8[2] + rs8[3])) + ((rs8[4] + rs8[5]) + (rs8[6] + rs8[7]));
        }
        if (ok && n > jl) {
            ok = mbar_wait(&pv_done[w], static_cast<uint32_t>(n - 1 - jl) & 1u, wc, 324);
            ok = __all_sync(0xffffffffu, ok);
        }
        if (ok && n > jl) {
            tc_fence_after();
            const float inv = 1.0f / l;
            // the row's log-sum-exp for a backward pass: P = 2^(s sc - (m + log2 l))
            if (kLse && valid)
                p.lse[static_cast<int64_t>(head) * p.req_start[p.n_req] + rs + qrow] = m + log2f(l);
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

template <int D, bool kLse>
cr_status launch_d(const CUtensorMap& tm, const AttnParams& p, cudaStream_t st) {
    using Cfg = AttnCfg<D>;
    auto kern = attn_kernel<D, kLse>;
    static unsigned long long attr_done = 0;   // one per template instantiation
    const cr_status sa = ensure_smem_attr(kern, static_cast<int>(Cfg::kSmemBytes), &attr_done);
    if (sa != CR_OK) return sa;
    // The softmax warpgroups raise their register budget inside the kernel;
    // that only completes if the launch reserved the 168 registers per thread
    // the split assumes.  Refuse to launch a build that reserves fewer.
    static int regs_ok = -1;   // per template instantiation; same answer on every device
    int ok = __atomic_load_n(&regs_ok, __ATOMIC_ACQUIRE);
    if (ok < 0) {
        cudaFuncAttributes fa;
        const cr_status sf = cuda_check(cudaFuncGetAttributes(&fa, kern));
        if (sf != CR_OK) return sf;
        ok = (fa.numRegs >= static_cast<int>(kRegsLaunch) && fa.maxThreadsPerBlock >= kThreads) ? 1 : 0;
        __atomic_store_n(&regs_ok, ok, __ATOMIC_RELEASE);
    }
    if (!ok) return CR_ERR_UNSUPPORTED;
    const int grid = p.n_items * p.n_heads;
    return launch_pdl(kern, dim3(grid), dim3(kThreads), Cfg::kSmemBytes, st, tm, p);
}

// chunk_start[t] = the request-local index of the first token of t's chunk:
// the smallest u with chunk_end[u] > i, i = t's request-local index (tokens of
// earlier chunks have chunk_end <= their chunk's end <= i, tokens of i's chunk
// have chunk_end > i).  One thread per token, binary searches over the
// request starts and over the request's non-decreasing chunk_end; the result
// lies in [0, i] whatever the map holds.
__global__ void __launch_bounds__(256)
    chunk_start_kernel(const int32_t* __restrict__ chunk_end, int32_t* __restrict__ chunk_start,
                       const __grid_constant__ AttnParams p, int n_tokens) {
    pdl_launch_dependents();
    pdl_wait();   // the chunk map comes from an earlier kernel
    const int t = static_cast<int>(blockIdx.x * blockDim.x + threadIdx.x);
    if (t >= n_tokens) return;
    int r0 = 0, r1 = p.n_req - 1;       // the request r with req_start[r] <= t
    while (r0 < r1) {
        const int mid = (r0 + r1 + 1) >> 1;
        if (p.req_start[mid] <= t) r0 = mid;
        else r1 = mid - 1;
    }
    const int rs = p.req_start[r0];
    const int i = t - rs;
    int a = 0, b = i;
    while (a < b) {
        const int mid = (a + b) >> 1;
        if (__ldg(chunk_end + rs + mid) > i) b = mid;
        else a = mid + 1;
    }
    chunk_start[t] = a;
}

}  // namespace

cr_status launch_chunk_starts(const int32_t* chunk_end, const AttnParams& p, int64_t n_tokens,
                              int32_t* chunk_start, cudaStream_t st) {
    if (n_tokens < 1) return CR_OK;
    const int grid = static_cast<int>((n_tokens + 255) / 256);
    return launch_pdl(chunk_start_kernel, dim3(grid), dim3(256), 0, st, chunk_end, chunk_start, p,
                      static_cast<int>(n_tokens));
}

cr_status launch_attention(const uint16_t* qkv, int64_t n_tokens, int head_dim,
                           const AttnParams& p, cudaStream_t st) {
    if (head_dim != 32 && head_dim != 64) return CR_ERR_UNSUPPORTED;
    if (p.n_items <= 0) return CR_OK;
    CUtensorMap tm;
    if (!make_tmap_2d(&tm, qkv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3ull * p.d_b, n_tokens,
                      3ull * p.d_b * 2, head_dim, 128,
                      head_dim == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B))
        return CR_ERR_INVALID_ARG;
    if (p.lse) return head_dim == 64 ? launch_d<64, true>(tm, p, st) : launch_d<32, true>(tm, p, st);
    return head_dim == 64 ? launch_d<64, false>(tm, p, st) : launch_d<32, false>(tm, p, st);
}

}  // namespace cr
