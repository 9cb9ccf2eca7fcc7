// tcgen05 GEMM for every dense linear of the repair path (Sec. 4.1):
//   C[M, N] = A[M, K] * W[N, K]^T + bias, with a fused epilogue.
//
// Design (sm_103a, persistent; every launch runs on CTA pairs, clusters of two
// CTAs on two SMs computing 256-row tiles with tcgen05 cta_group::2 MMAs):
//   warp 0      TMA producer: this CTA's 128 rows of A and half of the W tile,
//               64-wide k-slices (128B swizzle) into a shared-memory ring; both
//               CTAs' copies count on the even CTA's full barrier.
//   warp 1      TMEM owner (both CTAs); in the even CTA one elected lane of the
//               converged warp issues the M = 256, N = BN, K = 16 MMAs into a
//               double-buffered fp32 accumulator and multicasts its commits.
//   warp 2      epilogue-input loader: per tile, the bias (and sigma_delta)
//               slice by bulk copy and, for in-place epilogues, the output tile
//               itself (the stale cache tile, or for the training loss head the
//               stale and joint cache tiles) by TMA, as soon as the epilogue has
//               released its slot.
//   warp 3      TMA store issuer for the staged in-place tile.
//   warps 4..11 epilogue, two groups of four warps (one per TMEM lane
//               quarter) splitting each tile's columns: tcgen05.ld 32 lanes x
//               16 columns, bias from shared memory, then one of: bf16, GELU,
//               fp32, RoPE on Q/K (into 128B-swizzled staging buffers, one box
//               of 128 B-wide columns at a time, double-buffered per group,
//               each box stored by one thread of the group after a named
//               barrier; the fp32 residual stream as a TMA reduce-add,
//               x += acc + b in L2), or in place on the staged tile: cache
//               kv = kv + sigma_delta (acc + b) (+ R_M on K), stored by warp 3.
//               Staged data goes out with TMA (coalesced, asynchronous).  The
//               paged head and the loss head write from registers instead: the
//               repaired rows into the paged target cache, or the training
//               gradient dz = c (acc + b - (joint - stale) / sigma_delta) in
//               bf16 with each row's sum of squares of the residual.
// Warps 0..3 give registers to the epilogue warpgroups (setmaxnreg).
#include <cuda_bf16.h>

#include "cr_internal.h"
#include "cr_ptx.cuh"

namespace cr {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr uint32_t A_BYTES = BM * BK * 2;
constexpr uint32_t kSmemLimit = 232448;   // 227 KB opt-in per CTA
// 12 warps: 0 TMA producer, 1 MMA issuer (TMEM owner), 2 epilogue-input
// loader, 3 TMA store issuer, 4..11 epilogue in two groups of four warps that
// split each tile's columns.  The first warpgroup gives registers to the
// epilogue warpgroups (launch: 65536 / 384 = 168 per thread, checked on the
// host): 64 * 128 + 2 * 216 * 128 <= 168 * 384.
constexpr int kGemmThreads = 384;
constexpr uint32_t kGemmRegsLaunch = 168;
constexpr uint32_t kGemmRegsCtl = 64;
constexpr uint32_t kGemmRegsEpi = 216;
static_assert(kGemmRegsCtl * 128 + 2 * kGemmRegsEpi * 128 <= kGemmRegsLaunch * kGemmThreads,
              "register split exceeds the launch allocation");

template <int BN, int EPI, int CG>
struct GemmCfg {
    static constexpr bool kKV =
        (EPI == EPI_KV_BF16 || EPI == EPI_KV_F32 || EPI == EPI_KV_PAGED || EPI == EPI_KV_LOSS ||
         EPI == EPI_KV_POOL);
    // the stale tile comes from the chunk pool (a 128-row TMA box where a box's rows
    // are one chunk's; across a chunk boundary 8-row TMA boxes, and cp.async for the
    // rows of the 8-row group that crosses it), the repaired tile goes to the output
    static constexpr bool kPoolSrc = (EPI == EPI_KV_POOL);
    // the stale tile is staged as for the in-place update, but the repaired rows
    // go straight from registers to the paged target cache (no TMA store)
    static constexpr bool kPaged = (EPI == EPI_KV_PAGED);
    // training head: the residual r goes out as the bf16 gradient dz and row sums
    // of r^2, from registers (no TMA store)
    static constexpr bool kLoss = (EPI == EPI_KV_LOSS);
    static constexpr bool kDirect = kPaged || kLoss;
    static constexpr bool kInPlace = kKV;   // tile loaded, updated, stored
    // the fp32 residual add goes out as a TMA reduce-add of the staged box
    // (x += acc + bias in L2, one add per element: the same rounding as a
    // load, add and store, without staging the old tile)
    static constexpr bool kReduce = (EPI == EPI_ADD_F32);
    static constexpr int kTileEsize = (EPI == EPI_KV_F32 || EPI == EPI_ADD_F32 || EPI == EPI_F32) ? 4 : 2;
    static constexpr int kBoxCols = 128 / kTileEsize;          // one 128-byte swizzle row
    // in-place epilogues stage the whole [BM x BN] tile; store-only epilogues
    // stage one 16 KB box (128 rows x 128 B) at a time per epilogue group
    // (boxes alternate between the two groups), double-buffered where the
    // epilogue arithmetic is heavy (GELU, RoPE) and single otherwise, which
    // leaves room for a deeper operand ring
    static constexpr int kBoxes = BN / kBoxCols;                // boxes per tile
    static constexpr int kGroupBufs = (EPI == EPI_GELU_BF16 || EPI == EPI_QKV_ROPE) ? 2 : 1;
    // (the loss head stages two bf16 tiles: stale in the even, joint in the odd
    // 16 KB boxes, column box b at boxes 2 b and 2 b + 1)
    static constexpr uint32_t kTileBytes =
        kInPlace ? BM * BN * kTileEsize * (kLoss ? 2 : 1) : 2 * kGroupBufs * 16384;
    // the 256-wide bf16 heads read their bias and sigma slices straight from global
    // memory (every thread of a warp the same address: one broadcast load from L1),
    // so that the 4 KB of staged vectors go to a fifth operand stage beside the
    // 64 KB staged tile
    static constexpr bool kVecGlobal = (EPI == EPI_KV_BF16 || EPI == EPI_KV_POOL || EPI == EPI_KV_PAGED);
    static constexpr uint32_t kVecBytes = kVecGlobal ? 0u : BN * 4 * (kKV ? 2 : 1);   // bias (+ sigma)
    // in-place epilogues recycle the staged tile box by box, so the next tile's
    // vectors may land while this tile is still being finished: two buffers
    static constexpr int kVecBufs = kInPlace ? 2 : 1;
    static constexpr uint32_t kBBytes = (BN / CG) * BK * 2;      // this CTA's share of W
    static constexpr uint32_t kStageBytes = A_BYTES + kBBytes;
    static constexpr uint32_t kFixed = 1024 + kTileBytes + kVecBufs * kVecBytes + 512;
    static constexpr int kStagesFit = static_cast<int>((kSmemLimit - kFixed) / kStageBytes);
    static constexpr int kStages = kStagesFit > 8 ? 8 : kStagesFit;
    static_assert(kStages >= 4, "GEMM tile does not fit in shared memory");
    static constexpr uint32_t kSmemBytes = kFixed + kStages * kStageBytes;
    // double-buffered accumulator; TMEM is allocated in powers of two
    static constexpr uint32_t kTmemCols = (2 * BN <= 256) ? 256u : 512u;
};

// GELU(x) = x Phi(x) for a pair of values, branch-free.  Phi is written as a
// logistic function of its log2-odds: Phi(x) = 1 / (1 + 2^(x H(x^2))), with H a
// degree-6 polynomial fitted by gelu_sigmoid_fit.py in this directory (GELU's
// absolute error <= 8.3e-8 on [-12, 12] in float64; beyond the fitted range
// |x H| >= 34, so Phi is 0 or 1 to within 2^-34 there as the exact Phi is).
// Per pair: a packed square, six packed FMAs, a packed multiply, two 2^y, a
// packed add, two reciprocals and a packed multiply.
__device__ constexpr float kGeluH[7] = {-2.302209146e+00f, -1.048354083e-01f, 9.409242776e-05f,
                                        1.596513719e-04f, -1.146683675e-05f,
                                        3.847686963e-07f, -5.180393528e-09f};
__device__ __forceinline__ void gelu2(float& a, float& b) {
    float sa, sb;
    fmul2(sa, sb, a, b, a, b);
    float ha = kGeluH[6], hb = kGeluH[6];
#pragma unroll
    for (int i = 5; i >= 0; --i) ffma2(ha, hb, ha, hb, sa, sb, kGeluH[i], kGeluH[i]);
    fmul2(ha, hb, ha, hb, a, b);                        // -log2 odds of Phi
    float da, db;
    fadd2(da, db, ex2(ha), ex2(hb), 1.0f, 1.0f);        // 1 / Phi
    fmul2(a, b, a, b, rcp_approx(da), rcp_approx(db));
}

// This row's (cos, sin) for every pair index q of the repairer RoPE: from the
// angle-major table (entry q * M + row: a warp's 32 rows read 256 contiguous
// bytes per q), or computed in place when no table is given.
template <int NP>
__device__ __forceinline__ void rope_angles(const GemmParams& p, int row, float (&cs)[NP],
                                            float (&sn)[NP]) {
    const bool in = row < p.M;
    const int half = p.rope_dim / 2;
    if (p.rope_table) {
        const float2* tb = p.rope_table + (in ? row : 0);
#pragma unroll
        for (int q = 0; q < NP; ++q) {
            if (q < half) {
                const float2 v = __ldg(tb + static_cast<int64_t>(q) * p.M);
                cs[q] = v.x;
                sn[q] = v.y;
            }
        }
    } else {
        const float pr = in ? static_cast<float>(__ldg(p.pos + row)) : 0.0f;
#pragma unroll
        for (int q = 0; q < NP; ++q)
            if (q < half) sincos_prod(pr, p.inv_freq[q], &sn[q], &cs[q]);
    }
}

// 16 consecutive bf16 of a [128 x (64*k)] tile stored as 128B-swizzled boxes
// of 64 columns; col multiple of 16.  Byte offsets of its two 16-byte chunks.
__device__ __forceinline__ void swz_offsets_bf16(int row, int col, uint32_t* o0, uint32_t* o1) {
    const int box = col >> 6;
    const int ch = (col & 63) >> 3;
    const uint32_t base = box * 16384 + row * 128;
    *o0 = base + (((ch) ^ (row & 7)) << 4);
    *o1 = base + (((ch + 1) ^ (row & 7)) << 4);
}

__device__ __forceinline__ void load16_bf16_smem(const uint8_t* tile, int row, int col, float* v) {
    uint32_t o0, o1;
    swz_offsets_bf16(row, col, &o0, &o1);
    const uint4 a = *reinterpret_cast<const uint4*>(tile + o0);
    const uint4 b = *reinterpret_cast<const uint4*>(tile + o1);
    const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        v[2 * i] = __uint_as_float(w[i] << 16);
        v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ void store16_bf16_smem(uint8_t* tile, int row, int col, const float* v) {
    uint32_t o0, o1;
    swz_offsets_bf16(row, col, &o0, &o1);
    *reinterpret_cast<uint4*>(tile + o0) = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                                      pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
    *reinterpret_cast<uint4*>(tile + o1) =
        make_uint4(pack_bf16x2(v[8], v[9]), pack_bf16x2(v[10], v[11]), pack_bf16x2(v[12], v[13]),
                   pack_bf16x2(v[14], v[15]));
}

// fp32 tile: boxes of 32 columns (128 B rows), 4 chunks of 4 floats.
__device__ __forceinline__ uint32_t swz_offset_f32(int row, int col, int k) {
    const int box = col >> 5;
    const int ch = ((col & 31) >> 2) + k;
    return box * 16384 + row * 128 + ((ch ^ (row & 7)) << 4);
}

__device__ __forceinline__ void load16_f32_smem(const uint8_t* tile, int row, int col, float* v) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float4 a = *reinterpret_cast<const float4*>(tile + swz_offset_f32(row, col, k));
        v[4 * k] = a.x;
        v[4 * k + 1] = a.y;
        v[4 * k + 2] = a.z;
        v[4 * k + 3] = a.w;
    }
}

__device__ __forceinline__ void store16_f32_smem(uint8_t* tile, int row, int col, const float* v) {
#pragma unroll
    for (int k = 0; k < 4; ++k)
        *reinterpret_cast<float4*>(tile + swz_offset_f32(row, col, k)) =
            make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
}

template <int ES>
__device__ __forceinline__ void load16_tile(const uint8_t* t, int row, int col, float* v) {
    if constexpr (ES == 2)
        load16_bf16_smem(t, row, col, v);
    else
        load16_f32_smem(t, row, col, v);
}
template <int ES>
__device__ __forceinline__ void store16_tile(uint8_t* t, int row, int col, const float* v) {
    if constexpr (ES == 2)
        store16_bf16_smem(t, row, col, v);
    else
        store16_f32_smem(t, row, col, v);
}

__device__ __forceinline__ void store16_bf16_global(uint16_t* dst, const float* v) {
    reinterpret_cast<uint4*>(dst)[0] = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                                  pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
    reinterpret_cast<uint4*>(dst)[1] =
        make_uint4(pack_bf16x2(v[8], v[9]), pack_bf16x2(v[10], v[11]), pack_bf16x2(v[12], v[13]),
                   pack_bf16x2(v[14], v[15]));
}

// 16 consecutive floats of a shared-memory vector (all lanes read the same
// addresses: broadcast).
__device__ __forceinline__ void vec16(const float* v, int col, float* out) {
    const float4* p4 = reinterpret_cast<const float4*>(v + col);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const float4 x = p4[q];
        out[4 * q] = x.x;
        out[4 * q + 1] = x.y;
        out[4 * q + 2] = x.z;
        out[4 * q + 3] = x.w;
    }
}

// First output column of tile t.  Tiles are walked W-tile-major (t / num_m is
// the column tile); under an output choice (KV epilogues with col_block > 0)
// only the K or only the V column blocks are walked.
// Tile walk of a launch: t -> (linear tile, k-part).  The linear tile c num_m + m
// names row tile m of column tile c.  Default order: k-parts fastest, then row
// tiles, then column tiles (W-tile-major: the CTAs running together share a W
// tile, and the activations stay in L2).  n_fast: column tiles fastest, then
// row tiles, k-parts slowest, for an A operand much larger than L2: the tiles
// running together share their A rows and one k-range of W, so A is read once.
__device__ __forceinline__ int tile_lin(const GemmParams& p, int t) {
    if (p.n_fast) {
        const int r = t % (p.num_m * p.num_n);
        return (r % p.num_n) * p.num_m + r / p.num_n;
    }
    return t / p.split_k;
}
__device__ __forceinline__ int tile_part(const GemmParams& p, int t) {
    return p.n_fast ? t / (p.num_m * p.num_n) : t % p.split_k;
}

template <int BN, bool KV>
__device__ __forceinline__ int tile_n0(const GemmParams& p, int t) {
    const int c = t / p.num_m;
    if constexpr (KV) {
        if (p.col_block > 0) {
            const int per = p.col_block / BN;   // column tiles per block
            const int blk = c / per;
            return (2 * blk + p.col_phase) * p.col_block + (c - blk * per) * BN;
        }
    }
    return c * BN;
}

// The same rotation with (cos, sin) read from a per-call angle-major table
// (entry q * M + row, written by the RoPE-table kernel with sincos_prod's
// formula: the same rotation to the last bit of an angle).
__device__ __forceinline__ void rotate16_tab(float* a, float* b, const float2* tab, int64_t M, int row,
                                             int j0) {
    const float2* t = tab + static_cast<int64_t>(j0) * M + row;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const float2 v = __ldg(t + i * M);
        const float x = a[i], y = b[i];
        a[i] = x * v.x - y * v.y;
        b[i] = y * v.x + x * v.y;
    }
}

__device__ __forceinline__ void rotate16(float* a, float* b, float p, const float* inv_freq, int j0) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        float s, c;
        sincos_prod(p, inv_freq[j0 + i], &s, &c);
        const float x = a[i], y = b[i];
        a[i] = x * c - y * s;
        b[i] = y * c + x * s;
    }
}

// Operand layouts (LAY, cr_internal.h): LAY_KK = A [M, K] and W [N, K], both
// K-major (the forward's linears); LAY_KM = A K-major, W stored [K, N]
// (MN-major: dX = dY W of the backward); LAY_MM = A stored [K, M] and W [K, N],
// both MN-major (dW = dY^T X).  An MN-major operand arrives as 64-wide boxes of
// 64 K-rows (128B swizzle): the MMA descriptor steps 16 K-rows (2 KB) per
// K = 16 MMA and finds the next 64 M (or N) 8 KB further on (leading byte
// offset).

// all n threads at named barrier id agree on v (true only if every one passed true)
__device__ __forceinline__ bool named_bar_and(uint32_t id, uint32_t n, bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "barrier.cta.red.and.pred q, %2, %3, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(v ? 1u : 0u), "r"(id), "r"(n)
        : "memory");
    return r != 0;
}

template <int BN, int EPI, int CG, int LAY>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmC, const __grid_constant__ GemmParams p) {
    using Cfg = GemmCfg<BN, EPI, CG>;
    constexpr int STAGES = Cfg::kStages;
    constexpr bool kAMN = (LAY == LAY_MM), kBMN = (LAY == LAY_KM || LAY == LAY_MM);
    constexpr bool kPair = (LAY == LAY_KK2);
    static_assert(!kBMN || (BN / CG) % 64 == 0, "an MN-major W half must be whole 64-column boxes");
    constexpr uint32_t IDESC = idesc_bf16(BM * CG, BN, kAMN, kBMN);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* tile = smem + STAGES * Cfg::kStageBytes;              // staged output (part)
    float* vec = reinterpret_cast<float*>(tile + Cfg::kTileBytes);  // [buffer] bias [BN] (+ sigma [BN])
    uint64_t* bars = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(vec) +
                                                 Cfg::kVecBufs * Cfg::kVecBytes);
    uint64_t* full = bars;
    uint64_t* empty = bars + STAGES;
    uint64_t* tfull = bars + 2 * STAGES;
    uint64_t* tempty = tfull + 2;
    // loader -> epilogue: the vectors (+ box b of the in-place tile) landed; in-place
    // epilogues use one per box (box 0 also carries the vectors), the others only [0]
    uint64_t* epi_full = tempty + 2;     // [8]
    uint64_t* epi_empty = epi_full + 8;  // [8] back to the loader: box b (and the vectors) free
    uint64_t* drain = epi_empty + 8;
    uint64_t* epi_done = drain + 1;      // [8] in-place: box b written (to the store issuer)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(epi_done + 8);
    int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);

    const uint32_t warp = warp_id(), lane = lane_id();
    pdl_launch_dependents();
    // CTA pairs (CG = 2): cluster c computes 256-row tiles; rank r holds rows
    // 128 r .. 128 r + 127 of each and half of its W tile.
    const uint32_t rank = (CG == 2) ? cluster_ctarank() : 0u;
    const int cta0 = static_cast<int>(blockIdx.x) / CG;   // cluster index
    const int ncta = static_cast<int>(gridDim.x) / CG;    // clusters
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&tfull[s], 1);
            mbar_init(&tempty[s], 8 * CG);   // the epilogue warps of every CTA of the tile
        }
        for (int b = 0; b < 8; ++b) {
            mbar_init(&epi_full[b], 1);
            // store-only: epi_empty[0] takes one arrive from each epilogue group
            mbar_init(&epi_empty[b], (!Cfg::kInPlace && b == 0) ? 2 : 1);
            // in-place: one barrier per box for all 256 epilogue threads
            mbar_init(&epi_done[b], 256);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        if constexpr (CG == 2)
            tmem_alloc2(tmem_slot, Cfg::kTmemCols);
        else
            tmem_alloc(tmem_slot, Cfg::kTmemCols);
    }
    tc_fence_before();
    if constexpr (CG == 2)
        cluster_sync();   // both CTAs' barriers and TMEM exist before any pair traffic
    else
        __syncthreads();
    tc_fence_after();
    pdl_wait();   // operands, the in-place tile and positions come from earlier kernels
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx wc{abort_flag, p.status};

    // split-K (split_k > 1): tile t / split_k, k-blocks of part t % split_k; each
    // part's fp32 result goes to its own [M, N] slice of the output (rows
    // (t % split_k) M ..), summed later in a fixed order
    const int total = p.num_m * p.num_n * p.split_k;
    // a two-term A runs the W k-blocks twice: first against A_hi, then A_lo
    const int num_k = p.split_kb > 0 ? 2 * p.split_kb : (p.K + BK - 1) / BK;
    const int num_k2 = kPair ? (p.split_kb2 > 0 ? 2 * p.split_kb2 : (p.K2 + BK - 1) / BK) : 0;
    const int k_per = (num_k + p.split_k - 1) / p.split_k;
    // two products (n_split > 0): a tile belongs to the second one when its first
    // column is at or past n_split
    auto second = [&](int n0) { return kPair && n0 >= p.n_split; };
    // Two products, pair c taking tiles c, c + ncta, ...: the first product's H
    // (longer) tiles come first.  Where the launch has E = tiles - pairs > 0
    // second tiles to hand out and the second product's tiles can take them all
    // twice over, E of those lead instead, so that the pairs running two tiles
    // run two short ones: pairs 0..E-1 short + short, E..E+H-1 one long tile,
    // the rest one short tile.
    const int n_long = kPair ? p.num_m * (p.n_split / BN) : 0;
    const int n_extra = total - ncta;
    const bool reorder = kPair && n_extra > 0 && 2 * n_extra <= total - n_long && n_long + n_extra <= ncta;
    auto lin = [&](int t) {
        if constexpr (kPair) {
            if (reorder) return t < n_extra ? n_long + t : (t < n_extra + n_long ? t - n_extra : t);
        }
        return tile_lin(p, t);
    };
    auto k_range = [&](int t, int* kb0, int* kb1) {
        if constexpr (kPair) {
            *kb0 = 0;
            *kb1 = second(tile_n0<BN, Cfg::kKV>(p, lin(t))) ? num_k2 : num_k;
            return;
        }
        *kb0 = tile_part(p, t) * k_per;
        *kb1 = min(num_k, *kb0 + k_per);
    };
    const bool has_bias = p.bias != nullptr;
    // the epilogue consumes a per-tile load (vectors and/or the in-place tile)
    const bool epi_load = Cfg::kInPlace || has_bias;
    // the in-place tile is read unless a zero output offset makes every row's
    // stale value unused (no kept rows)
    const bool load_tile = Cfg::kInPlace && !(Cfg::kKV && p.kv_zero && p.keep_chunk == nullptr);

    // The producer, loader, store and MMA roles each run as a converged warp
    // (operands stay warp-uniform); one elected lane issues the copies and MMAs.
    if (warp < 4) {
    setmaxnreg_dec<kGemmRegsCtl>();
    if (warp == 0) {
        // ---------------------------------------------------- TMA producer
        if (elect_one()) {
            tma_prefetch(&tmA);
            tma_prefetch(&tmB);
            if (p.split_kb > 0) tma_prefetch(&p.tm_alo);
            if constexpr (Cfg::kInPlace) tma_prefetch(&tmC);
            if constexpr (kPair) {
                tma_prefetch(&p.tm_a2);
                tma_prefetch(&p.tm_b2);
                if (p.split_kb2 > 0) tma_prefetch(&p.tm_alo2);
            }
        }
        __syncwarp();
        uint32_t stage = 0, phase = 0;
        bool ok = true;
        for (int t = cta0; t < total && ok; t += ncta) {
            const int m0 = (lin(t) % p.num_m) * (BM * CG) + static_cast<int>(rank) * BM;
            const int n0 = tile_n0<BN, Cfg::kKV>(p, lin(t));
            int kbeg, kend;
            k_range(t, &kbeg, &kend);
            for (int kb = kbeg; kb < kend; ++kb) {
                if (!(ok = mbar_wait_warp(&empty[stage], phase ^ 1u, wc, 102))) break;
                uint8_t* sa = smem + stage * Cfg::kStageBytes;
                if (elect_one()) {
                    // W columns of this tile: its own column block, or (grouped
                    // rows) the block that belongs to its rows' group
                    const bool g2 = second(n0);
                    const int nw = p.bgroup_rows > 0
                                       ? ((lin(t) % p.num_m) * (BM * CG) / p.bgroup_rows) * BN
                                       : (g2 ? n0 - p.n_split : n0);
                    const int nb0 = nw + static_cast<int>(rank) * (BN / CG);
                    const int skb = g2 ? p.split_kb2 : p.split_kb;
                    const bool lo = skb > 0 && kb >= skb;
                    const CUtensorMap* ma = g2 ? (lo ? &p.tm_alo2 : &p.tm_a2) : (lo ? &p.tm_alo : &tmA);
                    const CUtensorMap* mb = g2 ? &p.tm_b2 : &tmB;
                    const int ka = (lo ? kb - skb : kb) * BK;   // A and W column
                    uint64_t* fq = &full[stage];
                    auto load = [&](uint8_t* dst, const CUtensorMap* m, int x, int y, uint32_t fb) {
                        if constexpr (CG == 1)
                            tma_load_2d(dst, m, fq, x, y);
                        else
                            tma_load_2d_pair(dst, m, fb, x, y);
                    };
                    // both CTAs' copies count on the even CTA's barrier, which
                    // expects the pair's bytes (its own arrive is the only one)
                    const uint32_t fb = CG == 2 ? mapa_shared(smem_u32(fq), 0) : 0u;
                    if (CG == 1)
                        mbar_expect_tx(fq, Cfg::kStageBytes);
                    else if (rank == 0)
                        mbar_expect_tx(fq, CG * Cfg::kStageBytes);
                    if constexpr (kAMN) {
                        load(sa, ma, m0, ka, fb);
                        load(sa + A_BYTES / 2, ma, m0 + 64, ka, fb);
                    } else {
                        load(sa, ma, ka, m0, fb);
                    }
                    if constexpr (kBMN) {
#pragma unroll
                        for (int i = 0; i < BN / CG / 64; ++i)
                            load(sa + A_BYTES + i * 8192, &tmB, nb0 + 64 * i, ka, fb);
                    } else {
                        load(sa + A_BYTES, mb, ka, nb0, fb);
                    }
                }
                __syncwarp();
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
        }
        if (!ok) {  // let copies already in flight land before the CTA exits
            const uint64_t t0 = globaltimer();
            while (globaltimer() - t0 < 50000ull) {
            }
        }
    } else if (warp == 2) {
        if (epi_load) {
            if (elect_one()) tma_prefetch(&tmC);
            __syncwarp();
            // ------------------------------------------------ epilogue-input loader:
            // per tile, the bias (and sigma) slice by bulk copy and, for in-place
            // epilogues, the output tile by TMA, as soon as the epilogue has
            // released the slot (independent of the A/B stream of warp 0)
            bool ok = true;
            int i = 0;
            for (int t = cta0; t < total && ok; t += ncta, ++i) {
                const int m0 = (lin(t) % p.num_m) * (BM * CG) + static_cast<int>(rank) * BM;
                const int n0 = tile_n0<BN, Cfg::kKV>(p, lin(t));
                const int nb = min(BN, p.N - n0);
                const uint32_t vbytes = static_cast<uint32_t>(nb) * 4u;
                if constexpr (Cfg::kInPlace) {
                    // box by box, each as soon as the previous tile's copy of it has
                    // been stored; box 0 also brings this tile's vectors (buffer i & 1)
                    float* vdst = vec + (i & 1) * (Cfg::kVecBytes / 4);
                    // pool source: this CTA's 128 rows as one pool box, or -1; then
                    // lane g < 16 holds the pool row of the tile's 8-row group g, or -1
                    const int64_t bsrc = (Cfg::kPoolSrc && load_tile && m0 < p.M) ? p.box_src[m0 / BM] : -1;
                    const bool straddle = Cfg::kPoolSrc && load_tile && bsrc < 0;
                    int64_t gsrc = -1;
                    uint32_t good = 0;   // groups loaded by TMA (8-row boxes)
                    int hg = -1;         // first group the warp copies, its rows' pool rows below
                    int64_t hs0 = -1, hs1 = -1;
                    if (straddle) {
                        if (lane < 16 && m0 < p.M) gsrc = p.grp_src[m0 / 8 + static_cast<int>(lane)];
                        good = __ballot_sync(0xffffffffu, gsrc >= 0) & 0xFFFFu;
                        if (good != 0xFFFFu) {
                            hg = __ffs(static_cast<int>(~good & 0xFFFFu)) - 1;
                            const int r0 = 8 * hg + (static_cast<int>(lane) >> 3);
                            if (m0 + r0 < p.M) hs0 = p.src_row[m0 + r0];
                            if (m0 + r0 + 4 < p.M) hs1 = p.src_row[m0 + r0 + 4];
                        }
                    }
                    for (int b = 0; b < Cfg::kBoxes; ++b) {
                        if (!(ok = mbar_wait_warp(&epi_empty[b], (static_cast<uint32_t>(i) & 1u) ^ 1u, wc, 101)))
                            break;
                        const uint32_t vb =
                            (b == 0 && !Cfg::kVecGlobal) ? (has_bias ? vbytes : 0u) + (Cfg::kKV ? vbytes : 0u) : 0u;
                        if (straddle) {
                            // a tile across chunk boundaries: its contiguous 8-row groups
                            // by TMA, the others copied by the warp, then one arrival
                            const uint32_t bytes = static_cast<uint32_t>(__popc(good)) * 1024u + vb;
                            if (elect_one()) {
                                if (bytes) mbar_add_tx(&epi_full[b], bytes);
                                if (b == 0 && !Cfg::kVecGlobal) {
                                    if (has_bias) bulk_load(vdst, p.bias + n0, vbytes, &epi_full[0]);
                                    if constexpr (Cfg::kKV) bulk_load(vdst + BN, p.sigma + n0, vbytes, &epi_full[0]);
                                }
                            }
                            __syncwarp();
                            uint8_t* dstb = tile + b * 16384;
                            const int col0 = n0 + b * Cfg::kBoxCols;
                            for (int g = 0; g < 16; ++g) {
                                const int64_t s = __shfl_sync(0xffffffffu, gsrc, g);
                                if (s >= 0 && lane == 0)
                                    tma_load_2d(dstb + g * 1024, &p.tm_pool8, &epi_full[b], col0, static_cast<int>(s));
                            }
                            // each 16-byte chunk c of row r to r * 128 + ((c ^ (r & 7)) << 4),
                            // where TMA places it, by asynchronous copies that the barrier
                            // waits for; rows past the request are zero-filled
                            for (uint32_t bad = ~good & 0xFFFFu; bad; bad &= bad - 1) {
                                const int g = __ffs(static_cast<int>(bad)) - 1;
                                const int c = static_cast<int>(lane) & 7;
                                const int r0 = 8 * g + (static_cast<int>(lane) >> 3), r1 = r0 + 4;
                                int64_t s0 = hs0, s1 = hs1;
                                if (g != hg) {
                                    s0 = m0 + r0 < p.M ? p.src_row[m0 + r0] : -1;
                                    s1 = m0 + r1 < p.M ? p.src_row[m0 + r1] : -1;
                                }
                                cp_async16(dstb + r0 * 128 + ((c ^ (r0 & 7)) << 4),
                                           p.kv_pool + (s0 >= 0 ? s0 : 0) * p.N + col0 + c * 8, s0 >= 0 ? 16u : 0u);
                                cp_async16(dstb + r1 * 128 + ((c ^ (r1 & 7)) << 4),
                                           p.kv_pool + (s1 >= 0 ? s1 : 0) * p.N + col0 + c * 8, s1 >= 0 ? 16u : 0u);
                            }
                            if (good != 0xFFFFu) cp_async_mbar_arrive(&epi_full[b]);
                            __syncwarp();
                            if (elect_one()) mbar_arrive(&epi_full[b]);
                            __syncwarp();
                            continue;
                        }
                        const bool tma_tile = load_tile;
                        uint32_t bytes = (tma_tile ? (Cfg::kLoss ? 32768u : 16384u) : 0u) + vb;
                        if (elect_one()) {
                            if (bytes) mbar_expect_tx(&epi_full[b], bytes);
                            else mbar_arrive(&epi_full[b]);
                            if (Cfg::kPoolSrc && tma_tile) {
                                tma_load_2d(tile + b * 16384, &p.tm_pool, &epi_full[b], n0 + b * Cfg::kBoxCols,
                                            static_cast<int>(bsrc));
                            } else if (tma_tile) {
                                if constexpr (Cfg::kLoss) {
                                    tma_load_2d(tile + 2 * b * 16384, &tmC, &epi_full[b], n0 + b * Cfg::kBoxCols, m0);
                                    tma_load_2d(tile + (2 * b + 1) * 16384, &p.tm_joint, &epi_full[b],
                                                n0 + b * Cfg::kBoxCols, m0);
                                } else {
                                    tma_load_2d(tile + b * 16384, &tmC, &epi_full[b], n0 + b * Cfg::kBoxCols, m0);
                                }
                            }
                            if (b == 0 && !Cfg::kVecGlobal) {
                                if (has_bias) bulk_load(vdst, p.bias + n0, vbytes, &epi_full[0]);
                                if constexpr (Cfg::kKV) bulk_load(vdst + BN, p.sigma + n0, vbytes, &epi_full[0]);
                            }
                        }
                        __syncwarp();
                    }
                } else {
                    if (!(ok = mbar_wait_warp(epi_empty, (static_cast<uint32_t>(i) & 1u) ^ 1u, wc, 101)))
                        break;
                    if (elect_one()) {
                        mbar_expect_tx(epi_full, vbytes);
                        bulk_load(vec, second(n0) ? p.bias2 + (n0 - p.n_split) : p.bias + n0, vbytes,
                                  epi_full);
                    }
                    __syncwarp();
                }
            }
            if (!ok) {
                const uint64_t t0 = globaltimer();
                while (globaltimer() - t0 < 50000ull) {
                }
            }
        }
    } else if (warp == 3) {
        // ---------------------------------------------------- TMA store issuer
        // of the in-place epilogues: writes each box of the staged tile back
        // once the 256 epilogue threads have updated it, and hands the box back
        // to the loader when TMA has read it (the store-only epilogues issue
        // their own stores).  The bulk-group waits belong to the elected lane
        // that committed the stores.
        if constexpr (Cfg::kInPlace) {
            const bool leader = elect_one();
            bool ok = true;
            uint32_t pk = 0;   // in-place tiles so far
            for (int t = cta0; t < total && ok; t += ncta) {
                const int m0 = (lin(t) % p.num_m) * (BM * CG) + static_cast<int>(rank) * BM;
                const int n0 = tile_n0<BN, Cfg::kKV>(p, lin(t));
                const bool rows_in = m0 < p.M;   // a pair tile's second half may lie below M
                for (int b = 0; b < Cfg::kBoxes && ok; ++b) {
                    if (!(ok = mbar_wait_warp(&epi_done[b], pk & 1u, wc, 401))) break;
                    if (leader) {
                        if (rows_in && !Cfg::kDirect) {
                            tma_store_2d(&tmC, tile + b * 16384, n0 + b * Cfg::kBoxCols, m0);
                            tma_store_commit();
                            tma_store_wait_read0();
                        }
                        mbar_arrive(&epi_empty[b]);
                    }
                    __syncwarp();
                }
                ++pk;
            }
            if (leader) tma_store_wait0();
            __syncwarp();
        }
    } else if (warp == 1 && (CG == 1 || rank == 0)) {
        // ---------------------------------------------------- MMA issuer
        // (for a pair: the even CTA, issuing M = 256 MMAs over both CTAs'
        // shared memory and TMEM, committing to the barriers of both)
        // Stage descriptors: a K=16 step adds 32 bytes (2 units of 16 B) to the
        // start address of a K-major operand and 16 rows (2 KB) to an MN-major
        // one, a stage kStageBytes, the W operand A_BYTES.
        const uint64_t da0 = smem_desc(smem_u32(smem), kAMN ? 8192 : 16, 1024, SWZ_128B);
        const uint64_t db0 = smem_desc(smem_u32(smem + A_BYTES), kBMN ? 8192 : 16, 1024, SWZ_128B);
        constexpr uint64_t kStageStep = Cfg::kStageBytes >> 4;
        constexpr uint64_t kAK = kAMN ? (2048 >> 4) : 2, kBK = kBMN ? (2048 >> 4) : 2;
        uint32_t stage = 0, phase = 0, acc = 0, acc_phase = 0;
        bool ok = true;
        for (int t = cta0; t < total && ok; t += ncta) {
            if (!(ok = mbar_wait_warp(&tempty[acc], acc_phase ^ 1u, wc, 201))) break;
            tc_fence_after();
            const uint32_t d = tmem_base + acc * BN;
            int kbeg, kend;
            k_range(t, &kbeg, &kend);
            for (int kb = kbeg; kb < kend; ++kb) {
                if (!(ok = mbar_wait_warp(&full[stage], phase, wc, 202))) break;
                tc_fence_after();
                const uint64_t da = da0 + stage * kStageStep;
                const uint64_t dw = db0 + stage * kStageStep;
                if (elect_one()) {
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        if constexpr (CG == 2)
                            mma_bf16_ss2(d, da + kAK * k, dw + kBK * k, IDESC, (kb != kbeg || k != 0) ? 1u : 0u);
                        else
                            mma_bf16_ss(d, da + kAK * k, dw + kBK * k, IDESC, (kb != kbeg || k != 0) ? 1u : 0u);
                    }
                    if constexpr (CG == 2)
                        mma_commit2_mc(&empty[stage], 0x3);
                    else
                        mma_commit(&empty[stage]);
                }
                __syncwarp();
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            if (elect_one()) {
                if constexpr (CG == 2)
                    mma_commit2_mc(&tfull[acc], 0x3);
                else
                    mma_commit(&tfull[acc]);
            }
            __syncwarp();
            acc ^= 1u;
            if (acc == 0) acc_phase ^= 1u;
        }
        // all MMAs of this warp retire before TMEM can be released
        if (elect_one()) {
            if constexpr (CG == 2)
                mma_commit2(drain);
            else
                mma_commit(drain);
        }
        __syncwarp();
        mbar_wait_warp(drain, 0, wc, 203);
    } else if (warp == 1) {
        // pair: the odd CTA's MMA warp only took part in the TMEM allocation
    }
    } else {
        setmaxnreg_inc<kGemmRegsEpi>();
        // ---------------------------------------------------- epilogue (warps 4..11)
        const uint32_t quad = warp & 3u;                       // TMEM lanes 32 quad ..
        const int eg = (static_cast<int>(warp) - 4) >> 2;      // column group 0 / 1
        const int r = static_cast<int>(quad * 32 + lane);     // row inside the tile
        constexpr int ES = Cfg::kTileEsize;
        const float* vb = vec;             // bias slice of the tile
        const float* vs = vec + BN;        // sigma_delta slice (KV epilogues)
        // hand the accumulator buffer back to the issuing CTA's MMA warp
        auto release_acc = [&](uint64_t* bar) {
            if (CG == 2 && rank != 0)
                mbar_arrive_cluster(mapa_shared(smem_u32(bar), 0));
            else
                mbar_arrive(bar);
        };
        uint32_t acc = 0, acc_phase = 0, pk = 0;
        bool ok = true;
        int i = 0;
        for (int t = cta0; t < total && ok; t += ncta, ++i) {
            const int m0 = (lin(t) % p.num_m) * (BM * CG) + static_cast<int>(rank) * BM;
            const int n0 = tile_n0<BN, Cfg::kKV>(p, lin(t));
            // QKV: the rotation angles depend on (row, pair index) only: cos/sin
            // for every head of the tile, fetched while the MMAs still run
            constexpr int NP = (EPI == EPI_QKV_ROPE) ? 32 : 1;
            float cs[NP], sn[NP];
            if constexpr (EPI == EPI_QKV_ROPE) rope_angles<NP>(p, m0 + r, cs, sn);
            if constexpr (Cfg::kVecGlobal) {
                // the tile's bias and sigma slices (BN fp32 each, 128-byte lines)
                // into L1 while the MMAs still run
                constexpr int kLines = BN * 4 / 128;
                if (lane < kLines) {
                    if (has_bias) prefetch_l1(p.bias + n0 + lane * 32);
                    prefetch_l1(p.sigma + n0 + lane * 32);
                }
            }
            ok = mbar_wait(&tfull[acc], acc_phase, wc, 301);
            // in-place epilogues wait box by box below
            if (epi_load && !Cfg::kInPlace) ok = ok && mbar_wait(epi_full, static_cast<uint32_t>(i) & 1u, wc, 302);
            if constexpr (!Cfg::kInPlace) {
                // the group's 128 threads take the same path (named barriers follow)
                if (!(ok = named_bar_and(1 + eg, 128, ok))) break;
            } else if (!__all_sync(0xffffffffu, ok)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const int row = m0 + r;
            const bool row_ok = row < p.M;
            const uint32_t taddr = tmem_base + ((quad * 32u) << 16) + acc * BN;

            if constexpr (Cfg::kInPlace) {
                // output choices: a kept row (first chunk) leaves its stale value,
                // a zero output offset drops the stale value from the sum
                bool keep = false, zero = false;
                if constexpr (Cfg::kKV) {
                    keep = p.keep_chunk != nullptr && row_ok && __ldg(p.keep_chunk + row) == 0;
                    zero = p.kv_zero != 0 && !keep;
                }
                // where a repaired 16-column chunk goes: back into the staged tile
                // (stored in place by TMA), or straight to the token's row of its
                // (layer, K|V) plane in the paged target cache
                uint16_t* prow = nullptr;
                if constexpr (Cfg::kPaged) {
                    const int64_t slot = row_ok ? __ldg(p.slot + row) : -1;
                    if (slot >= 0 && slot < p.num_slots) {
                        const int plane = n0 / p.seg_width;
                        prow = p.paged + (static_cast<int64_t>(plane) * p.num_slots + slot) * p.seg_width +
                               (n0 - plane * p.seg_width);
                    } else if (slot >= p.num_slots) {
                        report(p.status, CR_DEV_INDEX, 410);
                    }
                }
                // training head: this row's gradient row, loss weight and r^2 sum
                // over this group's columns of the tile (chunks in column order)
                uint16_t* dzrow = nullptr;
                float lsc = 0.0f, lsq = 0.0f;
                if constexpr (Cfg::kLoss) {
                    if (row_ok) {
                        dzrow = p.loss_dz + static_cast<int64_t>(row) * p.N + n0;
                        lsc = __ldg(p.row_scale + row);
                    }
                }
                auto put16 = [&](int col, const float* v) {
                    if constexpr (Cfg::kPaged) {
                        if (prow) store16_bf16_global(prow + col, v);
                    } else if constexpr (Cfg::kLoss) {
                        if (dzrow) {
                            float d[16];
#pragma unroll
                            for (int q = 0; q < 16; ++q) {
                                lsq = fmaf(v[q], v[q], lsq);
                                d[q] = lsc * v[q];
                            }
                            store16_bf16_global(dzrow + col, d);
                        }
                    } else {
                        store16_tile<ES>(tile, r, col, v);
                    }
                };
                // this tile's vectors, and the per-box hand-over: box b of the
                // staged tile is waited for before it is read and released to the
                // store as soon as both groups have written their part of it
                const float* vbt = Cfg::kVecGlobal ? p.bias + n0 : vb + (i & 1) * (Cfg::kVecBytes / 4);
                const float* vst = Cfg::kVecGlobal ? p.sigma + n0 : vbt + BN;
                auto wait_box = [&](int b) -> bool {
                    const bool w = mbar_wait(&epi_full[b], static_cast<uint32_t>(i) & 1u, wc, 302);
                    return __all_sync(0xffffffffu, w);
                };
                auto done_box = [&](int b) {
                    fence_async_smem();
                    mbar_arrive(&epi_done[b]);
                };
                if constexpr (Cfg::kLoss) {
                    // r = z + b - (joint - stale) / sigma_Delta, the stale and joint
                    // values from column box bx's two staged bf16 boxes; each group
                    // takes one half of the box's columns
                    constexpr int HALF = Cfg::kBoxCols / 2;
                    for (int bx = 0; bx < Cfg::kBoxes && ok; ++bx) {
                        if (!(ok = wait_box(bx))) break;
                        const uint8_t* sbox = tile + 2 * bx * 16384;
                        for (int c = bx * Cfg::kBoxCols + eg * HALF; c < bx * Cfg::kBoxCols + (eg + 1) * HALF;
                             c += 16) {
                            float a[16], st16[16], jt16[16], bv[16], sd[16];
                            __syncwarp();
                            tmem_ld16(taddr + c, a);
                            load16_bf16_smem(sbox, r, c - bx * Cfg::kBoxCols, st16);
                            load16_bf16_smem(sbox + 16384, r, c - bx * Cfg::kBoxCols, jt16);
                            if (has_bias) {
                                vec16(vbt, c, bv);
                            } else {
#pragma unroll
                                for (int q = 0; q < 16; ++q) bv[q] = 0.0f;
                            }
                            vec16(vst, c, sd);
                            tmem_wait_ld();
#pragma unroll
                            for (int q = 0; q < 16; ++q) {
                                const float nt = -(jt16[q] - st16[q]) / sd[q];
                                a[q] = (a[q] + bv[q]) + nt;
                            }
                            put16(c, a);
                        }
                        done_box(bx);
                    }
                } else if (Cfg::kKV && p.rope_on) {
                    // R_M pairs (d, d + d_h/2) live inside one d_h-wide segment, which
                    // spans d_h / kBoxCols boxes; each group takes half of its pairs
                    const int dh = p.rope_dim;
                    const int nbx = dh / Cfg::kBoxCols;
                    const float pr = row_ok ? static_cast<float>(__ldg(p.pos + row)) : 0.0f;
                    for (int s0 = 0; s0 < BN && ok; s0 += dh) {
                        const int bx0 = s0 / Cfg::kBoxCols;
                        for (int b = bx0; b < bx0 + nbx && ok; ++b) ok = wait_box(b);
                        if (!ok) break;
                        const int gseg = (n0 + s0) / dh;
                        const bool rot = ((gseg / p.n_kv_heads) & 1) == 0;
                        for (int j = eg * (dh / 4); j < (eg + 1) * (dh / 4); j += 16) {
                            float a[16], b[16], ka[16], kb[16], sa_[16], sb_[16], ba[16], bb[16];
                            const int ta = s0 + j, tb = s0 + dh / 2 + j;
                            __syncwarp();
                            tmem_ld16(taddr + ta, a);
                            tmem_ld16(taddr + tb, b);
                            if (zero) {
#pragma unroll
                                for (int q = 0; q < 16; ++q) ka[q] = kb[q] = 0.0f;
                            } else {
                                load16_tile<ES>(tile, r, ta, ka);
                                load16_tile<ES>(tile, r, tb, kb);
                            }
                            vec16(vst, ta, sa_);
                            vec16(vst, tb, sb_);
                            if (has_bias) {
                                vec16(vbt, ta, ba);
                                vec16(vbt, tb, bb);
                            } else {
#pragma unroll
                                for (int q = 0; q < 16; ++q) ba[q] = bb[q] = 0.0f;
                            }
                            tmem_wait_ld();
                            if (!keep) {
#pragma unroll
                                for (int q = 0; q < 16; ++q) {
                                    ka[q] = fmaf(sa_[q], a[q] + ba[q], ka[q]);
                                    kb[q] = fmaf(sb_[q], b[q] + bb[q], kb[q]);
                                }
                            }
                            if (rot) {
                                if (p.rope_table)
                                    rotate16_tab(ka, kb, p.rope_table, p.M, row_ok ? row : 0, j);
                                else
                                    rotate16(ka, kb, pr, p.inv_freq, j);
                            }
                            put16(ta, ka);
                            put16(tb, kb);
                        }
                        for (int b = bx0; b < bx0 + nbx; ++b) done_box(b);
                    }
                } else {
                    // box by box; each group takes one half of the box's columns
                    constexpr int HALF = Cfg::kBoxCols / 2;
                    for (int bx = 0; bx < Cfg::kBoxes && ok; ++bx) {
                      if (!(ok = wait_box(bx))) break;
                      for (int c = bx * Cfg::kBoxCols + eg * HALF; c < bx * Cfg::kBoxCols + (eg + 1) * HALF;
                           c += 16) {
                        float a[16], k[16], bv[16];
                        __syncwarp();
                        tmem_ld16(taddr + c, a);
                        if (zero) {
#pragma unroll
                            for (int q = 0; q < 16; ++q) k[q] = 0.0f;
                        } else {
                            load16_tile<ES>(tile, r, c, k);
                        }
                        if (has_bias) {
                            vec16(vbt, c, bv);
                        } else {
#pragma unroll
                            for (int q = 0; q < 16; ++q) bv[q] = 0.0f;
                        }
                        tmem_wait_ld();
                        if (!keep) {
                            float sv[16];
                            vec16(vst, c, sv);
#pragma unroll
                            for (int q = 0; q < 16; ++q) k[q] = fmaf(sv[q], a[q] + bv[q], k[q]);
                        }
                        put16(c, k);
                      }
                      done_box(bx);
                    }
                }
                if (!ok) break;
                if constexpr (Cfg::kLoss) {
                    if (row_ok) p.loss_part[static_cast<int64_t>((n0 / BN) * 2 + eg) * p.M + row] = lsq;
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) release_acc(&tempty[acc]);
                ++pk;
            } else {
                // store-only epilogues: one 128 B-wide box of columns at a time,
                // into alternating staging buffers
                constexpr int PC = Cfg::kBoxCols;
                // one thread of each group issues (and waits on) its stores; the
                // group meets at a named barrier before and after writing a box
                const bool glead = (quad == 0 && lane == 0);
                // boxes alternate between the groups; each group cycles its own
                // kGroupBufs staging buffers (pk counts this group's boxes)
                for (int k = eg; k < Cfg::kBoxes && ok; k += 2, ++pk) {
                    constexpr uint32_t GB = Cfg::kGroupBufs;
                    const uint32_t bsel = static_cast<uint32_t>(eg) * GB + (pk % GB);
                    // the group's leader stored this buffer GB boxes ago: once that
                    // store has read it, the group may rewrite it
                    if (glead && pk >= GB) {
                        if constexpr (GB == 1) tma_store_wait_read0();
                        else tma_store_wait_read<1>();
                    }
                    named_bar_sync(1 + eg, 128);
                    uint8_t* buf = tile + bsel * 16384;
                    const int c0 = k * PC;
                    if constexpr (EPI == EPI_QKV_ROPE) {
                        const int hd = p.rope_dim;
#pragma unroll
                        for (int j = 0; j < NP; j += 16) {
                            if (j >= hd / 2) break;
                            for (int h0 = c0; h0 < c0 + PC; h0 += hd) {
                                const bool rot = (n0 + h0) < p.rope_cols;
                                float a[16], b[16];
                                const int ta = h0 + j, tb = h0 + hd / 2 + j;
                                __syncwarp();
                                tmem_ld16(taddr + ta, a);
                                tmem_ld16(taddr + tb, b);
                                tmem_wait_ld();
                                if (has_bias) {
                                    float ba[16], bb[16];
                                    vec16(vb, ta, ba);
                                    vec16(vb, tb, bb);
#pragma unroll
                                    for (int q = 0; q < 16; ++q) {
                                        a[q] += ba[q];
                                        b[q] += bb[q];
                                    }
                                }
                                if (rot) {
#pragma unroll
                                    for (int q = 0; q < 16; ++q) {
                                        const float x = a[q], y = b[q];
                                        a[q] = x * cs[j + q] - y * sn[j + q];
                                        b[q] = y * cs[j + q] + x * sn[j + q];
                                    }
                                }
                                store16_tile<ES>(buf, r, ta - c0, a);
                                store16_tile<ES>(buf, r, tb - c0, b);
                            }
                        }
                    } else {
                        for (int c = c0; c < c0 + PC; c += 16) {
                            float v[16];
                            __syncwarp();
                            tmem_ld16(taddr + c, v);
                            tmem_wait_ld();
                            if (has_bias) {
                                float bv[16];
                                vec16(vb, c, bv);
#pragma unroll
                                for (int q = 0; q < 16; ++q) v[q] += bv[q];
                            }
                            if constexpr (EPI == EPI_GELU_BF16) {
#pragma unroll
                                for (int q = 0; q < 16; q += 2) gelu2(v[q], v[q + 1]);
                            }
                            store16_tile<ES>(buf, r, c - c0, v);
                        }
                    }
                    fence_async_smem();
                    named_bar_sync(1 + eg, 128);
                    if (glead) {
                        if (m0 < p.M) {
                            const bool g2 = second(n0);
                            const int x = (g2 ? n0 - p.n_split : n0) + k * PC, y = m0 + tile_part(p, t) * p.M;
                            if constexpr (Cfg::kReduce)
                                tma_reduce_add_2d(&tmC, buf, x, y);
                            else
                                tma_store_2d(g2 ? &p.tm_c2 : &tmC, buf, x, y);
                        }
                        tma_store_commit();
                    }
                }
                // this group has read its columns of the TMEM buffer
                tc_fence_before();
                __syncwarp();
                if (ok && lane == 0) release_acc(&tempty[acc]);
                if (ok && glead && epi_load) mbar_arrive(epi_empty);
            }
            acc ^= 1u;
            if (acc == 0) acc_phase ^= 1u;
        }
        if constexpr (!Cfg::kInPlace) {
            if ((warp & 3u) == 0 && lane == 0) tma_store_wait0();
        }
    }
    tc_fence_before();
    if constexpr (CG == 2)
        cluster_sync();   // no pair traffic (MMAs, remote arrives) is left in flight
    else
        __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        if constexpr (CG == 2)
            tmem_dealloc2(tmem_base, Cfg::kTmemCols);
        else
            tmem_dealloc(tmem_base, Cfg::kTmemCols);
    }
}

template <int BN, int EPI, int CG, int LAY = LAY_KK>
cr_status launch_bn(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc,
                    const GemmParams& p, cudaStream_t st) {
    using Cfg = GemmCfg<BN, EPI, CG>;
    auto kern = gemm_kernel<BN, EPI, CG, LAY>;
    static unsigned long long attr_done = 0;   // one per template instantiation
    const cr_status sa = ensure_smem_attr(kern, static_cast<int>(Cfg::kSmemBytes), &attr_done);
    if (sa != CR_OK) return sa;
    const int tiles = p.num_m * p.num_n;
    // the epilogue warpgroups raise their register budget inside the kernel,
    // which only completes if the launch reserved the 168 per thread assumed
    static int regs_ok = -1;
    int rok = __atomic_load_n(&regs_ok, __ATOMIC_ACQUIRE);
    if (rok < 0) {
        cudaFuncAttributes fa;
        const cr_status sf = cuda_check(cudaFuncGetAttributes(&fa, kern));
        if (sf != CR_OK) return sf;
        rok = (fa.numRegs >= static_cast<int>(kGemmRegsLaunch) && fa.maxThreadsPerBlock >= kGemmThreads)
                  ? 1 : 0;
        __atomic_store_n(&regs_ok, rok, __ATOMIC_RELEASE);
    }
    if (!rok) return CR_ERR_UNSUPPORTED;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.blockDim = dim3(kGemmThreads, 1, 1);
    cfg.dynamicSmemBytes = Cfg::kSmemBytes;
    cfg.stream = st;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see launch_pdl
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if constexpr (CG == 2) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = 2;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
        // persistent: as many pairs as can be resident at once (asked once)
        static int max_pairs = 0;
        int mp = __atomic_load_n(&max_pairs, __ATOMIC_ACQUIRE);
        if (mp <= 0) {
            cfg.gridDim = dim3(2 * (num_sms() / 2), 1, 1);
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) {
                (void)cudaGetLastError();
                n = num_sms() / 2;
            }
            mp = n;
            __atomic_store_n(&max_pairs, mp, __ATOMIC_RELEASE);
        }
        cfg.gridDim = dim3(2 * (tiles < mp ? tiles : mp), 1, 1);
    } else {
        cfg.gridDim = dim3(tiles < num_sms() ? tiles : num_sms(), 1, 1);
    }
    return cuda_check(cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, p));
}

// Every GEMM runs on CTA pairs: 256-row tiles whose MMAs span two SMs, each
// SM loading its own 128 rows of A and half of the W tile.
constexpr int kCG = 2;

}  // namespace

cr_status launch_gemm(const uint16_t* A, int64_t lda, const uint16_t* W, int64_t M, int64_t N,
                      int64_t K, int epi, GemmParams p, void* kv_base, int64_t ld_kv,
                      cudaStream_t st, const uint16_t* A_lo) {
    const bool kv = (epi == EPI_KV_BF16 || epi == EPI_KV_F32 || epi == EPI_KV_PAGED || epi == EPI_KV_LOSS ||
                     epi == EPI_KV_POOL);
    const bool f32_tile = (epi == EPI_KV_F32 || epi == EPI_ADD_F32);
    // Tile width.  Per 64-deep k-block a CTA of a pair moves 32 KB + 128 BN
    // bytes through shared memory (TMA writes and MMA operand reads of its A
    // rows and W half) at ~128 B/clock, and its MMAs take 2 BN clocks, so a
    // tile costs ~(256 + BN) clocks per k-block for BN <= 256; a launch takes
    // ceil(tiles / pairs) rounds.  Pick the instantiated width with the least
    // rounds x (256 + BN) (ties: the wider tile).  The width does not change
    // any output element's K order, so results do not depend on it.
    int BN;
    if (kv) {
        BN = (epi == EPI_KV_F32 || epi == EPI_KV_LOSS) ? 128 : 256;
    } else {
        const int64_t pairs = num_sms() / kCG > 0 ? num_sms() / kCG : 1;
        const int64_t mt = (M + BM * kCG - 1) / (BM * kCG);
        static const int kF32W[] = {160, 128};
        static const int kBf16W[] = {256, 192, 128};
        const int* cand = f32_tile ? kF32W : kBf16W;
        const int nc = f32_tile ? 2 : 3;
        BN = cand[0];
        int64_t best = -1;
        for (int i = 0; i < nc; ++i) {
            const int w = cand[i];
            if (epi == EPI_QKV_ROPE && (p.rope_dim <= 0 || w % p.rope_dim != 0)) continue;
            const int64_t tiles = mt * ((N + w - 1) / w);
            const int64_t cost = ((tiles + pairs - 1) / pairs) * (256 + w);
            if (best < 0 || cost < best) {
                best = cost;
                BN = w;
            }
        }
    }
    if (kv && (N % BN) != 0) return CR_ERR_UNSUPPORTED;
    if (epi == EPI_QKV_ROPE && (BN % p.rope_dim) != 0) return CR_ERR_UNSUPPORTED;
    if (p.bias && (N % 4) != 0) return CR_ERR_UNSUPPORTED;   // bias slices are 16-byte bulk copies
    p.M = static_cast<int32_t>(M);
    p.N = static_cast<int32_t>(N);
    p.K = static_cast<int32_t>(K);
    p.num_m = static_cast<int32_t>((M + BM * kCG - 1) / (BM * kCG));
    p.num_n = static_cast<int32_t>((N + BN - 1) / BN);
    p.split_k = 1;
    p.n_fast = 0;
    p.n_split = 0;
    if (kv && p.col_block > 0) {
        // output choice: half of the column blocks, each a whole number of tiles
        if (p.col_block % BN != 0 || N % (2 * static_cast<int64_t>(p.col_block)) != 0)
            return CR_ERR_UNSUPPORTED;
        p.num_n = static_cast<int32_t>(N / 2 / BN);
    } else {
        p.col_block = 0;
    }
    CUtensorMap ta, tb, tc;
    if (!make_tmap_2d(&ta, A, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, K, M, lda * 2, BK, BM,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    p.split_kb = 0;
    if (A_lo) {
        // columns past K read as zeros in both terms (TMA bounds), so the two
        // k-loops line up with the same W k-blocks
        if (!make_tmap_2d(&p.tm_alo, A_lo, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, K, M, lda * 2, BK, BM,
                          CU_TENSOR_MAP_SWIZZLE_128B))
            return CR_ERR_INVALID_ARG;
        p.split_kb = static_cast<int32_t>((K + BK - 1) / BK);
    }
    if (!make_tmap_2d(&tb, W, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, K, N, K * 2, BK, BN / kCG,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    // output (staged) tile map: bf16 boxes of 64 or fp32 boxes of 32 columns
    const bool f32_out = f32_tile || epi == EPI_F32;
    void* out_base = kv ? kv_base : p.out;
    const int64_t ld_out = kv ? ld_kv : p.ldo;
    if (!make_tmap_2d(&tc, out_base,
                      f32_out ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                      N, M, ld_out * (f32_out ? 4 : 2), f32_out ? 32 : 64, BM,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    switch (epi) {
        case EPI_BF16:
            return BN == 256   ? launch_bn<256, EPI_BF16, kCG>(ta, tb, tc, p, st)
                   : BN == 192 ? launch_bn<192, EPI_BF16, kCG>(ta, tb, tc, p, st)
                               : launch_bn<128, EPI_BF16, kCG>(ta, tb, tc, p, st);
        case EPI_GELU_BF16:
            return BN == 256   ? launch_bn<256, EPI_GELU_BF16, kCG>(ta, tb, tc, p, st)
                   : BN == 192 ? launch_bn<192, EPI_GELU_BF16, kCG>(ta, tb, tc, p, st)
                               : launch_bn<128, EPI_GELU_BF16, kCG>(ta, tb, tc, p, st);
        case EPI_ADD_F32:
            return BN == 160 ? launch_bn<160, EPI_ADD_F32, kCG>(ta, tb, tc, p, st)
                             : launch_bn<128, EPI_ADD_F32, kCG>(ta, tb, tc, p, st);
        case EPI_F32:
            return BN == 256   ? launch_bn<256, EPI_F32, kCG>(ta, tb, tc, p, st)
                   : BN == 192 ? launch_bn<192, EPI_F32, kCG>(ta, tb, tc, p, st)
                               : launch_bn<128, EPI_F32, kCG>(ta, tb, tc, p, st);
        case EPI_QKV_ROPE:
            return BN == 256   ? launch_bn<256, EPI_QKV_ROPE, kCG>(ta, tb, tc, p, st)
                   : BN == 192 ? launch_bn<192, EPI_QKV_ROPE, kCG>(ta, tb, tc, p, st)
                               : launch_bn<128, EPI_QKV_ROPE, kCG>(ta, tb, tc, p, st);
        case EPI_KV_BF16:
            return launch_bn<256, EPI_KV_BF16, kCG>(ta, tb, tc, p, st);
        case EPI_KV_F32:
            return launch_bn<128, EPI_KV_F32, kCG>(ta, tb, tc, p, st);
        case EPI_KV_LOSS:
            if (!p.loss_dz || !p.row_scale || !p.loss_part || !p.loss_joint || !p.sigma) return CR_ERR_INVALID_ARG;
            if (!make_tmap_2d(&p.tm_joint, p.loss_joint, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, N, M, ld_kv * 2, 64,
                              BM, CU_TENSOR_MAP_SWIZZLE_128B))
                return CR_ERR_INVALID_ARG;
            return launch_bn<128, EPI_KV_LOSS, kCG>(ta, tb, tc, p, st);
        case EPI_KV_PAGED:
            if (p.seg_width <= 0 || p.seg_width % 256 != 0 || p.num_slots < 1) return CR_ERR_UNSUPPORTED;
            return launch_bn<256, EPI_KV_PAGED, kCG>(ta, tb, tc, p, st);
        case EPI_KV_POOL:
            if (!p.kv_pool || !p.src_row || !p.box_src || !p.grp_src) return CR_ERR_INVALID_ARG;
            return launch_bn<256, EPI_KV_POOL, kCG>(ta, tb, tc, p, st);
        default:
            return CR_ERR_INVALID_ARG;
    }
}

namespace {
// C [M, N] (row stride ldc) = (or += with accumulate) the sum over u < s of
// part[u] ([M, N] slices, contiguous), in order u = 0, 1, ..: the split-K parts
// of one product, four columns per thread.
__global__ void __launch_bounds__(256)
    splitk_reduce_kernel(const float* __restrict__ part, int s, int64_t M, int64_t N, float* C, int64_t ldc,
                         int accumulate) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t n4 = N >> 2, total = M * n4;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t m = i / n4, c = (i - m * n4) << 2;
        float4 acc = *reinterpret_cast<const float4*>(part + m * N + c);
        for (int u = 1; u < s; ++u) {
            const float4 v = *reinterpret_cast<const float4*>(part + (u * M + m) * N + c);
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
        float4* dst = reinterpret_cast<float4*>(C + m * ldc + c);
        if (accumulate) {
            const float4 o = *dst;
            acc.x += o.x;
            acc.y += o.y;
            acc.z += o.z;
            acc.w += o.w;
        }
        *dst = acc;
    }
}
}  // namespace

cr_status launch_gemm_pair(const GemmProduct& a, const GemmProduct& b, int64_t M, GemmParams p,
                           cudaStream_t st) {
    constexpr int BN = 256;
    if (M < 1 || a.N < 1 || b.N < 1 || a.K < 1 || b.K < 1) return CR_ERR_INVALID_ARG;
    // tiles of 256 columns must not straddle the two products, and the tile's
    // vectors come from one bias array or none
    if (a.N % BN != 0 || (a.bias == nullptr) != (b.bias == nullptr) || a.N + b.N > (1 << 30)) {
        GemmParams pa = p;
        pa.bias = a.bias;
        pa.out = a.out;
        pa.ldo = a.ldo;
        const cr_status s = launch_gemm(a.A, a.lda, a.W, M, a.N, a.K, EPI_F32, pa, nullptr, 0, st, a.A_lo);
        if (s != CR_OK) return s;
        GemmParams pb = p;
        pb.bias = b.bias;
        pb.out = b.out;
        pb.ldo = b.ldo;
        return launch_gemm(b.A, b.lda, b.W, M, b.N, b.K, EPI_F32, pb, nullptr, 0, st, b.A_lo);
    }
    if ((b.bias && (b.N % 4) != 0)) return CR_ERR_UNSUPPORTED;   // bias slices are 16-byte bulk copies
    p.M = static_cast<int32_t>(M);
    p.N = static_cast<int32_t>(a.N + b.N);
    p.K = static_cast<int32_t>(a.K);
    p.K2 = static_cast<int32_t>(b.K);
    p.num_m = static_cast<int32_t>((M + BM * kCG - 1) / (BM * kCG));
    p.num_n = static_cast<int32_t>((a.N + b.N + BN - 1) / BN);
    p.split_k = 1;
    p.n_fast = 0;
    p.col_block = 0;
    p.bgroup_rows = 0;
    p.n_split = static_cast<int32_t>(a.N);
    p.bias = a.bias;
    p.bias2 = b.bias;
    p.out = a.out;
    p.ldo = a.ldo;
    const auto BF = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const auto SW = CU_TENSOR_MAP_SWIZZLE_128B;
    CUtensorMap ta, tb, tc;
    // columns past K read as zeros in both terms (TMA bounds)
    if (!make_tmap_2d(&ta, a.A, BF, a.K, M, a.lda * 2, BK, BM, SW) ||
        !make_tmap_2d(&tb, a.W, BF, a.K, a.N, a.K * 2, BK, BN / kCG, SW) ||
        !make_tmap_2d(&tc, a.out, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.N, M, a.ldo * 4, 32, BM, SW) ||
        !make_tmap_2d(&p.tm_a2, b.A, BF, b.K, M, b.lda * 2, BK, BM, SW) ||
        !make_tmap_2d(&p.tm_b2, b.W, BF, b.K, b.N, b.K * 2, BK, BN / kCG, SW) ||
        !make_tmap_2d(&p.tm_c2, b.out, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, b.N, M, b.ldo * 4, 32, BM, SW))
        return CR_ERR_INVALID_ARG;
    p.split_kb = 0;
    if (a.A_lo) {
        if (!make_tmap_2d(&p.tm_alo, a.A_lo, BF, a.K, M, a.lda * 2, BK, BM, SW)) return CR_ERR_INVALID_ARG;
        p.split_kb = static_cast<int32_t>((a.K + BK - 1) / BK);
    }
    p.split_kb2 = 0;
    if (b.A_lo) {
        if (!make_tmap_2d(&p.tm_alo2, b.A_lo, BF, b.K, M, b.lda * 2, BK, BM, SW)) return CR_ERR_INVALID_ARG;
        p.split_kb2 = static_cast<int32_t>((b.K + BK - 1) / BK);
    }
    return launch_bn<BN, EPI_F32, kCG, LAY_KK2>(ta, tb, tc, p, st);
}

cr_status launch_gemm_lay(const uint16_t* A, int64_t lda, int lay, const uint16_t* W, int64_t ldw,
                          int64_t M, int64_t N, int64_t K, int epi, GemmParams p, cudaStream_t st,
                          float* scratch, size_t scratch_bytes) {
    if (lay != LAY_KM && lay != LAY_MM) return CR_ERR_INVALID_ARG;
    if (epi != EPI_F32 && epi != EPI_ADD_F32) return CR_ERR_UNSUPPORTED;
    if (M < 1 || N < 1 || K < 1 || (N % 64) != 0 || (lay == LAY_MM && (M % 64) != 0))
        return CR_ERR_UNSUPPORTED;
    // Tile width as in launch_gemm (rounds x (256 + BN)); an MN-major W half is
    // whole 64-column boxes, so 256 or 128 (the accumulating form: 128).
    int BN = 128;
    if (epi == EPI_F32 && p.bgroup_rows == 0) {
        const int64_t pairs = num_sms() / kCG > 0 ? num_sms() / kCG : 1;
        const int64_t mt = (M + BM * kCG - 1) / (BM * kCG);
        const int64_t c256 = ((mt * ((N + 255) / 256) + pairs - 1) / pairs) * (256 + 256);
        const int64_t c128 = ((mt * ((N + 127) / 128) + pairs - 1) / pairs) * (256 + 128);
        BN = c256 <= c128 ? 256 : 128;
    }
    p.M = static_cast<int32_t>(M);
    p.N = static_cast<int32_t>(N);
    p.K = static_cast<int32_t>(K);
    p.num_m = static_cast<int32_t>((M + BM * kCG - 1) / (BM * kCG));
    p.num_n = static_cast<int32_t>((N + BN - 1) / BN);
    p.col_block = 0;
    p.split_kb = 0;
    p.split_k = 1;
    p.n_split = 0;
    // Split-K: when the tiles fill the CTA pairs poorly (the last round partly
    // empty), cut each tile's k-loop into s parts, each written to its own fp32
    // slice of the scratch and summed in a fixed order by a second kernel.  s
    // minimises rounds(s) x (tile time / s + a fixed cost per round for the
    // pipeline's fill and the epilogue's drain) + the sum's traffic, with every
    // part at least 64 k-blocks (measured on the training step's shapes: shorter
    // parts lose more to their fill, drain and sum than the idle CTA pairs cost;
    // the head's dX product, K = 65536, gains 30 % from 8 parts).
    const int64_t pairs = num_sms() / kCG > 0 ? num_sms() / kCG : 1;
    const int64_t tiles = static_cast<int64_t>(p.num_m) * p.num_n;
    const int64_t nkb = (K + BK - 1) / BK;
    // (whole 128-row boxes only: a part's rows must not spill into the next slice)
    if (scratch && p.bgroup_rows == 0 && M % BM == 0) {
        const double tile_us = static_cast<double>(nkb) * (256 + BN) / 1.9e3;   // ~1.9 GHz
        const double round_us = 6.0;
        double best = static_cast<double>((tiles + pairs - 1) / pairs) * (tile_us + round_us);
        for (int sk = 2; sk <= 8; sk *= 2) {
            const int64_t kp = (nkb + sk - 1) / sk;
            if (kp < 64 || (sk - 1) * kp >= nkb) break;
            const size_t need = static_cast<size_t>(sk) * M * N * 4;
            if (need > scratch_bytes) break;
            const double t = static_cast<double>((tiles * sk + pairs - 1) / pairs) * (tile_us / sk + round_us) +
                             static_cast<double>(need + static_cast<size_t>(M) * N * 4 * (epi == EPI_ADD_F32 ? 2 : 1)) /
                                 6.0e6;   // bytes at ~6 TB/s, in microseconds
            if (t < best * 0.95) {
                best = t;
                p.split_k = sk;
            }
        }
    }
    // an A operand far larger than L2 is walked once: column tiles fastest
    p.n_fast = (p.bgroup_rows == 0 && p.num_n > 1 && static_cast<double>(M) * K * 2 > 64e6) ? 1 : 0;
    float* const C = static_cast<float*>(p.out);
    const int64_t ldc = p.ldo;
    if (p.split_k > 1) {
        p.out = scratch;
        p.ldo = N;
    }
    if (p.bgroup_rows > 0) {
        // grouped rows: one column block per tile, the W block of the tile's group
        if (p.bgroup_rows % (BM * kCG) != 0 || N != BN) return CR_ERR_UNSUPPORTED;
        p.num_n = 1;
    }
    CUtensorMap ta, tb, tc;
    const bool amn = (lay == LAY_MM);
    if (!make_tmap_2d(&ta, A, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, amn ? M : K, amn ? K : M, lda * 2,
                      amn ? 64 : BK, amn ? BK : BM, CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    const int64_t wcols = p.bgroup_rows > 0 ? ldw : N;   // grouped: W blocks of every group
    if (!make_tmap_2d(&tb, W, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, wcols, K, ldw * 2, 64, BK,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    if (!make_tmap_2d(&tc, p.out, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, N, M * p.split_k, p.ldo * 4, 32, BM,
                      CU_TENSOR_MAP_SWIZZLE_128B))
        return CR_ERR_INVALID_ARG;
    cr_status s;
    if (p.split_k > 1) {
        // the parts are plain fp32 products; the sum adds into C for EPI_ADD_F32
        s = amn ? (BN == 256 ? launch_bn<256, EPI_F32, kCG, LAY_MM>(ta, tb, tc, p, st)
                             : launch_bn<128, EPI_F32, kCG, LAY_MM>(ta, tb, tc, p, st))
                : (BN == 256 ? launch_bn<256, EPI_F32, kCG, LAY_KM>(ta, tb, tc, p, st)
                             : launch_bn<128, EPI_F32, kCG, LAY_KM>(ta, tb, tc, p, st));
        if (s != CR_OK) return s;
        const int64_t n4 = M * (N / 4);
        int64_t blocks = (n4 + 255) / 256;
        if (blocks > static_cast<int64_t>(num_sms()) * 16) blocks = static_cast<int64_t>(num_sms()) * 16;
        return launch_pdl(splitk_reduce_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st,
                          static_cast<const float*>(scratch), static_cast<int>(p.split_k), M, N, C, ldc,
                          epi == EPI_ADD_F32 ? 1 : 0);
    }
    if (epi == EPI_ADD_F32)
        return amn ? launch_bn<128, EPI_ADD_F32, kCG, LAY_MM>(ta, tb, tc, p, st)
                   : launch_bn<128, EPI_ADD_F32, kCG, LAY_KM>(ta, tb, tc, p, st);
    if (amn)
        return BN == 256 ? launch_bn<256, EPI_F32, kCG, LAY_MM>(ta, tb, tc, p, st)
                         : launch_bn<128, EPI_F32, kCG, LAY_MM>(ta, tb, tc, p, st);
    return BN == 256 ? launch_bn<256, EPI_F32, kCG, LAY_KM>(ta, tb, tc, p, st)
                     : launch_bn<128, EPI_F32, kCG, LAY_KM>(ta, tb, tc, p, st);
}

}  // namespace cr
