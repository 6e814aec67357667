// Backward of the private branch on the 5th-generation tensor cores (G2,
// Sec. 2.2; Sec. 3.2 trains the private experts and the private router only).
// Three persistent grouped GEMM launches over the private experts, each in the
// TMA -> shared memory -> tcgen05.mma -> TMEM -> epilogue pipeline of the
// forward's expert GEMMs:
//
//   bwd_rows_tc_kernel<kRowsZ>    rows of an expert as M, K = H:
//     Z = D W_down                  (D: the rows' upstream gradients; W_down read
//                                    MN-major; so dL/da = w Z) -> BF16
//   bwd_rows_tc_kernel<kRowsGU>   rows of an expert as M, K = H:
//     G = A W_gate^T, U = A W_up^T  (A: the expert's dispatched rows; recomputed)
//   and in the epilogue, with Z read back, per row and column:
//     act = bf16(silu(G) U) (the forward's activation), dL/dw partial = sum Z act,
//     dG = w Z U silu'(G), dU = w Z silu(G)  -> BF16 [dG | dU];  w act -> BF16
//   Z, [dG | dU] and w act use a padded row layout: expert q's rows start at a
//   multiple of 128, and the rows past its count of the last two are zeros.
//
//   bwd_wgrad_tc_kernel   rows of an expert as the contracted K:
//     [dW_gate; dW_up]_q = [dG | dU]^T A     (M = 2I, N = H)
//     dW_down_q          = D^T (w act)        (M = H,  N = I)
//   both operands MN-major, read as stored (no transpose in memory); the zero
//   rows of the padded operand cancel what the other operand holds past the
//   expert's rows.  FP32 outputs.
//
// Every launch keeps four 48 KB operand stages in flight (a 128 x 256 x 64 MMA
// block each) and two 128 x 256 FP32 accumulators, so the epilogue of one tile
// overlaps the MMAs of the next.  CTA roles (192 threads), as in the forward:
// warp 0 lanes 0-2 issue TMA loads, warp 1 allocates TMEM and one thread
// issues the MMAs, warps 2-5 drain TMEM (one tile row per thread).  Every wait
// is bounded in time; on expiry the CTA records PMPE_STATUS_PIPELINE_TIMEOUT,
// stops, waits (bounded) for its copies and MMAs in flight, frees TMEM and exits.
#include <cuda.h>

#include <algorithm>
#include <cstring>

#include "pmpe_internal.cuh"
#include "tc_ptx.cuh"

namespace pmpe {
namespace {

constexpr int BM = 128;                        // MMA M (rows of a tile)
constexpr int BK = 64;                         // K per stage
constexpr int kABytes = BM * BK * 2;           // 16 KB
constexpr int kBBytes = 256 * BK * 2;          // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kMnBlockBytes = 64 * BK * 2;     // one 64-element MN block of an MN-major operand: 8 KB
constexpr int kThreads = 192;
constexpr int kLoaders = 3;
constexpr int kPad = 128;                      // padded row layout: each expert starts at a multiple of 128

// Four operand stages; outputs staged per epilogue warp in two 2 KB boxes of
// 32 rows x 64 bytes (32 BF16 or 16 FP32 columns, 64-byte swizzle).
constexpr int kStages = 4;
constexpr int kOutBoxBytes = 32 * 64;
constexpr int kOutBufs = 2;
constexpr int kDynSmem = kStages * kStageBytes + 4 * kOutBufs * kOutBoxBytes + 1024;
constexpr int kAccCols = 256;
constexpr int kTmemCols = 2 * kAccCols;

// Per private expert q: its rows, first row relative to the first private
// slot, first row of the padded layout; and the tiles of the experts before q.
struct GroupTable {
    int tiles[kMaxPool + 1];
    int rows[kMaxPool];
    int off[kMaxPool];
    int pad[kMaxPool];
};

// All threads: fill the table from the forward's dispatch offsets.
// tiles_per_row_block: tiles of an expert per 128-row block (0: every expert
// has `fixed_tiles` tiles whatever its rows).
__device__ void build_groups(GroupTable &gt, const uint32_t *offsets, int E_pub, int E_priv, int R,
                             int tiles_per_row_block, int fixed_tiles)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int p0 = (int)min(offsets[E_pub], (uint32_t)R);
    for (int q = tid; q < E_priv; q += blockDim.x) {
        const int b = min(max((int)offsets[E_pub + q], p0), R), e = min(max((int)offsets[E_pub + q + 1], b), R);
        const int rows = e - b;
        gt.rows[q] = rows;
        gt.off[q] = b - p0;
        gt.tiles[q + 1] = tiles_per_row_block ? ((rows + BM - 1) / BM) * tiles_per_row_block : fixed_tiles;
        gt.pad[q] = (rows + kPad - 1) / kPad * kPad;  // made exclusive prefix below
    }
    __syncthreads();
    if (warp < 2) {  // warp 0: inclusive scan of tiles; warp 1: exclusive scan of padded rows
        int carry = 0;
        for (int b = 0; b < E_priv; b += 32) {
            const int q = b + lane;
            const int v = q < E_priv ? (warp == 0 ? gt.tiles[q + 1] : gt.pad[q]) : 0;
            int x = v;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(~0u, x, off);
                if (lane >= off) x += y;
            }
            if (q < E_priv) {
                if (warp == 0) gt.tiles[q + 1] = carry + x;
                else gt.pad[q] = carry + x - v;
            }
            carry += __shfl_sync(~0u, x, 31);
        }
        if (warp == 0 && lane == 0) gt.tiles[0] = 0;
    }
    __syncthreads();
}

// This lane's 64-byte row of a staged output box: 16-byte chunk j of row r at
// chunk j ^ ((r >> 1) & 3), the TMA 64-byte swizzle (conflict-free for these
// 16-byte writes).
__device__ __forceinline__ void store_box_row(uint32_t sbuf, int lane, const uint32_t *w16)
{
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const uint32_t addr = sbuf + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4);
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(w16[4 * j]), "r"(w16[4 * j + 1]),
                     "r"(w16[4 * j + 2]), "r"(w16[4 * j + 3])
                     : "memory");
    }
}

// One epilogue warp's output path: stage a 32 x 64-byte box in one of two
// shared buffers and store it with TMA.
struct OutStager {
    uint32_t base;
    int ob;
    __device__ __forceinline__ void put(int lane, const uint32_t *w16, const CUtensorMap *map, int x, int y)
    {
        const uint32_t sbuf = base + (uint32_t)(ob * kOutBoxBytes);
        if (lane == 0) bulk_wait_read<kOutBufs - 1>();  // the store that used this buffer has read it
        __syncwarp();
        store_box_row(sbuf, lane, w16);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            tma_store_2d(map, sbuf, x, y);
            bulk_commit();
        }
        ob ^= 1;
    }
};

// Bounded wait for the drain at exit: every copy a loader issued has landed.
__device__ __forceinline__ void drain_stages(uint32_t bar0, int stages, uint32_t filled, uint32_t last_parity)
{
    for (int s = 0; s < stages; ++s)
        if ((filled >> s) & 1u) {
            const unsigned long long t0 = globaltimer_ns();
            while (!mbar_try_wait(bar0 + 8u * s, (last_parity >> s) & 1u))
                if (globaltimer_ns() - t0 > kWaitLimitNs) break;
        }
}

// ------------------------------------------------------------- rows

enum { kRowsZ = 0, kRowsGU = 1 };

struct RowsParams {
    int E_pub, E_priv, H, I, R;
    int bn;           // output columns per tile (Z: of I, 256 or 128; gate/up: 128 activation columns)
    const uint32_t *offsets;
    const float *w_of_slot;
    const bf16 *zpad;  // gate/up: Z in the padded row layout [RP][I]
    float *gw_part;    // gate/up: [R][I / 128] dL/dw partial of each private row per 128-column tile
    uint32_t *status;
    uint32_t idesc;
};

struct RowsMaps {
    CUtensorMap a;       // Z: dout rows [R + 64][H]; gate/up: A rows [R][H]; 64 x 128 box (K-major)
    CUtensorMap b0, b1;  // Z: W_down [E_priv H][I], 64 x 64 x bn/128 3-D box (MN-major); gate/up: gate, up, 64 x 128
    CUtensorMap out0;    // Z: Z [RP][I]; gate/up: [dG | dU] [RP][2I]  (32 x 32 BF16 boxes, 64-byte swizzle)
    CUtensorMap out1;    // gate/up: w act [RP][I]
};

struct RowsTile {
    int q, m0, n0, n_tile, rows;
};

__device__ __forceinline__ RowsTile decode_rows(const GroupTable &gt, int E_priv, int nt, int bn, int tile)
{
    int lo = 0, hi = E_priv - 1;  // last expert whose tile prefix is <= tile (skips empty experts)
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (gt.tiles[mid] <= tile) lo = mid; else hi = mid - 1;
    }
    RowsTile t;
    t.q = lo;
    const int mt = (gt.rows[lo] + BM - 1) / BM;
    const int local = tile - gt.tiles[lo];
    t.n_tile = local / mt;  // n-tile major inside an expert: its m tiles share the weight slice
    const int m_tile = local - t.n_tile * mt;
    t.m0 = m_tile * BM;
    t.n0 = t.n_tile * bn;
    t.rows = min(BM, gt.rows[lo] - t.m0);
    return t;
}

template <int kMode>
__global__ void __launch_bounds__(kThreads, 1) bwd_rows_tc_kernel(const RowsParams p, const __grid_constant__ RowsMaps maps)
{
    extern __shared__ uint8_t dsmem[];
    __shared__ GroupTable gt;
    __shared__ __align__(8) uint64_t bars[2 * kStages + 5];
    __shared__ uint32_t s_tmem;
    __shared__ volatile int s_abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t sbase = (smem_u32(dsmem) + 1023u) & ~1023u;
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (kStages + s); };
    auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * kStages + b); };
    auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * kStages + 2 + b); };
    const uint32_t done_bar = bar0 + 8u * (2 * kStages + 4);

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) { mbar_init(full_bar(s), kLoaders); mbar_init(empty_bar(s), 1); }
        for (int b = 0; b < 2; ++b) { mbar_init(tfull_bar(b), 1); mbar_init(tempty_bar(b), 4); }
        mbar_init(done_bar, 1);
        s_abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 1) tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    pdl_wait();
    const int nt = p.I / p.bn;
    build_groups(gt, p.offsets, p.E_pub, p.E_priv, p.R, nt, 0);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = s_tmem;
    const int total = gt.tiles[p.E_priv];
    const int nkb = p.H / BK;
    const int p0 = (int)min(p.offsets[p.E_pub], (uint32_t)p.R);

    if (warp == 0 && lane < kLoaders) {
        // ------------------------------------------------ TMA producers
        // lane 0: the tile's 128 rows x 64 K of A (16 KB).  Gate/up: lane 1 the
        // 128 gate rows, lane 2 the 128 up rows (16 KB each).  Z: lanes 1-2 half
        // of the bn / 64 MN blocks of W_down each, as one 3-D box (8 KB per block).
        int stage = 0;
        uint32_t phase = 0, filled = 0, last_parity = 0;
        const int half = p.bn / 128;  // Z: MN blocks per loader lane
        for (int tile = blockIdx.x; tile < total && !s_abort; tile += gridDim.x) {
            const RowsTile t = decode_rows(gt, p.E_priv, nt, p.bn, tile);
            const int arow = (kMode == kRowsGU ? p0 : 0) + gt.off[t.q] + t.m0;
            bool ok = true;
            for (int kb = 0; kb < nkb; ++kb) {
                if (!mbar_wait(empty_bar(stage), phase ^ 1u, &s_abort, p.status)) { ok = false; break; }
                const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
                const int kx = kb * BK;
                if (lane == 0) {
                    mbar_expect_tx(full_bar(stage), kABytes);
                    tma_load_2d(sA, &maps.a, full_bar(stage), kx, arow);
                } else if (kMode == kRowsGU) {
                    mbar_expect_tx(full_bar(stage), kABytes);
                    tma_load_2d(sB + (lane - 1) * kABytes, lane == 1 ? &maps.b0 : &maps.b1, full_bar(stage), kx,
                                t.q * p.I + t.n0);
                } else {
                    const int b0 = (lane - 1) * half;
                    mbar_expect_tx(full_bar(stage), (uint32_t)(half * kMnBlockBytes));
                    tma_load_3d(sB + b0 * kMnBlockBytes, &maps.b0, full_bar(stage), 0, t.q * p.H + kx, t.n0 / 64 + b0);
                }
                filled |= 1u << stage;
                last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
                if (++stage == kStages) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
        }
        drain_stages(bar0, kStages, filled, last_parity);
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------ MMA issuer
        // gate/up: one N = 256 MMA over the gate and up rows, G in accumulator
        // columns [0, 128) and U in [128, 256); Z: N = bn, W_down MN-major.
        int stage = 0, it = 0;
        uint32_t phase = 0;
        for (int tile = blockIdx.x; tile < total && !s_abort; tile += gridDim.x, ++it) {
            const int buf = it & 1;
            const uint32_t use = (uint32_t)(it >> 1) & 1u;
            if (!mbar_wait(tempty_bar(buf), use ^ 1u, &s_abort, p.status)) break;
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + (uint32_t)(buf * kAccCols);
            bool ok = true;
            for (int kb = 0; kb < nkb; ++kb) {
                if (!mbar_wait(full_bar(stage), phase, &s_abort, p.status)) { ok = false; break; }
                tc_fence_after();
                const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
                const uint64_t ad = sw128_desc(sA);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k) {
                    // K-major: +32 bytes of K per step inside the swizzle row;
                    // MN-major: 16 K rows = 2048 bytes per step
                    const uint64_t bd = kMode == kRowsGU ? sw128_desc(sB) + 2 * k
                                                         : mn_sw128_desc(sB + k * 2048, kMnBlockBytes);
                    tc_mma(d_tmem, ad + 2 * k, bd, p.idesc, (kb | k) != 0);
                }
                tc_commit(empty_bar(stage));
                if (++stage == kStages) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
            tc_commit(tfull_bar(buf));
        }
        tc_commit(done_bar);
        const unsigned long long t0 = globaltimer_ns();
        while (!mbar_try_wait(done_bar, 0))
            if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    } else if (warp >= 2) {
        // ------------------------------------------------ epilogue
        const int quarter = warp & 3;
        OutStager out{sbase + kStages * kStageBytes + (uint32_t)((warp - 2) * kOutBufs * kOutBoxBytes), 0};
        int it = 0;
        for (int tile = blockIdx.x; tile < total; tile += gridDim.x, ++it) {
            const RowsTile t = decode_rows(gt, p.E_priv, nt, p.bn, tile);
            const int buf = it & 1;
            const uint32_t use = (uint32_t)(it >> 1) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(tfull_bar(buf), use, &s_abort, p.status) ? 1 : 0;
            ok = __shfl_sync(~0u, ok, 0);
            if (!ok) break;
            __syncwarp();
            tc_fence_after();
            const int r = quarter * 32 + lane;
            const bool valid = r < t.rows;
            const int orow = gt.pad[t.q] + t.m0 + quarter * 32;  // this warp's 32 rows in the padded layout
            const uint32_t tb = tmem_base + (uint32_t)(buf * kAccCols) + ((uint32_t)(quarter * 32) << 16);
            if (kMode == kRowsZ) {
#pragma unroll 1
                for (int c = 0; c < p.bn / 32; ++c) {
                    float v[32];
                    tmem_ld32(tb + c * 32, v);
                    tmem_ld_wait();
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) pk[i] = pack_bf16x2(v[2 * i], v[2 * i + 1]);
                    out.put(lane, pk, &maps.out0, t.n0 + c * 32, orow);
                }
            } else {
                const int prow = gt.off[t.q] + t.m0 + r;  // private row (relative to the first private slot)
                const float w = valid ? p.w_of_slot[p0 + prow] : 0.f;
                const uint4 *zrow = reinterpret_cast<const uint4 *>(p.zpad + (size_t)(orow + lane) * p.I + t.n0);
                float gw = 0.f;
#pragma unroll 1
                for (int c = 0; c < 4; ++c) {
                    uint4 zq[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) zq[i] = valid ? zrow[c * 4 + i] : make_uint4(0u, 0u, 0u, 0u);
                    float g[32], u[32];
                    tmem_ld32(tb + c * 32, g);
                    tmem_ld32(tb + 128 + c * 32, u);
                    tmem_ld_wait();
                    const __nv_bfloat162 *zb = reinterpret_cast<const __nv_bfloat162 *>(zq);
                    uint32_t pg[16], pu[16], pa[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const float2 z2 = __bfloat1622float2(zb[i]);
                        float dg[2], du[2], wa[2];
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int j = 2 * i + h;
                            const float z = h ? z2.y : z2.x;
                            const float den = 1.f + __expf(-g[j]);
                            const float silu = __fdividef(g[j], den);  // the forward's silu(g) u, same arithmetic
                            const float a = __bfloat162float(__float2bfloat16_rn(silu * u[j]));
                            const float sg = __fdividef(1.f, den);
                            gw += z * a;
                            const float wz = w * z;
                            dg[h] = valid ? wz * u[j] * sg * (1.f + g[j] * (1.f - sg)) : 0.f;
                            du[h] = valid ? wz * silu : 0.f;
                            wa[h] = valid ? w * a : 0.f;
                        }
                        pg[i] = pack_bf16x2(dg[0], dg[1]);
                        pu[i] = pack_bf16x2(du[0], du[1]);
                        pa[i] = pack_bf16x2(wa[0], wa[1]);
                    }
                    out.put(lane, pg, &maps.out0, t.n0 + c * 32, orow);
                    out.put(lane, pu, &maps.out0, p.I + t.n0 + c * 32, orow);
                    out.put(lane, pa, &maps.out1, t.n0 + c * 32, orow);
                }
                if (valid) p.gw_part[(size_t)prow * nt + t.n_tile] = gw;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty_bar(buf));
        }
        if (lane == 0) bulk_wait_all();
    }

    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}

// ------------------------------------------------------------- wgrad

struct WgParams {
    int E_pub, E_priv, H, I, R;
    int bn_a, bn_b;  // output columns per tile: [dW_gate; dW_up] (N = H), dW_down (N = I)
    const uint32_t *offsets;
    uint32_t *status;
    uint32_t idesc_a, idesc_b;
};

struct WgMaps {
    // 3-D maps, boxes of 64 rows (K) x 64-element MN blocks (encode_3d_blocks)
    CUtensorMap dgu;        // [padded rows][2I], 2 blocks per box (MN-major A)
    CUtensorMap a_perm;     // [R][H], bn_a / 128 blocks per box (MN-major B)
    CUtensorMap dout_rows;  // [R + 64][H], 2 blocks per box (MN-major A)
    CUtensorMap wact;       // [padded rows][I], bn_b / 128 blocks per box (MN-major B)
    CUtensorMap d_gate, d_up, d_down;  // FP32 outputs, 16 x 32 boxes, 64-byte swizzle
};

struct WgTile {
    int prob, q, m0, n0, bn, nkb;
};

__device__ __forceinline__ WgTile decode_wg(const WgParams &p, const GroupTable &gt, int tile)
{
    WgTile t;
    const int na = p.H / p.bn_a, nta = (2 * p.I / BM) * na;
    const int nb = p.I / p.bn_b, ntb = (p.H / BM) * nb;
    int local;
    if (tile < p.E_priv * nta) {
        t.prob = 0;
        t.q = tile / nta;
        local = tile - t.q * nta;
        t.m0 = (local / na) * BM;
        t.n0 = (local % na) * p.bn_a;
        t.bn = p.bn_a;
    } else {
        tile -= p.E_priv * nta;
        t.prob = 1;
        t.q = tile / ntb;
        local = tile - t.q * ntb;
        t.m0 = (local / nb) * BM;
        t.n0 = (local % nb) * p.bn_b;
        t.bn = p.bn_b;
    }
    t.nkb = (gt.rows[t.q] + BK - 1) / BK;
    return t;
}

__global__ void __launch_bounds__(kThreads, 1) bwd_wgrad_tc_kernel(const WgParams p, const __grid_constant__ WgMaps maps)
{
    extern __shared__ uint8_t dsmem[];
    __shared__ GroupTable gt;
    __shared__ __align__(8) uint64_t bars[2 * kStages + 5];
    __shared__ uint32_t s_tmem;
    __shared__ volatile int s_abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t sbase = (smem_u32(dsmem) + 1023u) & ~1023u;
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (kStages + s); };
    auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * kStages + b); };
    auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * kStages + 2 + b); };
    const uint32_t done_bar = bar0 + 8u * (2 * kStages + 4);

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) { mbar_init(full_bar(s), kLoaders); mbar_init(empty_bar(s), 1); }
        for (int b = 0; b < 2; ++b) { mbar_init(tfull_bar(b), 1); mbar_init(tempty_bar(b), 4); }
        mbar_init(done_bar, 1);
        s_abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 1) tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    pdl_wait();
    build_groups(gt, p.offsets, p.E_pub, p.E_priv, p.R, 0, 0);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = s_tmem;
    const int total = p.E_priv * ((2 * p.I / BM) * (p.H / p.bn_a) + (p.H / BM) * (p.I / p.bn_b));
    const int p0 = (int)min(p.offsets[p.E_pub], (uint32_t)p.R);

    if (warp == 0 && lane < kLoaders) {
        // ------------------------------------------------ TMA producers
        // lane 0: the two 64-element MN blocks of A; lanes 1-2: half of B's
        // bn / 64 blocks each; one 3-D box per lane (64 MN elements x 64 rows of
        // K per block).
        int stage = 0;
        uint32_t phase = 0, filled = 0, last_parity = 0;
        for (int tile = blockIdx.x; tile < total && !s_abort; tile += gridDim.x) {
            const WgTile t = decode_wg(p, gt, tile);
            const int nbox = t.bn / 64, half = nbox / 2;
            const int rowA = t.prob == 0 ? gt.pad[t.q] : gt.off[t.q];
            const int rowB = t.prob == 0 ? p0 + gt.off[t.q] : gt.pad[t.q];
            const CUtensorMap *amap = t.prob == 0 ? &maps.dgu : &maps.dout_rows;
            const CUtensorMap *bmap = t.prob == 0 ? &maps.a_perm : &maps.wact;
            bool ok = true;
            for (int kb = 0; kb < t.nkb; ++kb) {
                if (!mbar_wait(empty_bar(stage), phase ^ 1u, &s_abort, p.status)) { ok = false; break; }
                const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
                const int ky = kb * BK;
                mbar_expect_tx(full_bar(stage), lane == 0 ? (uint32_t)kABytes : (uint32_t)(half * kMnBlockBytes));
                if (lane == 0) {
                    tma_load_3d(sA, amap, full_bar(stage), 0, rowA + ky, t.m0 / 64);
                } else {
                    const int b0 = (lane - 1) * half;
                    tma_load_3d(sB + b0 * kMnBlockBytes, bmap, full_bar(stage), 0, rowB + ky, t.n0 / 64 + b0);
                }
                filled |= 1u << stage;
                last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
                if (++stage == kStages) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
        }
        drain_stages(bar0, kStages, filled, last_parity);
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------ MMA issuer
        // two 128 x 256 FP32 accumulators: the epilogue of one tile overlaps the
        // MMAs of the next.  A tile of an expert without rows issues no MMA;
        // its epilogue writes zeros.
        int stage = 0, it = 0;
        uint32_t phase = 0;
        for (int tile = blockIdx.x; tile < total && !s_abort; tile += gridDim.x, ++it) {
            const WgTile t = decode_wg(p, gt, tile);
            const uint32_t idesc = t.prob == 0 ? p.idesc_a : p.idesc_b;
            const int buf = it & 1;
            const uint32_t use = (uint32_t)(it >> 1) & 1u;
            if (!mbar_wait(tempty_bar(buf), use ^ 1u, &s_abort, p.status)) break;
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + (uint32_t)(buf * 256);
            bool ok = true;
            for (int kb = 0; kb < t.nkb; ++kb) {
                if (!mbar_wait(full_bar(stage), phase, &s_abort, p.status)) { ok = false; break; }
                tc_fence_after();
                const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                    tc_mma(d_tmem, mn_sw128_desc(sA + k * 2048, kMnBlockBytes), mn_sw128_desc(sB + k * 2048, kMnBlockBytes),
                           idesc, (kb | k) != 0);
                tc_commit(empty_bar(stage));
                if (++stage == kStages) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
            tc_commit(tfull_bar(buf));
        }
        tc_commit(done_bar);
        const unsigned long long t0 = globaltimer_ns();
        while (!mbar_try_wait(done_bar, 0))
            if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    } else if (warp >= 2) {
        // ------------------------------------------------ epilogue
        const int quarter = warp & 3;
        OutStager out{sbase + kStages * kStageBytes + (uint32_t)((warp - 2) * kOutBufs * kOutBoxBytes), 0};
        int it = 0;
        for (int tile = blockIdx.x; tile < total; tile += gridDim.x, ++it) {
            const WgTile t = decode_wg(p, gt, tile);
            const int buf = it & 1;
            const uint32_t use = (uint32_t)(it >> 1) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(tfull_bar(buf), use, &s_abort, p.status) ? 1 : 0;
            ok = __shfl_sync(~0u, ok, 0);
            if (!ok) break;
            __syncwarp();
            tc_fence_after();
            const CUtensorMap *omap;
            int orow;
            if (t.prob == 0) {
                omap = t.m0 < p.I ? &maps.d_gate : &maps.d_up;
                orow = t.q * p.I + (t.m0 < p.I ? t.m0 : t.m0 - p.I);
            } else {
                omap = &maps.d_down;
                orow = t.q * p.H + t.m0;
            }
            orow += quarter * 32;
            const uint32_t tb = tmem_base + (uint32_t)(buf * 256) + ((uint32_t)(quarter * 32) << 16);
#pragma unroll 1
            for (int c = 0; c < t.bn / 32; ++c) {
                float v[32];
                if (t.nkb > 0) {
                    tmem_ld32(tb + c * 32, v);
                    tmem_ld_wait();
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = 0.f;
                }
                out.put(lane, reinterpret_cast<const uint32_t *>(v), omap, t.n0 + c * 32, orow);
                out.put(lane, reinterpret_cast<const uint32_t *>(v + 16), omap, t.n0 + c * 32 + 16, orow);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty_bar(buf));
        }
        if (lane == 0) bulk_wait_all();
    }

    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}

}  // namespace

// Rows of the padded layout (an upper bound over all routings).
size_t backward_padded_rows(const Shape &s) { return (size_t)s.T * s.k + (size_t)kPad * s.E_priv; }

cudaError_t launch_backward_rows(const Ctx &c, const bf16 *dout_rows, bf16 *zpad, bf16 *dgu, bf16 *wact,
                                 float *gw_part)
{
    const Shape &s = c.s;
    const uint64_t R = (uint64_t)s.T * s.k, RP = backward_padded_rows(s);
    static std::atomic<int> smem_limit[2][64];
    cudaError_t err;
    for (int mode = 0; mode < 2; ++mode) {
        RowsParams p;
        RowsMaps maps;
        memset(&p, 0, sizeof(p));
        memset(&maps, 0, sizeof(maps));
        p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.H = s.H; p.I = s.I; p.R = (int)R;
        p.offsets = c.offsets;
        p.w_of_slot = c.w_of_slot;
        p.zpad = zpad;
        p.gw_part = gw_part;
        p.status = c.audit.status;
        bool ok;
        if (mode == kRowsZ) {
            p.bn = s.I % 256 == 0 ? 256 : 128;
            p.idesc = make_idesc_major(BM, p.bn, false, true);
            ok = encode_2d(&maps.a, dout_rows, s.H, R + 64, BM);
            ok &= encode_3d_blocks(&maps.b0, c.down[1], s.I, (uint64_t)s.E_priv * s.H, 64, p.bn / 128);
            ok &= encode_2d_box(&maps.out0, zpad, s.I, RP, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
        } else {
            p.bn = 128;
            p.idesc = make_idesc(BM, 256);
            ok = encode_2d(&maps.a, c.a_perm, s.H, R, BM);
            ok &= encode_2d(&maps.b0, c.gate[1], s.H, (uint64_t)s.E_priv * s.I, 128);
            ok &= encode_2d(&maps.b1, c.up[1], s.H, (uint64_t)s.E_priv * s.I, 128);
            ok &= encode_2d_box(&maps.out0, dgu, 2 * (uint64_t)s.I, RP, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
            ok &= encode_2d_box(&maps.out1, wact, s.I, RP, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
        }
        if (!ok) return cudaErrorInvalidValue;
        auto kernel = mode == kRowsZ ? bwd_rows_tc_kernel<kRowsZ> : bwd_rows_tc_kernel<kRowsGU>;
        err = ensure_dynamic_smem(kernel, kDynSmem, smem_limit[mode]);
        if (err != cudaSuccess) return err;
        err = launch_pdl(kernel, dim3(c.num_sms), dim3(kThreads), kDynSmem, c.stream, p, maps);
        if (err != cudaSuccess) return err;
    }
    return cudaSuccess;
}

cudaError_t launch_backward_wgrad(const Ctx &c, const bf16 *dout_rows, const bf16 *dgu, const bf16 *wact,
                                  float *d_gate, float *d_up, float *d_down)
{
    const Shape &s = c.s;
    const uint64_t R = (uint64_t)s.T * s.k, RP = backward_padded_rows(s);
    WgParams p;
    WgMaps maps;
    memset(&p, 0, sizeof(p));
    memset(&maps, 0, sizeof(maps));
    p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.H = s.H; p.I = s.I; p.R = (int)R;
    p.bn_a = s.H % 256 == 0 ? 256 : 128;
    p.bn_b = s.I % 256 == 0 ? 256 : 128;
    p.offsets = c.offsets;
    p.status = c.audit.status;
    p.idesc_a = make_idesc_major(BM, p.bn_a, true, true);
    p.idesc_b = make_idesc_major(BM, p.bn_b, true, true);
    // A: both 64-element MN blocks in one box; B: half of its blocks per box
    bool ok = encode_3d_blocks(&maps.dgu, dgu, 2 * (uint64_t)s.I, RP, 64, 2);
    ok &= encode_3d_blocks(&maps.a_perm, c.a_perm, s.H, R, 64, p.bn_a / 128);
    ok &= encode_3d_blocks(&maps.dout_rows, dout_rows, s.H, R + 64, 64, 2);
    ok &= encode_3d_blocks(&maps.wact, wact, s.I, RP, 64, p.bn_b / 128);
    const CUtensorMapSwizzle osw = CU_TENSOR_MAP_SWIZZLE_64B;
    ok &= encode_2d_f32(&maps.d_gate, d_gate, s.H, (uint64_t)s.E_priv * s.I, 16, 32, osw);
    ok &= encode_2d_f32(&maps.d_up, d_up, s.H, (uint64_t)s.E_priv * s.I, 16, 32, osw);
    ok &= encode_2d_f32(&maps.d_down, d_down, s.I, (uint64_t)s.E_priv * s.H, 16, 32, osw);
    if (!ok) return cudaErrorInvalidValue;
    static std::atomic<int> smem_limit[64];
    cudaError_t err = ensure_dynamic_smem(bwd_wgrad_tc_kernel, kDynSmem, smem_limit);
    if (err != cudaSuccess) return err;
    return launch_pdl(bwd_wgrad_tc_kernel, dim3(c.num_sms), dim3(kThreads), kDynSmem, c.stream, p, maps);
}

}  // namespace pmpe
