// Backward of the private branch on the 5th-generation tensor cores (G2,
// Sec. 2.2; Sec. 3.2 trains the private experts and the private router only).
// Three persistent grouped GEMM launches over the private experts, each in the
// TMA -> shared memory -> tcgen05.mma -> TMEM -> epilogue pipeline of the
// forward's expert GEMMs:
//
//   bwd_rows_tc_kernel<kRowsMN>   rows of an expert as M, K = H:
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
// The same two row kernels, over all routed experts and the shared experts,
// and an MN-mode launch dA = [dG | dU] [W_gate; W_up] give the gradient of
// the layer's input (launch_rows_z, launch_rows_gu, launch_rows_da).
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

// Groups of a launch: the routed experts g0 .. g0 + G - 1 (rows = their
// dispatch slots), or G shared experts that each run every one of shared_T
// tokens.  Per group q: its rows, its first row relative to the first slot of
// expert g0 (0 for shared groups), its first row of the padded layout; and the
// tiles of the groups before q.
constexpr int kMaxGroups = 2 * kMaxPool;
struct GroupTable {
    int tiles[kMaxGroups + 1];
    int rows[kMaxGroups];
    int off[kMaxGroups];
    int pad[kMaxGroups];
};

// All threads: fill the table (routed groups from the forward's dispatch
// offsets).  tiles_per_row_block: tiles of a group per 128-row block (0:
// every group has `fixed_tiles` tiles whatever its rows).
__device__ void build_groups(GroupTable &gt, const uint32_t *offsets, int g0, int G, int R, int shared_T,
                             int tiles_per_row_block, int fixed_tiles)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int p0 = shared_T ? 0 : (int)min(offsets[g0], (uint32_t)R);
    for (int q = tid; q < G; q += blockDim.x) {
        int b = 0, e = shared_T;
        if (!shared_T) {
            b = min(max((int)offsets[g0 + q], p0), R);
            e = min(max((int)offsets[g0 + q + 1], b), R);
        }
        const int rows = e - b;
        gt.rows[q] = rows;
        gt.off[q] = b - p0;
        gt.tiles[q + 1] = tiles_per_row_block ? ((rows + BM - 1) / BM) * tiles_per_row_block : fixed_tiles;
        gt.pad[q] = (rows + kPad - 1) / kPad * kPad;  // made exclusive prefix below
    }
    __syncthreads();
    if (warp < 2) {  // warp 0: inclusive scan of tiles; warp 1: exclusive scan of padded rows
        int carry = 0;
        for (int b = 0; b < G; b += 32) {
            const int q = b + lane;
            const int v = q < G ? (warp == 0 ? gt.tiles[q + 1] : gt.pad[q]) : 0;
            int x = v;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(~0u, x, off);
                if (lane >= off) x += y;
            }
            if (q < G) {
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

enum { kRowsMN = 0, kRowsGU = 1 };
enum { kArowsTight = 0, kArowsSlot = 1, kArowsPad = 2 };

// One launch of the row GEMMs.  Mode kRowsMN: C = A B with A K-major rows
// (K = K) and B read MN-major from a weight tensor of the group's expert
// (K blocks below k_split from b0, the rest from b1; kb_rows rows of K per
// expert in those tensors), C -> BF16 [padded rows][N].  Mode kRowsGU: the
// gate/up recompute (K = H) and the SwiGLU backward epilogue.
struct RowsParams {
    int E_pub, H, I, R;
    int g0, G, shared_T;  // the groups (see build_groups)
    int K, N, bn;         // contracted size, output columns, output columns per tile
    int kb_rows, k_split; // MN mode: K rows of B per expert; first K block taken from b1
    int a_rows;           // A row of a tile row: kArowsTight (relative to expert g0's first slot),
                          // kArowsSlot (the dispatch slot; the token for shared groups), kArowsPad
    const uint32_t *offsets;
    const float *w_of_slot;  // gate/up: routing weights per slot (shared groups: weight 1)
    const bf16 *zpad;     // gate/up: Z in the padded row layout [RP][I]
    float *gw_part;       // gate/up (routed, may be null): [R][I / 128] dL/dw partial per 128-column tile
    int wact;             // gate/up: 1 to write w act to out1 for the private experts' rows
    int reverse;          // 1: walk the tiles from the last group to the first
    uint32_t *status;
    uint32_t idesc;
};

struct RowsMaps {
    CUtensorMap a;           // A rows, 64 x 128 box (K-major)
    CUtensorMap b0[2], b1[2];  // per weight pool (public, private; shared groups use [0]): MN mode:
                             // 64 x 64 x bn/128 3-D boxes (MN-major); gate/up: gate, up, 64 x 128 (K-major)
    CUtensorMap out0;        // MN: C [RP][N]; gate/up: [dG | dU] [RP][2I]  (32 x 32 BF16 boxes, 64-byte swizzle)
    CUtensorMap out1;        // gate/up: w act [RP][I]
};

struct RowsTile {
    int q, m0, n0, n_tile, rows;
};

__device__ __forceinline__ RowsTile decode_rows(const GroupTable &gt, int G, int nt, int bn, int tile, int reverse)
{
    if (reverse) tile = gt.tiles[G] - 1 - tile;
    int lo = 0, hi = G - 1;  // last group whose tile prefix is <= tile (skips empty groups)
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (gt.tiles[mid] <= tile) lo = mid; else hi = mid - 1;
    }
    RowsTile t;
    t.q = lo;
    const int mt = (gt.rows[lo] + BM - 1) / BM;
    const int local = tile - gt.tiles[lo];
    t.n_tile = local / mt;  // n-tile major inside a group: its m tiles share the weight slice
    const int m_tile = local - t.n_tile * mt;
    t.m0 = m_tile * BM;
    t.n0 = t.n_tile * bn;
    t.rows = min(BM, gt.rows[lo] - t.m0);
    return t;
}

// Weight pool (0 public or shared, 1 private) and index inside it of group q.
__device__ __forceinline__ int2 group_weights(const RowsParams &p, int q)
{
    if (p.shared_T) return make_int2(0, q);
    const int e = p.g0 + q;
    return e >= p.E_pub ? make_int2(1, e - p.E_pub) : make_int2(0, e);
}

// SwiGLU backward of one element, from the gate and up accumulators g, u,
// the row's Z value z and routing weight w: a = bf16(silu(g) u) with the
// forward's arithmetic, dG = w z u silu'(g), dU = w z silu(g), and w a.
__device__ __forceinline__ void swiglu_bwd(float g, float u, float z, float w, float &a, float &dg, float &du,
                                           float &wa)
{
    const float den = 1.f + __expf(-g);
    const float silu = __fdividef(g, den);
    a = __bfloat162float(__float2bfloat16_rn(silu * u));
    const float sg = __fdividef(1.f, den);
    const float wz = w * z;
    dg = wz * u * sg * (1.f + g * (1.f - sg));
    du = wz * silu;
    wa = w * a;
}

// dL/dw over 32 columns of a row: the products z a of four consecutive
// columns summed pairwise, then those eight sums pairwise.  The order is the
// butterfly of eight lanes holding four columns each, so a thread holding all
// 32 (the gate/up epilogue) and a warp holding the row's columns four per
// lane (bwd_swiglu_saved_kernel) get the same bits.
__device__ __forceinline__ float chunk_tree_sum(const float (&q)[32])
{
    float s[8];
#pragma unroll
    for (int l = 0; l < 8; ++l)
        s[l] = __fadd_rn(__fadd_rn(q[4 * l], q[4 * l + 1]), __fadd_rn(q[4 * l + 2], q[4 * l + 3]));
    const float t0 = __fadd_rn(s[0], s[1]), t1 = __fadd_rn(s[2], s[3]);
    const float t2 = __fadd_rn(s[4], s[5]), t3 = __fadd_rn(s[6], s[7]);
    return __fadd_rn(__fadd_rn(t0, t1), __fadd_rn(t2, t3));
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
    const int nt = p.N / p.bn;
    build_groups(gt, p.offsets, p.g0, p.G, p.R, p.shared_T, nt, 0);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = s_tmem;
    const int total = gt.tiles[p.G];
    const int nkb = p.K / BK;
    const int p0 = p.shared_T ? 0 : (int)min(p.offsets[p.g0], (uint32_t)p.R);

    if (warp == 0 && lane < kLoaders) {
        // ------------------------------------------------ TMA producers
        // lane 0: the tile's 128 rows x 64 K of A (16 KB).  Gate/up: lane 1 the
        // 128 gate rows, lane 2 the 128 up rows (16 KB each).  MN mode: lanes 1-2
        // half of the bn / 64 MN blocks of B each, as one 3-D box (8 KB per block).
        int stage = 0;
        uint32_t phase = 0, filled = 0, last_parity = 0;
        const int half = p.bn / 128;  // MN mode: MN blocks per loader lane
        for (int tile = blockIdx.x; tile < total && !s_abort; tile += gridDim.x) {
            const RowsTile t = decode_rows(gt, p.G, nt, p.bn, tile, p.reverse);
            const int2 wq = group_weights(p, t.q);
            const int arow = (p.a_rows == kArowsPad ? gt.pad[t.q] : (p.a_rows == kArowsSlot ? p0 : 0) + gt.off[t.q]) + t.m0;
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
                    tma_load_2d(sB + (lane - 1) * kABytes, lane == 1 ? &maps.b0[wq.x] : &maps.b1[wq.x], full_bar(stage),
                                kx, wq.y * p.I + t.n0);
                } else {
                    const int b0 = (lane - 1) * half;
                    const bool second = kb >= p.k_split;
                    const int krow = wq.y * p.kb_rows + (second ? kx - p.k_split * BK : kx);
                    mbar_expect_tx(full_bar(stage), (uint32_t)(half * kMnBlockBytes));
                    tma_load_3d(sB + b0 * kMnBlockBytes, second ? &maps.b1[wq.x] : &maps.b0[wq.x], full_bar(stage), 0,
                                krow, t.n0 / 64 + b0);
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
            const RowsTile t = decode_rows(gt, p.G, nt, p.bn, tile, p.reverse);
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
            if (kMode == kRowsMN) {
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
                const int prow = gt.off[t.q] + t.m0 + r;  // row relative to expert g0's first slot (shared: token)
                const float w = valid ? (p.shared_T ? 1.f : p.w_of_slot[p0 + prow]) : 0.f;
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
                    float zq_a[32];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const float2 z2 = __bfloat1622float2(zb[i]);
                        float dg[2], du[2], wa[2];
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int j = 2 * i + h;
                            float a;
                            const float z = h ? z2.y : z2.x;
                            swiglu_bwd(g[j], u[j], z, w, a, dg[h], du[h], wa[h]);
                            zq_a[j] = __fmul_rn(z, a);
                            if (!valid) dg[h] = du[h] = wa[h] = 0.f;
                        }
                        pg[i] = pack_bf16x2(dg[0], dg[1]);
                        pu[i] = pack_bf16x2(du[0], du[1]);
                        pa[i] = pack_bf16x2(wa[0], wa[1]);
                    }
                    gw = __fadd_rn(gw, chunk_tree_sum(zq_a));
                    out.put(lane, pg, &maps.out0, t.n0 + c * 32, orow);
                    out.put(lane, pu, &maps.out0, p.I + t.n0 + c * 32, orow);
                    if (p.wact && !p.shared_T && p.g0 + t.q >= p.E_pub)
                        out.put(lane, pa, &maps.out1, t.n0 + c * 32, orow);
                }
                if (valid && p.gw_part) p.gw_part[(size_t)(p0 + prow) * nt + t.n_tile] = gw;
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

// ------------------------------------------------------------- saved G | U

// The gate/up launch's outputs from the forward's saved accumulators G | U
// ([R][2I] FP32) instead of a recomputing GEMM: one warp per routed row and
// 128-column tile, four columns per lane (coalesced rows), with the
// epilogue's per-element arithmetic and its dL/dw summation order
// (chunk_tree_sum, then the four 32-column chunks in order), so [dG | dU],
// w act and the dL/dw partials are bitwise those of kRowsGU.  Tiles and the
// padded layout come from the same group table; padded tail rows are written
// as zeros.
__global__ void __launch_bounds__(256) bwd_swiglu_saved_kernel(const RowsParams p, const float *saved_gu, bf16 *dgu,
                                                               bf16 *wact)
{
    __shared__ GroupTable gt;
    pdl_wait();
    const int nt = p.I / 128;
    build_groups(gt, p.offsets, p.g0, p.G, p.R, p.shared_T, nt, 0);
    const int total = gt.tiles[p.G];
    const int p0 = p.shared_T ? 0 : (int)min(p.offsets[p.g0], (uint32_t)p.R);
    // saved rows: routed [R][2I] (G | U), then shared [T][2 G I] (all G, then all U)
    const int ld2 = p.shared_T ? 2 * p.G * p.I : 2 * p.I;
    const float *sbase = p.shared_T ? saved_gu + (size_t)p.R * 2 * p.I : saved_gu;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
        const RowsTile t = decode_rows(gt, p.G, nt, 128, tile, 0);
        const bool wa_out = p.wact && !p.shared_T && p.g0 + t.q >= p.E_pub;
        const int gcol = p.shared_T ? t.q * p.I : 0;  // the group's G columns in its saved row
        for (int r = warp; r < BM; r += nwarps) {
            const bool valid = r < t.rows;  // warp-uniform
            const int prow = gt.off[t.q] + t.m0 + r;
            const int orow = gt.pad[t.q] + t.m0 + r;
            const int col = t.n0 + 4 * lane;
            float g[4] = {0.f, 0.f, 0.f, 0.f}, u[4] = {0.f, 0.f, 0.f, 0.f}, z[4] = {0.f, 0.f, 0.f, 0.f};
            float w = 0.f;
            if (valid) {
                const float *grow = sbase + (size_t)(p0 + prow) * ld2 + gcol;
                const float4 gv = *reinterpret_cast<const float4 *>(grow + col);
                const float4 uv = *reinterpret_cast<const float4 *>(grow + ld2 / 2 + col);
                const uint2 zv = *reinterpret_cast<const uint2 *>(p.zpad + (size_t)orow * p.I + col);
                g[0] = gv.x; g[1] = gv.y; g[2] = gv.z; g[3] = gv.w;
                u[0] = uv.x; u[1] = uv.y; u[2] = uv.z; u[3] = uv.w;
                const float2 z01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&zv.x));
                const float2 z23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&zv.y));
                z[0] = z01.x; z[1] = z01.y; z[2] = z23.x; z[3] = z23.y;
                w = p.shared_T ? 1.f : p.w_of_slot[p0 + prow];
            }
            float dg[4], du[4], wa[4], q[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                float a;
                swiglu_bwd(g[h], u[h], z[h], w, a, dg[h], du[h], wa[h]);
                q[h] = __fmul_rn(z[h], a);
                if (!valid) dg[h] = du[h] = wa[h] = 0.f;
            }
            bf16 *dst = dgu + (size_t)orow * 2 * p.I + col;
            *reinterpret_cast<uint2 *>(dst) = make_uint2(pack_bf16x2(dg[0], dg[1]), pack_bf16x2(dg[2], dg[3]));
            *reinterpret_cast<uint2 *>(dst + p.I) = make_uint2(pack_bf16x2(du[0], du[1]), pack_bf16x2(du[2], du[3]));
            if (wa_out)
                *reinterpret_cast<uint2 *>(wact + (size_t)orow * p.I + col) =
                    make_uint2(pack_bf16x2(wa[0], wa[1]), pack_bf16x2(wa[2], wa[3]));
            // the 32-column chunk sums in chunk_tree_sum's order: four columns in
            // the lane, then the butterfly over the chunk's eight lanes
            float sum = __fadd_rn(__fadd_rn(q[0], q[1]), __fadd_rn(q[2], q[3]));
            sum = __fadd_rn(sum, __shfl_xor_sync(~0u, sum, 1));
            sum = __fadd_rn(sum, __shfl_xor_sync(~0u, sum, 2));
            sum = __fadd_rn(sum, __shfl_xor_sync(~0u, sum, 4));
            const float c0 = __shfl_sync(~0u, sum, 0), c1 = __shfl_sync(~0u, sum, 8);
            const float c2 = __shfl_sync(~0u, sum, 16), c3 = __shfl_sync(~0u, sum, 24);
            if (lane == 0 && valid && p.gw_part) {
                float gw = 0.f;
                gw = __fadd_rn(gw, c0);
                gw = __fadd_rn(gw, c1);
                gw = __fadd_rn(gw, c2);
                gw = __fadd_rn(gw, c3);
                p.gw_part[(size_t)(p0 + prow) * nt + t.n_tile] = gw;
            }
        }
    }
}

// ------------------------------------------------------------- wgrad

struct WgParams {
    int E_pub, E_priv, H, I, R;
    // the group table's groups (the private experts alone, g0 = E_pub, or all
    // routed experts, g0 = 0, whose padded layout the operands then use) and
    // the table index of private expert 0
    int g0, G, q_off;
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
    t.nkb = (gt.rows[t.q + p.q_off] + BK - 1) / BK;
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
    build_groups(gt, p.offsets, p.g0, p.G, p.R, 0, 0, 0);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = s_tmem;
    const int total = p.E_priv * ((2 * p.I / BM) * (p.H / p.bn_a) + (p.H / BM) * (p.I / p.bn_b));
    const int p0 = (int)min(p.offsets[p.g0], (uint32_t)p.R);

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
            const int gq = t.q + p.q_off;  // the expert's entry in the group table
            const int rowA = t.prob == 0 ? gt.pad[gq] : gt.off[gq];
            const int rowB = t.prob == 0 ? p0 + gt.off[gq] : gt.pad[gq];
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

namespace {

// Fields shared by every row launch over the groups `g`.
RowsParams rows_params(const Ctx &c, const RowsGroups &g)
{
    const Shape &s = c.s;
    RowsParams p;
    memset(&p, 0, sizeof(p));
    p.E_pub = s.E_pub; p.H = s.H; p.I = s.I; p.R = s.T * s.k;
    p.g0 = g.g0; p.G = g.G; p.shared_T = g.shared_T;
    p.offsets = c.offsets;
    p.w_of_slot = c.w_of_slot;
    p.status = c.audit.status;
    return p;
}

// The weight tensor of pool q (0 public, 1 private) for routed groups, or the
// shared one, with its rows: experts x rows_per_expert.
const bf16 *pool_tensor(const Ctx &c, const RowsGroups &g, const bf16 *const *w, int q, int rows_per_expert,
                        uint64_t *rows)
{
    const Shape &s = c.s;
    const int n = g.shared_T ? s.E_sh : (q ? s.E_priv : s.E_pub);
    *rows = (uint64_t)n * rows_per_expert;
    return g.shared_T ? w[2] : w[q];
}

cudaError_t run_rows(int mode, const Ctx &c, const RowsParams &p, const RowsMaps &maps)
{
    static std::atomic<int> smem_limit[2][64];
    auto kernel = mode == kRowsMN ? bwd_rows_tc_kernel<kRowsMN> : bwd_rows_tc_kernel<kRowsGU>;
    cudaError_t err = ensure_dynamic_smem(kernel, kDynSmem, smem_limit[mode]);
    if (err != cudaSuccess) return err;
    return launch_pdl(kernel, dim3(c.num_sms), dim3(kThreads), kDynSmem, c.stream, p, maps);
}

}  // namespace

cudaError_t launch_rows_z(const Ctx &c, const RowsGroups &g, const bf16 *d, uint64_t d_rows, int tight, bf16 *zpad)
{
    const Shape &s = c.s;
    RowsParams p = rows_params(c, g);
    RowsMaps maps;
    memset(&maps, 0, sizeof(maps));
    p.K = s.H; p.N = s.I; p.bn = s.I % 256 == 0 ? 256 : 128;
    p.kb_rows = s.H; p.k_split = s.H / BK;
    p.a_rows = tight ? kArowsTight : kArowsSlot;
    p.idesc = make_idesc_major(BM, p.bn, false, true);
    bool ok = encode_2d(&maps.a, d, s.H, d_rows, BM);
    for (int q = 0; q < (g.shared_T ? 1 : 2); ++q) {
        uint64_t rows;
        const bf16 *w = pool_tensor(c, g, c.down, q, s.H, &rows);
        ok &= encode_3d_blocks(&maps.b0[q], w, s.I, rows, 64, p.bn / 128);
    }
    ok &= encode_2d_box(&maps.out0, zpad, s.I, g.padded_rows, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
    if (!ok) return cudaErrorInvalidValue;
    return run_rows(kRowsMN, c, p, maps);
}

cudaError_t launch_rows_gu(const Ctx &c, const RowsGroups &g, const bf16 *a, uint64_t a_rows, const bf16 *zpad,
                           bf16 *dgu, bf16 *wact, float *gw_part)
{
    const Shape &s = c.s;
    RowsParams p = rows_params(c, g);
    if (c.saved_gu) {  // the forward saved the G | U accumulators of these rows
        p.K = s.H; p.N = s.I; p.bn = 128;
        p.zpad = zpad;
        p.gw_part = gw_part;
        p.wact = wact ? 1 : 0;
        return launch_pdl(bwd_swiglu_saved_kernel, dim3(c.num_sms * 8), dim3(256), 0, c.stream, p,
                          (const float *)c.saved_gu, dgu, wact);
    }
    RowsMaps maps;
    memset(&maps, 0, sizeof(maps));
    p.K = s.H; p.N = s.I; p.bn = 128;
    p.a_rows = kArowsSlot;
    // last group first: the Z launch before ended on the last groups, whose
    // rows are still in L2, and the launch after starts on the first groups,
    // whose operands this one read last
    p.reverse = 1;
    p.zpad = zpad;
    p.gw_part = gw_part;
    p.wact = wact ? 1 : 0;
    p.idesc = make_idesc(BM, 256);
    bool ok = encode_2d(&maps.a, a, s.H, a_rows, BM);
    for (int q = 0; q < (g.shared_T ? 1 : 2); ++q) {
        uint64_t rows;
        const bf16 *wg = pool_tensor(c, g, c.gate, q, s.I, &rows);
        const bf16 *wu = pool_tensor(c, g, c.up, q, s.I, &rows);
        ok &= encode_2d(&maps.b0[q], wg, s.H, rows, 128);
        ok &= encode_2d(&maps.b1[q], wu, s.H, rows, 128);
    }
    ok &= encode_2d_box(&maps.out0, dgu, 2 * (uint64_t)s.I, g.padded_rows, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
    if (wact) ok &= encode_2d_box(&maps.out1, wact, s.I, g.padded_rows, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
    if (!ok) return cudaErrorInvalidValue;
    return run_rows(kRowsGU, c, p, maps);
}

cudaError_t launch_rows_da(const Ctx &c, const RowsGroups &g, const bf16 *dgu, bf16 *da)
{
    const Shape &s = c.s;
    RowsParams p = rows_params(c, g);
    RowsMaps maps;
    memset(&maps, 0, sizeof(maps));
    p.K = 2 * s.I; p.N = s.H; p.bn = s.H % 256 == 0 ? 256 : 128;
    p.kb_rows = s.I; p.k_split = s.I / BK;  // K blocks of dG take W_gate, those of dU take W_up
    p.a_rows = kArowsPad;
    p.idesc = make_idesc_major(BM, p.bn, false, true);
    bool ok = encode_2d(&maps.a, dgu, 2 * (uint64_t)s.I, g.padded_rows, BM);
    for (int q = 0; q < (g.shared_T ? 1 : 2); ++q) {
        uint64_t rows;
        const bf16 *wg = pool_tensor(c, g, c.gate, q, s.I, &rows);
        const bf16 *wu = pool_tensor(c, g, c.up, q, s.I, &rows);
        ok &= encode_3d_blocks(&maps.b0[q], wg, s.H, rows, 64, p.bn / 128);
        ok &= encode_3d_blocks(&maps.b1[q], wu, s.H, rows, 64, p.bn / 128);
    }
    ok &= encode_2d_box(&maps.out0, da, s.H, g.padded_rows, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
    if (!ok) return cudaErrorInvalidValue;
    return run_rows(kRowsMN, c, p, maps);
}

cudaError_t launch_backward_rows(const Ctx &c, const bf16 *dout_rows, bf16 *zpad, bf16 *dgu, bf16 *wact,
                                 float *gw_part)
{
    const Shape &s = c.s;
    const RowsGroups g{s.E_pub, s.E_priv, 0, backward_padded_rows(s)};
    cudaError_t err = launch_rows_z(c, g, dout_rows, (uint64_t)s.T * s.k + 64, 1, zpad);
    if (err != cudaSuccess) return err;
    return launch_rows_gu(c, g, c.a_perm, (uint64_t)s.T * s.k, zpad, dgu, wact, gw_part);
}

cudaError_t launch_backward_wgrad(const Ctx &c, const bf16 *dout_rows, const bf16 *dgu, const bf16 *wact,
                                  float *d_gate, float *d_up, float *d_down, const RowsGroups *all)
{
    const Shape &s = c.s;
    const uint64_t R = (uint64_t)s.T * s.k, RP = all ? all->padded_rows : backward_padded_rows(s);
    WgParams p;
    WgMaps maps;
    memset(&p, 0, sizeof(p));
    memset(&maps, 0, sizeof(maps));
    p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.H = s.H; p.I = s.I; p.R = (int)R;
    p.g0 = all ? 0 : s.E_pub;
    p.G = all ? s.E() : s.E_priv;
    p.q_off = all ? s.E_pub : 0;
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
