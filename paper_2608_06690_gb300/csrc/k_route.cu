// Stage 1 of the layer: fail-closed policy resolve, masked router, top-k and
// the route log (Sec. 3.1 Eq. 4; App. B.1 steps 2, 4, 5).
//
// router_tc_kernel: the tokens of each pool form 128-token tiles (DENY tiles
// first, then ALLOW tiles, each in ascending token order), and each tile is
// split by 32-expert chunks of its pool's router: one CTA per (tile, chunk).
// Every CTA resolves the policy bytes itself (only the trusted byte 0x01 is
// ALLOW) and ranks the tokens inside their pool, which gives it its tile.  A
// TMA ring streams the tile's token rows and the chunk's 32 router rows as
// 128-byte-swizzled tiles into shared memory: straight from `hidden` when
// the tile's tokens are consecutive, otherwise from a contiguous workspace
// block the CTA first fills by token index.  tcgen05.mma computes the
// 128 x 32 logits of the chunk in tensor memory.  A DENY row is only ever
// multiplied by public router rows and an ALLOW row only by private ones: an
// ineligible expert never becomes a candidate.
//
// One epilogue thread per token sorts its 32 logits (descending score, ties
// to the lower expert id; a bitonic network in registers) and publishes the
// first k with the chunk's softmax partial to the workspace.  The CTA that
// completes a tile last (an integer atomic per tile, after a memory fence)
// merges the chunk lists in chunk order, writes the softmax weights and the
// route log, and ranks each row among the tile's rows of its expert by token
// order (a 128-bit token mask per expert: the rank is a popcount), so that
// the dispatch order is deterministic; it records the tile's per-expert
// counts in its column of tile_counts.
#include <cuda.h>

#include "pmpe_internal.cuh"
#include "tc_ptx.cuh"

namespace pmpe {
namespace {

constexpr int kRThreads = 192;  // warp 0 TMA, warp 1 TMEM + MMA, warps 2..5 epilogue (one thread per token)
constexpr int kRMaxStages = 10;
constexpr int kTileRows = 128;
constexpr int kChunk = 32;                  // experts per CTA (MMA N)
constexpr int kMaxChunks = 2 * kMaxPool / kChunk;  // chunks of one tile: 8 per pool, 16 unmasked
constexpr int kABytes = kTileRows * 128;    // 128 rows x 64 BF16
constexpr int kBBytes = kChunk * 128;       // 32 router rows x 64 BF16
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kEpi = 128;                   // epilogue threads

struct RouterParams {
    int T, H, E_pub, E_priv, k, renorm;
    int nch[3];          // 32-expert chunks of the public pool, the private pool, and both (unmasked)
    int nch_max;         // CTAs per tile slot
    int unmasked;        // the soft-router control: one pool of all experts, no hard mask
    uint32_t idesc;      // M = 128, N = 32
    int stages;
    const uint8_t *policy;
    const bf16 *hidden;
    bf16 *rows_ws;       // [slots * nch_max * 128, H] copied tile rows, one block per CTA
    float2 *lists;       // [slots * nch_max][128][k] (score, id) sorted per chunk
    float4 *meta;        // [slots * nch_max][128] (chunk max, sum exp(x - max), entries, -)
    uint32_t *tile_done; // [slots] chunk CTAs finished (zeroed before the launch)
    uint8_t *tau;
    int32_t *idx;
    float *w;
    uint32_t *counts;    // per-expert row counters (zeroed before the launch)
    uint32_t *tile_counts;  // [E][slots4] rows of each expert per tile (a column per tile slot)
    int slots4;
    int32_t *ticket;     // [T, k] 128 * tile slot + position among the tile's rows of its expert
    uint32_t *route_count, *route_priv_rows, *status;
};

struct RouterMaps {
    CUtensorMap hidden;     // [T, H], box 64 x 128 (tiles of consecutive tokens)
    CUtensorMap rows;       // rows_ws, box 64 x 128 (copied tiles)
    CUtensorMap router[2];  // [E_pool, H], box 64 x 32
};

// Exclusive scan over the block of one int per thread (kRThreads threads).
__device__ __forceinline__ int block_scan(int v, int *warp_tot, int &total)
{
    constexpr int kW = kRThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(~0u, x, off);
        if (lane >= off) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    int before = 0;
    total = 0;
#pragma unroll
    for (int i = 0; i < kW; ++i) {
        const int t = warp_tot[i];
        before += i < warp ? t : 0;
        total += t;
    }
    __syncthreads();
    return before + x - v;
}

__device__ __forceinline__ bool is_allow(const uint8_t *policy, int t)
{
    return policy != nullptr && policy[t] == 0x01;
}

// Bytes of policy[t0, t1) equal to the trusted ALLOW value 0x01.  Whole
// 16-byte groups inside the range are read with vector loads when the
// pointer allows it (the caller's runs start at multiples of 16); any other
// byte is read on its own.  Nothing outside [t0, t1) is read.
__device__ __forceinline__ int count_allow(const uint8_t *policy, int t0, int t1)
{
    if (policy == nullptr || t0 >= t1) return 0;
    int n = 0, t = t0;
    if ((((uintptr_t)(policy + t0)) & 15u) == 0) {
        const uint4 *v = reinterpret_cast<const uint4 *>(policy + t0);
        const int groups = (t1 - t0) >> 4;
        constexpr int kBatch = 4;  // independent 16-byte loads in flight
        for (int g0 = 0; g0 < groups; g0 += kBatch) {
            uint4 x[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u)
                if (g0 + u < groups) x[u] = __ldg(v + g0 + u);
#pragma unroll
            for (int u = 0; u < kBatch; ++u)
                if (g0 + u < groups) {
                    // __vcmpeq4 sets each equal byte to 0xff: eight set bits per ALLOW byte
                    n += (__popc(__vcmpeq4(x[u].x, 0x01010101u)) + __popc(__vcmpeq4(x[u].y, 0x01010101u)) +
                          __popc(__vcmpeq4(x[u].z, 0x01010101u)) + __popc(__vcmpeq4(x[u].w, 0x01010101u))) >> 3;
                }
        }
        t = t0 + (groups << 4);
    }
    for (; t < t1; ++t) n += policy[t] == 0x01;
    return n;
}

// (x, e) ranks above (bx, be): larger logit, or equal logit and lower id.
// Evaluated without short-circuit branches (it sits inside sorting networks).
__device__ __forceinline__ bool ranks_above(float x, int e, float bx, int be)
{
    return (x > bx) | ((x == bx) & (e < be));
}

// One compare-exchange of the bitonic network on positions I < J: after it,
// position I holds the pair that ranks higher when `best_first`, else lower.
template <int I, int J, bool kBestFirst>
__device__ __forceinline__ void cex(float (&v)[32], int (&e)[32])
{
    const bool sw = kBestFirst ? ranks_above(v[J], e[J], v[I], e[I]) : ranks_above(v[I], e[I], v[J], e[J]);
    const float tv = v[I];
    const int te = e[I];
    v[I] = sw ? v[J] : v[I];
    e[I] = sw ? e[J] : e[I];
    v[J] = sw ? tv : v[J];
    e[J] = sw ? te : e[J];
}

// All compare-exchanges of one (SIZE, STRIDE) step for positions I .. 31.
template <int SIZE, int STRIDE, int I>
__device__ __forceinline__ void bitonic_step(float (&v)[32], int (&e)[32])
{
    if constexpr (I < 32) {
        if constexpr ((I ^ STRIDE) > I) cex<I, (I ^ STRIDE), (I & SIZE) == 0>(v, e);
        bitonic_step<SIZE, STRIDE, I + 1>(v, e);
    }
}

template <int SIZE, int STRIDE>
__device__ __forceinline__ void bitonic_merge(float (&v)[32], int (&e)[32])
{
    if constexpr (STRIDE > 0) {
        bitonic_step<SIZE, STRIDE, 0>(v, e);
        bitonic_merge<SIZE, STRIDE / 2>(v, e);
    }
}

template <int SIZE>
__device__ __forceinline__ void bitonic_sort(float (&v)[32], int (&e)[32])
{
    if constexpr (SIZE <= 32) {
        bitonic_merge<SIZE, SIZE / 2>(v, e);
        bitonic_sort<SIZE * 2>(v, e);
    }
}

// Sort 32 (score, id) pairs held in registers into rank order (best first)
// with a bitonic network whose every index is a compile-time constant.
__device__ __forceinline__ void sort32(float (&v)[32], int (&e)[32]) { bitonic_sort<2>(v, e); }

// The best pair among positions not yet taken (bit i of `taken`), by two
// interleaved chains of a branch-free scan; returns its position (-1: none).
__device__ __forceinline__ int best_untaken(const float (&v)[32], const int (&e)[32], uint32_t taken, float &bv,
                                            int &be)
{
    float cv[2] = {-INFINITY, -INFINITY};
    int ce[2] = {0x7fffffff, 0x7fffffff}, ci[2] = {-1, -1};
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const int c = i & 1;
        const bool better = !((taken >> i) & 1u) & ((ci[c] < 0) | ranks_above(v[i], e[i], cv[c], ce[c]));
        cv[c] = better ? v[i] : cv[c];
        ce[c] = better ? e[i] : ce[c];
        ci[c] = better ? i : ci[c];
    }
    const bool second = ci[1] >= 0 && (ci[0] < 0 || ranks_above(cv[1], ce[1], cv[0], ce[0]));
    bv = second ? cv[1] : cv[0];
    be = second ? ce[1] : ce[0];
    return second ? ci[1] : ci[0];
}

__global__ void __launch_bounds__(kRThreads, 1) router_tc_kernel(const RouterParams p,
                                                                  const __grid_constant__ RouterMaps maps)
{
    extern __shared__ uint8_t dsmem[];
    __shared__ int s_tok[kTileRows];
    __shared__ int warp_tot[kRThreads / 32];
    __shared__ __align__(8) uint64_t bars[2 * kRMaxStages + 2];
    __shared__ uint32_t s_tmem;
    __shared__ volatile int s_abort;
    __shared__ int s_last;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int slot = blockIdx.x / p.nch_max, chunk = blockIdx.x - slot * p.nch_max;
    pdl_trigger();
    pdl_wait();  // the caller's hidden states / policy may come from the previous kernel

    // ---- resolve and rank in one pass: each thread takes a contiguous run of
    // tokens (a multiple of 16 long, so that runs start 16-byte aligned); the
    // scan of its ALLOW count gives the pool sizes and its ranks
    const int per = ((p.T + kRThreads - 1) / kRThreads + 15) & ~15;
    const int t0 = min(p.T, tid * per), t1 = min(p.T, t0 + per);
    // the unmasked control tiles all tokens as one pool, in token order
    const int a = p.unmasked ? 0 : count_allow(p.policy, t0, t1);
    int na;
    const int a_before = block_scan(a, warp_tot, na);
    const int nd = p.T - na;
    const int tiles_d = (nd + kTileRows - 1) / kTileRows;
    int pool, m0;
    if (slot < tiles_d) {
        pool = 0;
        m0 = slot * kTileRows;
    } else {
        pool = 1;
        m0 = (slot - tiles_d) * kTileRows;
        if (m0 >= na) return;  // uniform: no tile for this slot
    }
    const int rows = min(kTileRows, (pool ? na : nd) - m0);
    // only a thread whose ranks in the tile's pool overlap the tile walks its run
    if ((pool ? a_before : t0 - a_before) < m0 + rows &&
        (pool ? a_before + a : t1 - a_before - a) > m0) {
        int ra = a_before, rd = t0 - a_before;  // ranks inside the ALLOW / DENY pools
        for (int t = t0; t < t1; ++t) {
            const bool al_byte = is_allow(p.policy, t);
            const bool al = al_byte && !p.unmasked;
            const int rank = al ? ra++ : rd++;
            if ((al ? 1 : 0) == pool && rank >= m0 && rank < m0 + rows) {
                s_tok[rank - m0] = t;
                if (chunk == 0) p.tau[t] = al_byte ? 1 : 0;  // every token is written by exactly one CTA
            }
        }
    }
    if (p.unmasked) pool = 2;
    if (chunk >= p.nch[pool]) return;  // uniform: the pool has fewer chunks
    __syncthreads();
    for (int r = rows + tid; r < kTileRows; r += kRThreads) s_tok[r] = s_tok[0];  // padding rows name a real token
    // The TMA ring reads the tile's rows as one 128-row tile.  When the tile's
    // tokens are consecutive (a request with one policy) that tile is read
    // from `hidden` directly; otherwise the CTA first copies its token rows
    // into its own contiguous block (padding rows are not copied: their logits
    // are never read) and makes the generic-proxy writes visible to the async
    // proxy of the TMA reads.
    const int contiguous = __syncthreads_and(tid >= rows || s_tok[tid < kTileRows ? tid : 0] == s_tok[0] + tid);
    if (!contiguous) {
        constexpr int kBatch = 16;  // independent 16-byte loads in flight per thread
        const int nv = p.H / 8;
        const uint4 *src = reinterpret_cast<const uint4 *>(p.hidden);
        uint4 *dst = reinterpret_cast<uint4 *>(p.rows_ws) + (size_t)blockIdx.x * kTileRows * nv;
        const int total = rows * nv;
        for (int i0 = tid; i0 < total; i0 += kBatch * kRThreads) {
            uint4 v[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int q = i0 + u * kRThreads;
                if (q < total) {
                    const int r = q / nv;
                    v[u] = __ldg(src + (size_t)s_tok[r] * nv + (q - r * nv));
                }
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u)
                if (i0 + u * kRThreads < total) dst[i0 + u * kRThreads] = v[u];
        }
        asm volatile("fence.proxy.async.global;\n" ::: "memory");
    }
    const uint32_t sbase = (smem_u32(dsmem) + 1023u) & ~1023u;
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (kRMaxStages + s); };
    const uint32_t tfull_bar = bar0 + 8u * (2 * kRMaxStages);
    const uint32_t done_bar = bar0 + 8u * (2 * kRMaxStages + 1);
    if (tid == 0) {
        for (int s = 0; s < p.stages; ++s) { mbar_init(full_bar(s), 2); mbar_init(empty_bar(s), 1); }
        mbar_init(tfull_bar, 1);
        mbar_init(done_bar, 1);
        s_abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 1) tmem_alloc(smem_u32(&s_tmem), kChunk);
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    const int nkb = p.H / 64;
    // This CTA's chunk: router tensor q (0 public, 1 private) and chunk lc in
    // it.  Pool ids run 0 .. P-1 (the concatenated ids in the unmasked pool);
    // base is the global id of pool id 0; c0 the pool id of column 0.
    const int q = pool == 2 ? (chunk < p.nch[0] ? 0 : 1) : pool;
    const int lc = (pool == 2 && q == 1) ? chunk - p.nch[0] : chunk;
    const int P = pool == 2 ? p.E_pub + p.E_priv : (pool ? p.E_priv : p.E_pub);
    const int base = pool == 1 ? p.E_pub : 0;
    const int c0 = (pool == 2 && q == 1 ? p.E_pub : 0) + lc * kChunk;
    const int nvalid = min(kChunk, (q ? p.E_priv : p.E_pub) - lc * kChunk);

    if (warp == 0 && lane < 2) {
        // ---- TMA producers: lane 0 the 128 tile rows, lane 1 the chunk's 32
        // router rows (one box each; router rows past the pool read as zeros)
        int stage = 0;
        uint32_t phase = 0, filled = 0, last_parity = 0;
        const uint32_t my_tx = lane == 0 ? (uint32_t)kABytes : (uint32_t)kBBytes;
        for (int kb = 0; kb < nkb; ++kb) {
            if (!mbar_wait(empty_bar(stage), phase ^ 1u, &s_abort, p.status)) break;
            const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
            mbar_expect_tx(full_bar(stage), my_tx);
            if (lane == 1)
                tma_load_2d(sB, &maps.router[q], full_bar(stage), kb * 64, lc * kChunk);
            else if (contiguous)
                tma_load_2d(sA, &maps.hidden, full_bar(stage), kb * 64, s_tok[0]);
            else
                tma_load_2d(sA, &maps.rows, full_bar(stage), kb * 64, blockIdx.x * kTileRows);
            filled |= 1u << stage;
            last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
            if (++stage == p.stages) { stage = 0; phase ^= 1u; }
        }
        // every copy this thread issued has landed before the CTA exits
        for (int s = 0; s < p.stages; ++s)
            if ((filled >> s) & 1u) {
                const unsigned long long w0 = globaltimer_ns();
                while (!mbar_try_wait(full_bar(s), (last_parity >> s) & 1u))
                    if (globaltimer_ns() - w0 > kWaitLimitNs) break;
            }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer: logits[128, 32] += rows[128, 64] x router[32, 64]^T per stage
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb) {
            if (!mbar_wait(full_bar(stage), phase, &s_abort, p.status)) { ok = false; break; }
            tc_fence_after();
            const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
            const uint64_t ad = sw128_desc(sA), bd = sw128_desc(sB);
#pragma unroll
            for (int k = 0; k < 4; ++k) tc_mma(tmem, ad + 2 * k, bd + 2 * k, p.idesc, (kb | k) != 0);
            tc_commit(empty_bar(stage));
            if (++stage == p.stages) { stage = 0; phase ^= 1u; }
        }
        if (ok) tc_commit(tfull_bar);
        tc_commit(done_bar);
        const unsigned long long w0 = globaltimer_ns();
        while (!mbar_try_wait(done_bar, 0))
            if (globaltimer_ns() - w0 > kWaitLimitNs) break;
    } else if (warp >= 2) {
        // ---- epilogue: thread r owns TMEM lane r (one token) and the chunk's 32 columns
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const int et = (warp - 2) * 32 + lane;  // 0 .. 127 over the epilogue threads
        int ok = 1;
        if (lane == 0) ok = mbar_wait(tfull_bar, 0, &s_abort, p.status) ? 1 : 0;
        ok = __shfl_sync(~0u, ok, 0);
        const size_t list_base = (size_t)blockIdx.x * kTileRows;  // this CTA's lists
        const int nl = p.nch[pool];
        const int K = p.k;
        // A pool of one chunk needs no cross-CTA merge: the CTA keeps its lists
        // in shared memory and merges at once.  Shared scratch of the merge
        // (the ring is idle: all loads were consumed by the MMAs):
        float *sv = reinterpret_cast<float *>(dsmem + (sbase - smem_u32(dsmem)));  // [nl][128][K] scores
        uint16_t *se = reinterpret_cast<uint16_t *>(sv + nl * kTileRows * K);      // [nl][128][K] ids
        uint32_t *smask = reinterpret_cast<uint32_t *>(se + ((nl * kTileRows * K + 1) & ~1));  // [P][4] token bits
        uint32_t *scum = smask + 4 * 2 * kMaxPool;                                  // [P] tokens before words 1-3
        float4 *smeta = reinterpret_cast<float4 *>(scum + 2 * kMaxPool);           // [nl][128]
        if (ok) {
            __syncwarp();
            tc_fence_after();
            float v[32];
            int e[32];
            tmem_ld32(tmem + ((uint32_t)(q * 32) << 16), v);
            tmem_ld_wait();
            float mx = -INFINITY;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                float x = v[i];
                if (x != x) x = -INFINITY;  // NaN never outranks a number
                const bool in_pool = i < nvalid;
                v[i] = in_pool ? x : -INFINITY;
                e[i] = in_pool ? c0 + i : 0x7fffffff;  // columns past the pool rank below every expert
                mx = in_pool ? fmaxf(mx, x) : mx;
            }
            float ssum = 0.f;
            if (!p.renorm) {
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (i < nvalid) ssum += expf(v[i] - mx);
            }
            const int cnt = min(K, nvalid);
            // the chunk's best K pairs in rank order: k selection passes for
            // small K, the sorting network otherwise
            float2 *lst = p.lists + (list_base + r) * K;
            if (K <= 8) {
                uint32_t taken = nvalid >= 32 ? 0u : ~((1u << nvalid) - 1u);  // columns past the pool
                for (int j = 0; j < cnt; ++j) {
                    float bv;
                    int be;
                    const int bi = best_untaken(v, e, taken, bv, be);
                    taken |= 1u << bi;
                    if (nl == 1) {
                        sv[r * K + j] = bv;
                        se[r * K + j] = (uint16_t)be;
                    } else {
                        lst[j] = make_float2(bv, __int_as_float(be));
                    }
                }
            } else {
                sort32(v, e);
#pragma unroll
                for (int j = 0; j < 32; ++j)  // constant indices keep v, e in registers
                    if (j < K) {
                        if (nl == 1) {
                            sv[r * K + j] = v[j];
                            se[r * K + j] = (uint16_t)min(e[j], 0xffff);
                        } else {
                            lst[j] = make_float2(v[j], __int_as_float(e[j]));
                        }
                    }
            }
            if (nl == 1) smeta[r] = make_float4(mx, ssum, __int_as_float(cnt), 0.f);
            else p.meta[list_base + r] = make_float4(mx, ssum, __int_as_float(cnt), 0.f);
        }
        // publish, then count this chunk done for the tile; the CTA that
        // completes the tile merges (the fence orders the lists before the count)
        if (nl > 1) __threadfence();
        asm volatile("bar.sync 1, %0;\n" ::"r"(kEpi) : "memory");
        if (et == 0)
            s_last = ok && (nl == 1 || atomicAdd(&p.tile_done[slot], 1u) == (unsigned)(nl - 1));
        asm volatile("bar.sync 1, %0;\n" ::"r"(kEpi) : "memory");
        if (s_last) {
            if (nl > 1) {
                __threadfence();
                const size_t tile_lists = (size_t)slot * p.nch_max * kTileRows;
                constexpr int kB = 8;  // loads in flight per thread
                const int n_ent = nl * kTileRows * K;
                for (int i0 = et; i0 < n_ent; i0 += kB * kEpi) {
                    float2 x[kB];
#pragma unroll
                    for (int u = 0; u < kB; ++u)
                        if (i0 + u * kEpi < n_ent) x[u] = __ldcg(p.lists + tile_lists * K + i0 + u * kEpi);
#pragma unroll
                    for (int u = 0; u < kB; ++u)
                        if (i0 + u * kEpi < n_ent) {
                            sv[i0 + u * kEpi] = x[u].x;
                            se[i0 + u * kEpi] = (uint16_t)min(__float_as_int(x[u].y), 0xffff);
                        }
                }
                float4 m[kMaxChunks];
#pragma unroll
                for (int u = 0; u < kMaxChunks; ++u)
                    if (u < nl) m[u] = __ldcg(p.meta + tile_lists + u * kTileRows + et);
#pragma unroll
                for (int u = 0; u < kMaxChunks; ++u)
                    if (u < nl) smeta[u * kTileRows + et] = m[u];
            }
            for (int i = et; i < 4 * P; i += kEpi) smask[i] = 0u;
            asm volatile("bar.sync 1, %0;\n" ::"r"(kEpi) : "memory");
            // merge the chunk lists of token r in chunk order
            const bool valid = et < rows;
            float sel_v[kMaxTopK];
            int sel_e[kMaxTopK];
            float top = 0.f, S = 0.f;
            int npriv = 0;
            if (valid) {
                int head[kMaxChunks], n[kMaxChunks];
#pragma unroll
                for (int u = 0; u < kMaxChunks; ++u) {
                    head[u] = 0;
                    n[u] = u < nl ? __float_as_int(smeta[u * kTileRows + et].z) : 0;
                }
                for (int j = 0; j < K; ++j) {
                    int bu = -1, be = 0;
                    float bv = 0.f;
#pragma unroll
                    for (int u = 0; u < kMaxChunks; ++u) {
                        if (head[u] < n[u]) {
                            const int o = (u * kTileRows + et) * K + head[u];
                            const float x = sv[o];
                            const int ee = se[o];
                            if (bu < 0 || ranks_above(x, ee, bv, be)) { bu = u; bv = x; be = ee; }
                        }
                    }
                    if (bu < 0) break;  // unreachable for k <= pool size
#pragma unroll
                    for (int u = 0; u < kMaxChunks; ++u) head[u] += (u == bu) ? 1 : 0;
                    sel_v[j] = bv;
                    sel_e[j] = be;
                    if (j == 0) top = bv;
                    npriv += base + be >= p.E_pub;
                    atomicOr(&smask[be * 4 + (et >> 5)], 1u << (et & 31));
                }
                if (p.renorm) {
                    for (int j = 0; j < K; ++j) S += expf(sel_v[j] - top);
                } else {
                    for (int u = 0; u < nl; ++u) {  // fixed order: deterministic
                        const float4 m = smeta[u * kTileRows + et];
                        if (__float_as_int(m.z) > 0) S += m.y * expf(m.x - top);
                    }
                }
            }
            asm volatile("bar.sync 1, %0;\n" ::"r"(kEpi) : "memory");
            // the tile's rows per expert of the pool: its entries of tile_counts
            // (zeroed before the launch) and one global atomic per expert for the
            // totals; scum packs the tokens of mask words < 1, < 2, < 3 (8 bits each)
            for (int i = et; i < P; i += kEpi) {
                const uint32_t c0 = __popc(smask[i * 4]), c1 = __popc(smask[i * 4 + 1]);
                const uint32_t c2 = __popc(smask[i * 4 + 2]), c3 = __popc(smask[i * 4 + 3]);
                scum[i] = c0 | ((c0 + c1) << 8) | ((c0 + c1 + c2) << 16);
                const uint32_t c = c0 + c1 + c2 + c3;
                if (c) {
                    p.tile_counts[(size_t)(base + i) * p.slots4 + slot] = c;
                    atomicAdd(&p.counts[base + i], c);
                    if (p.route_count) atomicAdd(&p.route_count[base + i], c);
                }
            }
            asm volatile("bar.sync 1, %0;\n" ::"r"(kEpi) : "memory");
            if (valid) {
                const int t = s_tok[et];
                const int wd = et >> 5;
                const uint32_t below = (1u << (et & 31)) - 1u;
                for (int j = 0; j < K; ++j) {
                    const int be = sel_e[j];
                    // rank among the tile's rows of expert be: its tokens before t
                    const int rank = (int)__popc(smask[be * 4 + wd] & below) +
                                     (wd ? (int)((scum[be] >> (8 * (wd - 1))) & 0xffu) : 0);
                    p.idx[(size_t)t * K + j] = base + be;
                    p.ticket[(size_t)t * K + j] = (int32_t)(slot * kTileRows + rank);
                    p.w[(size_t)t * K + j] = expf(sel_v[j] - top) / S;
                }
                if (p.route_priv_rows) atomicAdd(&p.route_priv_rows[t], (unsigned)npriv);
            }
        }
    }

    // every warp reconverges before the block barrier: __syncthreads is a
    // warp-aligned barrier, and the single-thread roles above diverge from
    // their warps; TMEM is freed only after all epilogue reads completed
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kChunk);
    }
}

// ---------------------------------------------------------------------------
// router_cluster_kernel: the same routing with the reduction over H split
// across a cluster of nq CTAs (4, or 2 when H is not a multiple of 256, or 8
// for batches small enough to fit the GPU in clusters of 8) and no cross-CTA
// traffic through global memory.
//
// Each cluster takes one pool-homogeneous 128-token tile (the tile assignment
// of router_tc_kernel).  CTA q of the cluster multiplies the tile's token rows
// by the pool's router over the q-th 1/nq of H: tcgen05.mma with the router
// rows as M (128 experts per MMA, one or two MMAs for pools up to 256; rows
// past the pool read as zeros) and the 128 tokens as N, so the CTA reads
// H/nq of each token row and of each router row.  CTA q owns the tokens
// [q 128/nq, (q+1) 128/nq) of the tile.  Once every CTA of the cluster has
// finished its MMAs (a cluster barrier: the rings are then free), each CTA
// pushes its partial logits straight from tensor memory into the owner's
// shared memory with remote stores (distributed shared memory), one slot per
// source CTA; after a second barrier, the owner sums them in CTA order from
// its own shared memory (deterministic), masks, sorts each 32-expert chunk's
// best candidates with a bitonic network and merges the chunk lists of a
// token by lane shuffles.  The
// rank of each row among the tile's rows of its expert comes from the tile's
// 128-bit token mask per expert, whose words the CTAs of the cluster exchange
// after a third cluster barrier.  CTA 0 writes the tile's column of
// tile_counts for every expert (zero for the other pool), so nothing has to
// be cleared before the launch; a cluster whose slot holds no tile writes
// zeros there.  The dispatch sums the columns into the per-expert counts.
//
// Every CTA of a cluster reaches every cluster barrier: the waits before them
// are bounded, and a CTA that gave up skips work, not barriers.
constexpr int kCThreads = 192;       // warp 0 TMA, warp 1 TMEM + MMA, warps 2..5 gather / epilogue / finalize
constexpr int kCTile = 128;          // tokens per tile (MMA N)
constexpr int kCRingBytes = 192 * 1024;
// Staged partial logits: a token's row holds its 32-expert chunks at a stride
// of 36 floats, so that the lanes of a token, one chunk each, read different
// shared-memory banks in the selection (a stride of 32 put them all on one).
constexpr int kChunkPitch = 36;
__device__ __forceinline__ int chunk_pos(int e) { return (e >> 5) * kChunkPitch + (e & 31); }
constexpr int kCMaxStages = 6;

struct ClusterRouterParams {
    int T, H, E_pub, E_priv, k, renorm;
    int nq;              // CTAs per cluster: H is split into nq ranges
    int slots4;
    uint32_t idesc;      // M = 128, N = 128
    const uint8_t *policy;
    const bf16 *hidden;
    uint8_t *tau;
    int32_t *idx;
    float *w;
    int32_t *ticket;     // [T, k] 128 * tile slot + position among the tile's rows of its expert
    uint32_t *tile_counts;  // [E][slots4] rows of each expert per tile (a column per tile slot)
    uint32_t *route_count, *route_priv_rows, *status;
    uint32_t *gemm_bar;  // the expert launch's grid barrier counter, zeroed here
    // With dispatch != 0 (T <= 128: each pool fills at most one tile) the
    // router also writes the dispatch order, and clears the expert launch's
    // gemm_ready_words readiness counters, so that no dispatch step follows.
    int dispatch;
    uint32_t *offsets, *counts, *gemm_ready;
    int gemm_ready_words;
    int32_t *slot_of, *tok_of_slot;
    float *w_of_slot;
};

struct ClusterRouterMaps {
    CUtensorMap hidden;     // [T, H], box 64 x 128 (tiles of consecutive tokens)
    CUtensorMap router[2];  // [E_pool, H], box 64 x 128
};

// Shared-memory bytes of router_cluster_kernel for a pool of P experts (the
// larger pool), top-k k and nq CTAs per cluster: the ring, and after it the
// partial logits [128][P rounded to 128 + 4] FP32 with the chunk lists.
static int cluster_router_smem(int P, int k, int nq)
{
    const int pp = (P + 127) / 128 * 128;
    const int tpc = kCTile / nq;
    const int partial = kCTile * (pp / kChunk * kChunkPitch) * 4;  // staged partials, then the receive buffer
    const int lists = tpc * k * 8 + tpc * 8;
    const int after = 2 * partial + lists;
    return (after > kCRingBytes ? after : kCRingBytes) + 1024;
}

__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cluster_sync_all()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}
__device__ __forceinline__ uint32_t dsmem_addr(uint32_t local, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}
__device__ __forceinline__ uint32_t dsmem_ld_u32(uint32_t addr)
{
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];\n" : "=r"(v) : "r"(addr));
    return v;
}

// Bulk copy of `bytes` (a multiple of 16, both addresses 16-byte aligned)
// from this CTA's shared memory to a shared::cluster address of another CTA
// of the cluster, completing as transaction bytes on that CTA's mbarrier.
__device__ __forceinline__ void bulk_copy_to_peer(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t bar)
{
    asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(dst),
                 "r"(src), "r"(bytes), "r"(bar)
                 : "memory");
}
// Selection key of a logit of pool-local expert `id` (< 256): the logit's
// order-preserving 32-bit image with its low 8 bits replaced by 255 - id.
// Keys are unique and nonzero, compare like (logit desc, id asc) except
// between logits in the same 256-ulp bucket (key >> 8), and carry the id.
__device__ __forceinline__ uint32_t logit_key(float x, int id)
{
    x = x == 0.f ? 0.f : x;  // -0 and +0 are equal logits
    const uint32_t b = __float_as_uint(x);
    const uint32_t m = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
    return (m & 0xffffff00u) | (uint32_t)(255 - id);
}

// A summed logit as the mask treats it: NaN never outranks a number.
__device__ __forceinline__ float clean_logit(float x) { return x != x ? -INFINITY : x; }

// Finalize of the tile's tokens [q tpc, q tpc + ntok) owned by this CTA, by
// all threads of the CTA (a warp-uniform loop; the code is kept compact,
// since each CTA runs it once, from a cold instruction cache).
//
// Thread pair (token tl, chunk c) sums the chunk's 32 partial logits over
// the cluster's CTAs in CTA order (rcv[src][tl][expert]; the sums replace
// slot 0), turns them into selection keys held in registers and records the
// chunk's softmax partial (max, sum of exp(x - max)); experts past the pool
// have no key.  The ncp lanes of a token (ncp = chunks rounded up to a power
// of two; padding lanes hold no key) then take k + 1 passes: the group's
// largest key left (a max over the lane's keys, then over the lanes by
// shuffles), which its owner removes.  The keys of the passes are the candidates in key
// order; they are the exact top k in the exact order whenever no two
// consecutive ones of the first k + 1 share a bucket.  Otherwise (near-equal
// logits) the warp repeats the selection with the exact comparison of
// (logit, id).  The token's k pool-local ids go to sel_e, the logits to
// sel_v, its top logit and the softmax denominator (over the k selected
// logits, or over the whole pool from the chunk partials in chunk order) to
// tmeta, and every selected (expert, token) sets its bit in the CTA's mask.
__device__ void finalize_tokens(const ClusterRouterParams &p, float *rcv, int pitch, int q, int tpc,
                                int ntok, int nc, int P, float *sel_v, int *sel_e, float2 *tmeta,
                                uint32_t *smask)
{
    const int ncp = nc <= 1 ? 1 : (nc <= 2 ? 2 : (nc <= 4 ? 4 : 8));
    const int lg = ncp == 1 ? 0 : (ncp == 2 ? 1 : (ncp == 4 ? 2 : 3));
    const int npairs = tpc * ncp;
    const int K = p.k;
    for (int pb = 0; pb < npairs; pb += kCThreads) {  // the same trip count in every lane
        const int pi = pb + (int)threadIdx.x;
        const int tl = pi >> lg, c = pi & (ncp - 1);
        const bool tok_ok = pi < npairs && tl < ntok;
        const int nvalid = (tok_ok && c < nc) ? min(kChunk, P - c * kChunk) : 0;
        float *row = rcv + (size_t)(tok_ok ? tl : 0) * pitch;  // slot 0: the token's summed logits
        float *sum = row + c * kChunkPitch;
        float mx = -INFINITY, ssum = 0.f;
        uint32_t key[32];  // this lane's selection keys (0: no candidate)
#pragma unroll
        for (int i = 0; i < 32; ++i) key[i] = 0u;
        if (nvalid > 0) {
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = 0.f;
            for (int s2 = 0; s2 < p.nq; ++s2) {
                const float4 *r4 = reinterpret_cast<const float4 *>(sum + (size_t)s2 * tpc * pitch);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float4 x = r4[i];
                    v[4 * i] += x.x;
                    v[4 * i + 1] += x.y;
                    v[4 * i + 2] += x.z;
                    v[4 * i + 3] += x.w;
                }
            }
            float4 *w4 = reinterpret_cast<float4 *>(sum);
#pragma unroll
            for (int i = 0; i < 8; ++i) w4[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const float x = clean_logit(v[i]);
                key[i] = i < nvalid ? logit_key(x, c * kChunk + i) : 0u;
                mx = i < nvalid ? fmaxf(mx, x) : mx;
            }
            if (!p.renorm)
                for (int i = 0; i < nvalid; ++i) ssum += expf(clean_logit(sum[i]) - mx);
        }
        __syncwarp();
        // ---- fast path: k + 1 passes over the keys, held in registers
        bool amb = false;
        uint32_t prev = 0u;
        for (int j = 0; j <= K; ++j) {
            uint32_t m8[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) m8[i] = max(max(key[4 * i], key[4 * i + 1]), max(key[4 * i + 2], key[4 * i + 3]));
            uint32_t m = max(max(max(m8[0], m8[1]), max(m8[2], m8[3])), max(max(m8[4], m8[5]), max(m8[6], m8[7])));
            for (int d = 1; d < ncp; d <<= 1) m = max(m, __shfl_xor_sync(~0u, m, d));
            // keys are unique: the lane holding the winner removes it
#pragma unroll
            for (int i = 0; i < 32; ++i) key[i] = key[i] == m ? 0u : key[i];
            const int id = 255 - (int)(m & 255u);
            if (j > 0) amb |= (m >> 8) == (prev >> 8);
            if (j < K && c == 0 && tok_ok) sel_e[tl * K + j] = id;
            prev = m;
        }
        __syncwarp();
        amb &= tok_ok;
        if (__any_sync(~0u, amb)) {
            // ---- exact path for the whole warp: the chunk's logits in
            // registers (an entry taken, or past the pool, reads as (-inf, no
            // id), which never outranks a candidate); per pass a pairwise tree
            // of the exact comparison of (logit, id), ties to the lower id,
            // then the maximum over the token's lanes, whose owner removes it
            float xv[32];
            int xe[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const bool in = i < nvalid;
                xv[i] = in ? clean_logit(sum[i]) : -INFINITY;
                xe[i] = in ? c * kChunk + i : 0x7fffffff;
            }
            for (int j = 0; j < K; ++j) {
                float tv[16];
                int te[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const bool hi = ranks_above(xv[2 * i + 1], xe[2 * i + 1], xv[2 * i], xe[2 * i]);
                    tv[i] = hi ? xv[2 * i + 1] : xv[2 * i];
                    te[i] = hi ? xe[2 * i + 1] : xe[2 * i];
                }
#pragma unroll
                for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
                    for (int i = 0; i < w; ++i) {
                        const bool hi = ranks_above(tv[i + w], te[i + w], tv[i], te[i]);
                        tv[i] = hi ? tv[i + w] : tv[i];
                        te[i] = hi ? te[i + w] : te[i];
                    }
                float bv = tv[0];
                int be = te[0];
                for (int d = 1; d < ncp; d <<= 1) {
                    const float ov = __shfl_xor_sync(~0u, bv, d);
                    const int oe = __shfl_xor_sync(~0u, be, d);
                    if (ranks_above(ov, oe, bv, be)) {
                        bv = ov;
                        be = oe;
                    }
                }
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (xe[i] == be) {
                        xv[i] = -INFINITY;
                        xe[i] = 0x7fffffff;
                    }
                if (c == 0 && tok_ok) sel_e[tl * K + j] = be;
            }
            __syncwarp();
        }
        // ---- the selected logits, the mask bits, top and denominator
        float top = 0.f, den = 0.f;
        if (tok_ok) {
            const int tt = q * tpc + tl;
            for (int j = c; j < K; j += ncp) {
                const int e = sel_e[tl * K + j];
                sel_v[tl * K + j] = clean_logit(row[chunk_pos(e)]);
                atomicOr(&smask[e * 4 + (tt >> 5)], 1u << (tt & 31));
            }
            top = clean_logit(row[chunk_pos(sel_e[tl * K])]);
            if (p.renorm)
                for (int j = 0; j < K; ++j) den += expf(clean_logit(row[chunk_pos(sel_e[tl * K + j])]) - top);
        }
        if (!p.renorm) {
            const int g0 = (int)(threadIdx.x & 31) & ~(ncp - 1);
            for (int u = 0; u < ncp; ++u) {  // chunk order: deterministic
                const float mu = __shfl_sync(~0u, mx, g0 + u), su = __shfl_sync(~0u, ssum, g0 + u);
                if (u < nc) den += su * expf(mu - top);
            }
        }
        if (tok_ok && c == 0) tmeta[tl] = make_float2(top, den);
    }
}

__global__ void __launch_bounds__(kCThreads, 1) router_cluster_kernel(const ClusterRouterParams p,
                                                                       const __grid_constant__ ClusterRouterMaps maps)
{
    extern __shared__ uint8_t dsmem[];
    __shared__ int s_tok[kCTile];
    __shared__ int warp_tot[kCThreads / 32];
    __shared__ __align__(8) uint64_t bars[2 * kCMaxStages + 3];
    __shared__ uint32_t s_tmem;
    __shared__ volatile int s_abort;
    __shared__ uint32_t smask[kMaxPool * 4];  // this CTA's tokens of the tile, per pool expert, 4 x 32 bits
    __shared__ uint32_t sfull[kMaxPool * 4];  // the whole tile's mask (OR over the cluster)

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q = (int)cluster_ctarank();
    const int slot = blockIdx.x / p.nq;
    if (tid == 0) {
        prefetch_tmap(&maps.hidden);
        prefetch_tmap(&maps.router[0]);
        prefetch_tmap(&maps.router[1]);
    }
    pdl_trigger();
    pdl_wait();  // the caller's hidden states / policy may come from the previous kernel
    if (blockIdx.x == 0 && tid == 0 && p.gemm_bar) *p.gemm_bar = 0u;  // read by the expert launch after this grid
    if (p.dispatch && blockIdx.x == 0) {
        for (int i = tid; i < p.gemm_ready_words; i += kCThreads) p.gemm_ready[i] = 0u;
        if (tid == 0) p.offsets[p.E_pub + p.E_priv] = (uint32_t)(p.T * p.k);
    }

    // ---- tile assignment (as router_tc_kernel): resolve and rank in one pass
    const int per = ((p.T + kCThreads - 1) / kCThreads + 15) & ~15;
    const int t0 = min(p.T, tid * per), t1 = min(p.T, t0 + per);
    const int a = count_allow(p.policy, t0, t1);
    int na;
    const int a_before = block_scan(a, warp_tot, na);
    const int nd = p.T - na;
    const int tiles_d = (nd + kCTile - 1) / kCTile;
    int pool, m0;
    bool has_tile = true;
    if (slot < tiles_d) {
        pool = 0;
        m0 = slot * kCTile;
    } else {
        pool = 1;
        m0 = (slot - tiles_d) * kCTile;
        has_tile = m0 < na;
    }
    const int E = p.E_pub + p.E_priv;
    if (!has_tile) {  // uniform over the cluster: no tile for this slot
        if (q == 0) {
            for (int e = tid; e < E; e += kCThreads) p.tile_counts[(size_t)e * p.slots4 + slot] = 0u;
            if (p.dispatch) {  // a pool without tokens: its experts have no rows
                for (int e = tid; e < E; e += kCThreads)
                    if (e < p.E_pub ? nd == 0 : na == 0) {
                        p.offsets[e] = e < p.E_pub ? 0u : (uint32_t)(nd * p.k);
                        p.counts[e] = 0u;
                    }
            }
        }
        return;
    }
    const int rows = min(kCTile, (pool ? na : nd) - m0);
    if ((pool ? a_before : t0 - a_before) < m0 + rows && (pool ? a_before + a : t1 - a_before - a) > m0) {
        int ra = a_before, rd = t0 - a_before;
        for (int t = t0; t < t1; ++t) {
            const bool al = is_allow(p.policy, t);
            const int rank = al ? ra++ : rd++;
            if ((al ? 1 : 0) == pool && rank >= m0 && rank < m0 + rows) s_tok[rank - m0] = t;
        }
    }
    __syncthreads();
    for (int r = rows + tid; r < kCTile; r += kCThreads) s_tok[r] = s_tok[0];
    const int contiguous = __syncthreads_and(tid >= rows || s_tok[tid < kCTile ? tid : 0] == s_tok[0] + tid);

    const int P = pool ? p.E_priv : p.E_pub;
    const int base = pool ? p.E_pub : 0;
    const int nm = (P + 127) / 128;                 // MMAs of 128 experts
    const int pp = nm * 128;
    const int nc = (P + kChunk - 1) / kChunk;       // 32-expert chunks
    const int kq = p.H / p.nq, k0 = q * kq, nkb = kq / 64;
    const uint32_t a_bytes = (uint32_t)nm * 16384u, stage_bytes = a_bytes + 16384u;
    const int stages = min(kCMaxStages, kCRingBytes / (int)stage_bytes);
    const uint32_t sbase = (smem_u32(dsmem) + 1023u) & ~1023u;
    uint8_t *sgen = dsmem + (sbase - smem_u32(dsmem));
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int st) { return bar0 + 8u * st; };
    auto empty_bar = [&](int st) { return bar0 + 8u * (kCMaxStages + st); };
    const uint32_t tfull_bar = bar0 + 8u * (2 * kCMaxStages);
    const uint32_t done_bar = bar0 + 8u * (2 * kCMaxStages + 1);
    const uint32_t rcv_bar = bar0 + 8u * (2 * kCMaxStages + 2);  // partial logits received from the cluster
    const int tpc = kCTile / p.nq;
    const int pitch = pp / kChunk * kChunkPitch;  // floats per token row of partial logits
    const uint32_t slice_bytes = (uint32_t)(tpc * pitch * 4);  // one source CTA's partials of this CTA's tokens
    const uint32_t part_bytes = (uint32_t)(kCTile * pitch * 4);
    if (tid == 0) {
        for (int st = 0; st < stages; ++st) {
            mbar_init(full_bar(st), contiguous ? 2 : 1 + 128);
            mbar_init(empty_bar(st), 1);
        }
        mbar_init(tfull_bar, 1);
        mbar_init(done_bar, 1);
        mbar_init(rcv_bar, 1);
        mbar_expect_tx(rcv_bar, (uint32_t)p.nq * slice_bytes);
        s_abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    for (int i = tid; i < kMaxPool * 4; i += kCThreads) smask[i] = 0u;
    if (warp == 1) tmem_alloc(smem_u32(&s_tmem), 256);
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;

    if (warp == 0) {
        if (lane < (contiguous ? 2 : 1)) {
            // ---- TMA: lane 0 the router rows of this CTA's range of H, lane 1
            // the token rows when the tile's tokens are consecutive (a thread's
            // boxes are processed one after another: two lanes, two streams)
            const uint32_t tx = lane == 0 ? a_bytes : 16384u;
            uint32_t filled = 0, last_parity = 0;
            for (int kb = 0; kb < nkb; ++kb) {
                const int st = kb % stages;
                const uint32_t ph = (uint32_t)(kb / stages) & 1u;
                if (!mbar_wait(empty_bar(st), ph ^ 1u, &s_abort, p.status)) break;
                const uint32_t sA = sbase + st * stage_bytes, sB = sA + a_bytes;
                mbar_expect_tx(full_bar(st), tx);
                if (lane == 0) {
                    for (int mi = 0; mi < nm; ++mi)
                        tma_load_2d(sA + mi * 16384u, &maps.router[pool], full_bar(st), k0 + kb * 64, mi * 128);
                } else {
                    tma_load_2d(sB, &maps.hidden, full_bar(st), k0 + kb * 64, s_tok[0]);
                }
                filled |= 1u << st;
                last_parity = (last_parity & ~(1u << st)) | (ph << st);
            }
            for (int st = 0; st < stages; ++st)
                if ((filled >> st) & 1u) {
                    const unsigned long long w0 = globaltimer_ns();
                    while (!mbar_try_wait(full_bar(st), (last_parity >> st) & 1u))
                        if (globaltimer_ns() - w0 > kWaitLimitNs) break;
                }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---- MMA: logits[128 experts, 128 tokens] += router x rows^T per stage
            bool ok = true;
            for (int kb = 0; kb < nkb; ++kb) {
                const int st = kb % stages;
                const uint32_t ph = (uint32_t)(kb / stages) & 1u;
                if (!mbar_wait(full_bar(st), ph, &s_abort, p.status)) { ok = false; break; }
                tc_fence_after();
                fence_proxy_async_smem();  // gathered rows (generic proxy) read by the tensor cores
                const uint32_t sA = sbase + st * stage_bytes, sB = sA + a_bytes;
                const uint64_t bd = sw128_desc(sB);
                for (int mi = 0; mi < nm; ++mi) {
                    const uint64_t ad = sw128_desc(sA + mi * 16384u);
#pragma unroll
                    for (int k4 = 0; k4 < 4; ++k4)
                        tc_mma(tmem + (uint32_t)(mi * 128), ad + 2 * k4, bd + 2 * k4, p.idesc, (kb | k4) != 0);
                }
                tc_commit(empty_bar(st));
            }
            if (ok) tc_commit(tfull_bar);
            tc_commit(done_bar);
            const unsigned long long w0 = globaltimer_ns();
            while (!mbar_try_wait(done_bar, 0))
                if (globaltimer_ns() - w0 > kWaitLimitNs) break;
        }
    } else {
        // ---- gather (tiles of non-consecutive tokens): thread gi copies 16-byte
        // chunk (gi & 7) of tile rows (gi >> 3) + 16 j, swizzled as TMA would
        const int gi = tid - 64;
        if (!contiguous) {
            const int chunk = gi & 7, row0 = gi >> 3;
            const bf16 *src[8];
            uint32_t nbytes[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int r = row0 + 16 * j;
                const bool in = r < rows;
                src[j] = p.hidden + (in ? (size_t)s_tok[r] * p.H : 0) + k0 + chunk * 8;
                nbytes[j] = in ? 16u : 0u;
            }
            for (int kb = 0; kb < nkb; ++kb) {
                const int st = kb % stages;
                const uint32_t ph = (uint32_t)(kb / stages) & 1u;
                int free_ = 1;
                if (lane == 0) free_ = mbar_wait(empty_bar(st), ph ^ 1u, &s_abort, p.status) ? 1 : 0;
                free_ = __shfl_sync(~0u, free_, 0);
                if (!free_) break;
                const uint32_t sB = sbase + st * stage_bytes + a_bytes;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int r = row0 + 16 * j;
                    cp_async16(sB + r * 128 + ((chunk ^ (r & 7)) << 4), src[j] + kb * 64, (int)nbytes[j]);
                }
                cp_async_arrive_noinc(full_bar(st));
            }
            cp_async_wait<0>();
        }
        // ---- epilogue: the partial logits to shared memory, [token][expert]
        // FP32 (chunks of 32 experts at a stride of kChunkPitch; the ring is
        // free once every MMA has completed)
        int ok = 1;
        if (lane == 0) ok = mbar_wait(tfull_bar, 0, &s_abort, p.status) ? 1 : 0;
        ok = __shfl_sync(~0u, ok, 0);
        if (ok) {
            __syncwarp();
            tc_fence_after();
            const int quarter = warp & 3;
            float *S = reinterpret_cast<float *>(sgen);
            for (int mi = 0; mi < nm; ++mi) {
                const int e = mi * 128 + quarter * 32 + lane;
                for (int cc = 0; cc < kCTile / 32; ++cc) {
                    float v[32];
                    tmem_ld32(tmem + (uint32_t)(mi * 128 + cc * 32) + ((uint32_t)(quarter * 32) << 16), v);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) S[(cc * 32 + i) * pitch + chunk_pos(e)] = v[i];
                }
            }
            fence_proxy_async_smem();  // the bulk copies below read these rows
        }
    }
    __syncwarp();
    tc_fence_before();
    // #1: every CTA of the cluster has staged its partial logits, and every
    // ring is free to receive the others'
    cluster_sync_all();
    tc_fence_after();

    // ---- exchange: CTA q sends the rows of owner o's tokens [o tpc, (o + 1)
    // tpc) to slot q of o's receive buffer (after the staging rows) with one
    // bulk copy per owner, completing on o's rcv_bar; every CTA then waits
    // for its nq slots.  The wait is bounded but ignores the abort flag: no
    // copy into this CTA's shared memory may still be in flight at its exit.
    if (tid == 0) {
        for (int o = 0; o < p.nq; ++o)
            bulk_copy_to_peer(dsmem_addr(sbase + part_bytes + (uint32_t)q * slice_bytes, (uint32_t)o),
                              sbase + (uint32_t)o * slice_bytes, slice_bytes, dsmem_addr(rcv_bar, (uint32_t)o));
    }
    bool received = true;
    {
        const unsigned long long w0 = globaltimer_ns();
        while (!mbar_try_wait(rcv_bar, 0))
            if (globaltimer_ns() - w0 > kWaitLimitNs) {
                received = false;
                break;
            }
    }
    if (!received && tid == 0) {
        s_abort = 1;
        if (p.status) atomicOr(p.status, PMPE_STATUS_PIPELINE_TIMEOUT);
    }
    __syncthreads();

    // ---- finalize this CTA's tokens: per (token, 32-expert chunk) one thread
    // sums the chunk's partials over the cluster in CTA order, sorts its best
    // KP candidates (a bitonic network), and the ncp lanes of a token merge
    // their lists by shuffles into the token's top k
    const int ntok = max(0, min(rows - q * tpc, tpc));
    const int K = p.k;
    const bool abort_now = s_abort != 0;
    float *rcv = reinterpret_cast<float *>(sgen + part_bytes);                   // [nq][tpc][pitch]
    float *sel_v = reinterpret_cast<float *>(sgen + 2 * (size_t)part_bytes);     // [tpc][K] scores
    int *sel_e = reinterpret_cast<int *>(sel_v + (size_t)tpc * K);                // [tpc][K] pool-local ids
    float2 *tmeta = reinterpret_cast<float2 *>(sel_e + (size_t)tpc * K);          // [tpc] (top, denominator)
    if (!abort_now) {
        finalize_tokens(p, rcv, pitch, q, tpc, ntok, nc, P, sel_v, sel_e, tmeta, smask);
    }
    __syncthreads();
    cluster_sync_all();  // #2: every CTA's token masks are in its shared memory

    // ---- the tile's mask per expert (OR over the cluster), its counts, and
    // each row's position among the tile's rows of its expert (token order)
    for (int i0 = tid; i0 < P * 4; i0 += 2 * kCThreads) {  // up to 16 remote loads in flight per thread
        uint32_t m[2][8];
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int qq = 0; qq < 8; ++qq)
                m[u][qq] = (qq < p.nq && i0 + u * kCThreads < P * 4)
                               ? dsmem_ld_u32(dsmem_addr(smem_u32(&smask[i0 + u * kCThreads]), (uint32_t)qq))
                               : 0u;
#pragma unroll
        for (int u = 0; u < 2; ++u)
            if (i0 + u * kCThreads < P * 4) {
                uint32_t o = 0u;
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) o |= m[u][qq];
                sfull[i0 + u * kCThreads] = o;
            }
    }
    __syncthreads();
    if (q == 0) {
        for (int eg = tid; eg < E; eg += kCThreads) {
            const int i = eg - base;
            uint32_t c = 0u;
            if (i >= 0 && i < P)
                c = __popc(sfull[i * 4]) + __popc(sfull[i * 4 + 1]) + __popc(sfull[i * 4 + 2]) + __popc(sfull[i * 4 + 3]);
            p.tile_counts[(size_t)eg * p.slots4 + slot] = c;
            if (c && p.route_count) atomicAdd(&p.route_count[eg], c);
        }
    }
    // Dispatch order (when the tile is its pool's only one): the pool's rows
    // start after every earlier pool's (the public pool's nd tokens, k rows
    // each), its experts' rows follow one another in id order, and a row's
    // slot adds its position among its expert's rows of the tile, i.e. the
    // order offset[e] + (rows of e in earlier tiles, none) + position.
    uint32_t *s_first = reinterpret_cast<uint32_t *>(sgen);  // [P] first slot per pool expert (ring, free again)
    if (p.dispatch) {
        if (warp == 0) {
            uint32_t carry = pool ? (uint32_t)(nd * K) : 0u;
            for (int b = 0; b < P; b += 32) {
                const int i = b + lane;
                const uint32_t c =
                    i < P ? __popc(sfull[i * 4]) + __popc(sfull[i * 4 + 1]) + __popc(sfull[i * 4 + 2]) + __popc(sfull[i * 4 + 3])
                          : 0u;
                uint32_t v = c;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const uint32_t y = __shfl_up_sync(~0u, v, off);
                    if (lane >= off) v += y;
                }
                if (i < P) {
                    s_first[i] = carry + v - c;
                    if (q == 0) {
                        p.offsets[base + i] = carry + v - c;
                        p.counts[base + i] = c;
                    }
                }
                carry += __shfl_sync(~0u, v, 31);
            }
        }
        __syncthreads();
    }
    // one thread per routed row (token, j) of this CTA's tokens
    if (!abort_now) {
        for (int wi = tid; wi < ntok * K; wi += kCThreads) {
            const int tl = wi / K, j = wi - tl * K;
            const int tt = q * tpc + tl;
            const int t = s_tok[tt];
            const int wd = tt >> 5;
            const uint32_t below = (1u << (tt & 31)) - 1u;
            const int be = sel_e[wi];
            int rank = (int)__popc(sfull[be * 4 + wd] & below);
            for (int w2 = 0; w2 < wd; ++w2) rank += (int)__popc(sfull[be * 4 + w2]);
            const float2 m = tmeta[tl];
            const float wt = expf(sel_v[wi] - m.x) / m.y;
            p.idx[(size_t)t * K + j] = base + be;
            p.ticket[(size_t)t * K + j] = (int32_t)(slot * kCTile + rank);
            p.w[(size_t)t * K + j] = wt;
            if (p.dispatch) {
                const uint32_t sl = s_first[be] + (uint32_t)rank;
                if (sl < (uint32_t)(p.T * K)) {  // only a lost cluster exchange could fail this
                    p.slot_of[(size_t)t * K + j] = (int32_t)sl;
                    p.tok_of_slot[sl] = t;
                    p.w_of_slot[sl] = wt;
                }
            }
            if (j == 0) {
                p.tau[t] = pool ? 1 : 0;
                if (p.route_priv_rows) atomicAdd(&p.route_priv_rows[t], pool ? (unsigned)K : 0u);
            }
        }
    }
    __syncthreads();
    cluster_sync_all();  // #3: no CTA leaves while another still reads its shared memory
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

// Per-request policy bytes to per-token bytes, in one CTA: the offsets are
// checked first (cu[0] == 0, non-decreasing, cu[n] <= T); any violation is
// malformed metadata and every token becomes DENY.  Otherwise token t takes
// the byte of the request whose range holds it (the last request starting at
// or before t; empty requests hold no token), and tokens after cu[n] are DENY.
__global__ void __launch_bounds__(1024) policy_from_requests_kernel(const uint8_t *rp, const int32_t *cu, int n, int T,
                                                                    uint8_t *out)
{
    int bad = 0;
    if (threadIdx.x == 0) bad = (cu[0] != 0) | (cu[n] > T) | (n > 0 && rp == nullptr);
    for (int r = threadIdx.x; r < n; r += blockDim.x) bad |= cu[r + 1] < cu[r];
    const int any_bad = __syncthreads_or(bad);
    const int end = any_bad ? 0 : cu[n];
    for (int t = threadIdx.x; t < T; t += blockDim.x) {
        uint8_t v = 0x00;
        if (t < end) {
            int lo = 0, hi = n - 1;
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (cu[mid] <= t) lo = mid; else hi = mid - 1;
            }
            v = rp[lo];
        }
        out[t] = v;
    }
}

__global__ void resolve_kernel(const uint8_t *policy, int T, uint8_t *tau)
{
    for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T; t += gridDim.x * blockDim.x)
        tau[t] = (policy != nullptr && policy[t] == 0x01) ? 1 : 0;
}

}  // namespace

// Chunks of a pool (32 experts each) and the router's per-tile sizes.
int router_chunks(int pool_size) { return (pool_size + kChunk - 1) / kChunk; }
int router_slots(int T) { return (T + kTileRows - 1) / kTileRows + 1; }
int router_slots4(int T) { return (router_slots(T) + 3) & ~3; }

// The router of the unmasked control, and of shapes whose merge scratch does
// not fit router_cluster_kernel: one CTA per (tile, 32-expert chunk), the
// chunk lists merged by the tile's last CTA through global memory.
static cudaError_t launch_route_chunked(const Ctx &c)
{
    const Shape &s = c.s;
    RouterParams p;
    RouterMaps maps;
    memset(&maps, 0, sizeof(maps));
    p.T = s.T; p.H = s.H; p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.k = s.k; p.renorm = s.renorm;
    p.nch[0] = router_chunks(s.E_pub);
    p.nch[1] = router_chunks(s.E_priv);
    p.nch[2] = p.nch[0] + p.nch[1];
    p.unmasked = c.unmasked;
    p.nch_max = p.unmasked ? p.nch[2] : (p.nch[0] > p.nch[1] ? p.nch[0] : p.nch[1]);
    const int slots = router_slots(s.T);
    // per-expert counters, per-tile completion counts, the expert GEMMs'
    // readiness counters and the per-tile expert counts start at zero (the
    // workspace places them side by side: one memset clears all four)
    cudaError_t merr;
    const size_t nready = gemm_ready_words(s);
    const size_t ntc = (size_t)s.E() * router_slots4(s.T);
    // tile_counts starts 16-byte aligned right after gemm_ready (at most 3 words between)
    if (c.tile_done == c.counts + s.E() && c.gemm_ready == c.tile_done + slots &&
        c.tile_counts >= c.gemm_ready + nready && c.tile_counts <= c.gemm_ready + nready + 3) {
        merr = cudaMemsetAsync(c.counts, 0, sizeof(uint32_t) * (size_t)(c.tile_counts + ntc - c.counts), c.stream);
    } else {
        merr = cudaMemsetAsync(c.counts, 0, sizeof(uint32_t) * s.E(), c.stream);
        if (merr == cudaSuccess) merr = cudaMemsetAsync(c.tile_done, 0, sizeof(uint32_t) * slots, c.stream);
        if (merr == cudaSuccess) merr = cudaMemsetAsync(c.gemm_ready, 0, sizeof(uint32_t) * nready, c.stream);
        if (merr == cudaSuccess) merr = cudaMemsetAsync(c.tile_counts, 0, sizeof(uint32_t) * ntc, c.stream);
    }
    if (merr != cudaSuccess) return merr;
    p.idesc = make_idesc(kTileRows, kChunk);
    p.stages = kRMaxStages;
    p.policy = c.policy;
    p.hidden = c.hidden;
    p.rows_ws = c.router_rows;
    p.lists = c.router_lists;
    p.meta = c.router_meta;
    p.tile_done = c.tile_done;
    p.tau = c.tau;
    p.idx = c.idx;
    p.w = c.w;
    p.counts = c.counts;
    p.tile_counts = c.tile_counts;
    p.slots4 = router_slots4(s.T);
    p.ticket = c.ticket;
    p.route_count = c.audit.route_count;
    p.route_priv_rows = c.audit.route_priv_rows;
    p.status = c.audit.status;
    const int grid = slots * p.nch_max;
    bool ok = encode_2d(&maps.rows, c.router_rows, s.H, (uint64_t)grid * kTileRows, kTileRows);
    ok &= encode_2d(&maps.hidden, c.hidden, s.H, s.T, kTileRows);
    ok &= encode_2d(&maps.router[0], c.router_pub, s.H, s.E_pub, kChunk);
    ok &= encode_2d(&maps.router[1], c.router_priv, s.H, s.E_priv, kChunk);
    if (!ok) return cudaErrorInvalidValue;
    const int ring = p.stages * kStageBytes + 1024;
    const int merge = p.nch_max * kTileRows * s.k * 6 + 4 + 5 * 2 * kMaxPool * 4 + p.nch_max * kTileRows * 16 +
                      1024 + 16;
    const int smem = ring > merge ? ring : merge;
    static std::atomic<int> smem_limit[64];
    cudaError_t err = ensure_dynamic_smem(router_tc_kernel, smem, smem_limit);
    if (err != cudaSuccess) return err;
    return launch_pdl(router_tc_kernel, dim3(grid), dim3(kRThreads), smem, c.stream, p, maps);
}

// CTAs per cluster of router_cluster_kernel for hidden size H and T tokens
// (one CTA per SM): 8 when H allows and the clusters of 8 fit on the GPU at
// once, so that each CTA's share of H fits its ring in one round; else 4 (2
// when H is not a multiple of 256); and 2 when clusters of 4 would not fit
// the GPU in one wave (one wave of clusters of 2 measured faster than two
// waves of clusters of 4: 35 vs 57 us at T = 8192).
static int cluster_router_nq(int H, int T, int num_sms)
{
    if (H % 512 == 0 && router_slots(T) * 8 <= num_sms) return 8;
    if (router_slots(T) * 4 > num_sms) return 2;
    return H % 256 == 0 ? 4 : 2;
}
// Dynamic shared memory the cluster router may take beside its static arrays.
constexpr int kCMaxDynSmem = 208 * 1024;

bool route_uses_cluster_kernel(const Shape &s, int unmasked, int num_sms)
{
    if (unmasked) return false;
    const int P = s.E_pub > s.E_priv ? s.E_pub : s.E_priv;
    return cluster_router_smem(P, s.k, cluster_router_nq(s.H, s.T, num_sms)) <= kCMaxDynSmem;
}

bool route_writes_dispatch(const Ctx &c)
{
    return c.s.T <= kCTile && route_uses_cluster_kernel(c.s, c.unmasked, c.num_sms);
}

cudaError_t launch_route(const Ctx &c, bool write_dispatch)
{
    const Shape &s = c.s;
    if (!route_uses_cluster_kernel(s, c.unmasked, c.num_sms)) return write_dispatch ? cudaErrorInvalidValue : launch_route_chunked(c);
    ClusterRouterParams p;
    ClusterRouterMaps maps;
    memset(&p, 0, sizeof(p));
    memset(&maps, 0, sizeof(maps));
    p.T = s.T; p.H = s.H; p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.k = s.k; p.renorm = s.renorm;
    p.nq = cluster_router_nq(s.H, s.T, c.num_sms);
    p.slots4 = router_slots4(s.T);
    p.idesc = make_idesc(128, kCTile);
    p.policy = c.policy;
    p.hidden = c.hidden;
    p.tau = c.tau;
    p.idx = c.idx;
    p.w = c.w;
    p.ticket = c.ticket;
    p.tile_counts = c.tile_counts;
    p.route_count = c.audit.route_count;
    p.route_priv_rows = c.audit.route_priv_rows;
    p.status = c.audit.status;
    p.gemm_bar = c.gemm_ready + gemm_ready_words(s) - 1;
    if (write_dispatch) {
        if (s.T > kCTile) return cudaErrorInvalidValue;
        p.dispatch = 1;
        p.offsets = c.offsets;
        p.counts = c.counts;
        p.gemm_ready = c.gemm_ready;
        p.gemm_ready_words = (int)gemm_ready_words(s);
        p.slot_of = c.slot_of;
        p.tok_of_slot = c.tok_of_slot;
        p.w_of_slot = c.w_of_slot;
    }
    bool ok = encode_2d(&maps.hidden, c.hidden, s.H, s.T, kCTile);
    ok &= encode_2d(&maps.router[0], c.router_pub, s.H, s.E_pub, 128);
    ok &= encode_2d(&maps.router[1], c.router_priv, s.H, s.E_priv, 128);
    if (!ok) return cudaErrorInvalidValue;
    const int P = s.E_pub > s.E_priv ? s.E_pub : s.E_priv;
    const int smem = cluster_router_smem(P, s.k, p.nq);
    static std::atomic<int> smem_limit[64];
    cudaError_t err = ensure_dynamic_smem(router_cluster_kernel, smem, smem_limit);
    if (err != cudaSuccess) return err;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(router_slots(s.T) * p.nq);
    cfg.blockDim = dim3(kCThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = c.stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = p.nq;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, router_cluster_kernel, p, maps);
}

cudaError_t launch_policy_from_requests(const uint8_t *req_policy, const int32_t *cu_seqlens, int n_req, int T,
                                        uint8_t *policy_out, cudaStream_t stream)
{
    policy_from_requests_kernel<<<1, 1024, 0, stream>>>(req_policy, cu_seqlens, n_req, T, policy_out);
    return cudaGetLastError();
}

cudaError_t launch_resolve(const uint8_t *policy, int T, uint8_t *tau, cudaStream_t stream)
{
    const int threads = 256;
    int grid = (T + threads - 1) / threads;
    if (grid > 4096) grid = 4096;
    resolve_kernel<<<grid, threads, 0, stream>>>(policy, T, tau);
    return cudaGetLastError();
}

}  // namespace pmpe
