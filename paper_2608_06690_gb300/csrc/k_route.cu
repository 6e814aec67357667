// Stage 1 of the layer: fail-closed policy resolve, masked router, top-k and
// the route log (Sec. 3.1 Eq. 4; App. B.1 steps 2, 4, 5).
//
// router_tc_kernel: each CTA owns one 128-token tile of ONE pool.  It first
// resolves the policy bytes itself (only the trusted byte 0x01 is ALLOW) and
// ranks the tokens inside their pool, so that the DENY tokens form tiles
// 0 .. ceil(n_deny/128)-1 and the ALLOW tokens the tiles after them, each in
// ascending token order.  A TMA ring streams the tile's token rows and the
// pool's router rows as 128-byte-swizzled tiles into shared memory: straight
// from `hidden` when the tile's tokens are consecutive, otherwise from a
// contiguous workspace block the CTA first fills by token index (row gathers
// through TMA gather4 or cp.async ran 2.5-5x slower than copy + tile loads).
// tcgen05.mma computes the 128 x E_pool logits in tensor memory.  A DENY row
// is therefore only ever multiplied by public router rows and an ALLOW row
// only by private ones: an ineligible expert never becomes a candidate.
// Sixteen epilogue warps read the logits: four threads per token (one TMEM
// lane, four column slices) each select the top-k of their slice (descending
// score, ties to the lower expert id) by ordered passes with four independent
// selection chains, and one thread per token merges the four sorted lists and
// writes the softmax weights and the route log, and takes the row's position
// inside its expert (an integer atomic ticket) for the dispatch stage.
#include <cuda.h>

#include "pmpe_internal.cuh"
#include "tc_ptx.cuh"

namespace pmpe {
namespace {

constexpr int kEpiWarps = 16;    // 4 per TMEM lane quarter, each on a quarter of the logit columns
constexpr int kRThreads = 64 + 32 * kEpiWarps;  // warp 0 TMA, warp 1 TMEM + MMA, warps 2..17 epilogue
constexpr int kRMaxStages = 8;
constexpr int kTileRows = 128;
constexpr int kABytes = kTileRows * 128;  // 128 rows x 64 BF16

struct RouterParams {
    int T, H, E_pub, E_priv, k, renorm;
    int n_pad[2];        // MMA N of each pool: pool size rounded up to 16 (>= 16)
    uint32_t idesc[2];
    uint32_t tmem_cols;  // power of two >= max n_pad
    int stages;
    uint32_t stage_bytes;
    const uint8_t *policy;
    const bf16 *hidden;
    bf16 *rows_ws;       // [grid * 128, H] tile rows in pool order (workspace)
    uint8_t *tau;
    int32_t *idx;
    float *w;
    uint32_t *counts;  // per-expert row counters (zeroed before the launch)
    int32_t *ticket;   // [T, k] row position inside its expert
    uint32_t *route_count, *route_priv_rows, *status;
};

struct RouterMaps {
    CUtensorMap hidden;     // [T, H], box 64 x 128 (tiles of consecutive tokens)
    CUtensorMap rows;       // rows_ws, box 64 x 128 (copied tiles)
    CUtensorMap router[2];  // [E_pool, H], box 64 x n_pad
};

// Exclusive scan over the block of one int per thread (kRThreads threads).
__device__ __forceinline__ int block_scan(int v, int *warp_tot, int &total)
{
    constexpr int kW = kRThreads / 32;  // 18
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

// (x, e) ranks above (bx, be): larger logit, or equal logit and lower id.
__device__ __forceinline__ bool ranks_above(float x, int e, float bx, int be)
{
    return x > bx || (x == bx && e < be);
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

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    pdl_trigger();
    pdl_wait();  // the caller's hidden states / policy may come from the previous kernel

    // ---- resolve and rank: pass 1 counts the ALLOW tokens
    int my_allow = 0;
    for (int t = tid; t < p.T; t += kRThreads) my_allow += is_allow(p.policy, t);
    int na_total;
    block_scan(my_allow, warp_tot, na_total);
    const int na = na_total, nd = p.T - na;
    const int tiles_d = (nd + kTileRows - 1) / kTileRows;
    int pool, m0;
    if ((int)blockIdx.x < tiles_d) {
        pool = 0;
        m0 = blockIdx.x * kTileRows;
    } else {
        pool = 1;
        m0 = (blockIdx.x - tiles_d) * kTileRows;
        if (m0 >= na) return;  // uniform: no tile for this CTA
    }
    const int rows = min(kTileRows, (pool ? na : nd) - m0);
    // pass 2: each thread takes a contiguous run of tokens, ranks them in
    // their pool, and keeps the ones that fall into this CTA's tile
    {
        const int per = (p.T + kRThreads - 1) / kRThreads;
        const int t0 = tid * per, t1 = min(p.T, t0 + per);
        int a = 0;
        for (int t = t0; t < t1; ++t) a += is_allow(p.policy, t);
        int dummy;
        const int a_before = block_scan(a, warp_tot, dummy);
        int ra = a_before, rd = t0 - a_before;  // ranks inside the ALLOW / DENY pools
        for (int t = t0; t < t1; ++t) {
            const bool al = is_allow(p.policy, t);
            const int rank = al ? ra++ : rd++;
            if ((al ? 1 : 0) == pool && rank >= m0 && rank < m0 + rows) {
                s_tok[rank - m0] = t;
                p.tau[t] = al ? 1 : 0;  // every token is written by exactly one CTA
            }
        }
    }
    __syncthreads();
    for (int r = rows + tid; r < kTileRows; r += kRThreads) s_tok[r] = s_tok[0];  // padding rows name a real token
    // The TMA ring reads the tile's rows as one 128-row tile.  When the tile's
    // tokens are consecutive (a request with one policy) that tile is read
    // from `hidden` directly; otherwise the CTA first copies its token rows
    // into a contiguous block (padding rows are not copied: their logits are
    // never read) and makes the generic-proxy writes visible to the async
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
    if (warp == 1) tmem_alloc(smem_u32(&s_tmem), p.tmem_cols);
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    const int N = p.n_pad[pool];
    const int nkb = p.H / 64;

    if (warp == 0 && lane < 2) {
        // ---- TMA producers: lane 0 the 128 tile rows, lane 1 the pool's router
        // rows (one box each: boxes of one issuing thread are serialised)
        int stage = 0;
        uint32_t phase = 0, filled = 0, last_parity = 0;
        const uint32_t my_tx = lane == 0 ? (uint32_t)kABytes : (uint32_t)N * 128u;
        for (int kb = 0; kb < nkb; ++kb) {
            if (!mbar_wait(empty_bar(stage), phase ^ 1u, &s_abort, p.status)) break;
            const uint32_t sA = sbase + stage * p.stage_bytes, sB = sA + kABytes;
            mbar_expect_tx(full_bar(stage), my_tx);
            if (lane == 1)
                tma_load_2d(sB, &maps.router[pool], full_bar(stage), kb * 64, 0);
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
                const unsigned long long t0 = globaltimer_ns();
                while (!mbar_try_wait(full_bar(s), (last_parity >> s) & 1u))
                    if (globaltimer_ns() - t0 > kWaitLimitNs) break;
            }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer: logits[128, N] += rows[128, 64] x router[N, 64]^T per stage
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb) {
            if (!mbar_wait(full_bar(stage), phase, &s_abort, p.status)) { ok = false; break; }
            tc_fence_after();
            const uint32_t sA = sbase + stage * p.stage_bytes, sB = sA + kABytes;
            const uint64_t ad = sw128_desc(sA), bd = sw128_desc(sB);
#pragma unroll
            for (int k = 0; k < 4; ++k) tc_mma(tmem, ad + 2 * k, bd + 2 * k, p.idesc[pool], (kb | k) != 0);
            tc_commit(empty_bar(stage));
            if (++stage == p.stages) { stage = 0; phase ^= 1u; }
        }
        if (ok) tc_commit(tfull_bar);
        tc_commit(done_bar);
        const unsigned long long t0 = globaltimer_ns();
        while (!mbar_try_wait(done_bar, 0))
            if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    } else if (warp >= 2) {
        // ---- epilogue.  Thread (quarter q, slice sl) owns TMEM lane 32q + lane
        // (one token) and the logit columns of chunks sl, sl+4, ... (32 each);
        // it selects the top-k of its columns, then one thread per token merges
        // the four sorted slice lists.
        int ok = 1;
        if (lane == 0) ok = mbar_wait(tfull_bar, 0, &s_abort, p.status) ? 1 : 0;
        ok = __shfl_sync(~0u, ok, 0);
        const int q = warp & 3, sl = (warp - 2) >> 2;
        const int r = q * 32 + lane;
        const int P = pool ? p.E_priv : p.E_pub;
        const int base = pool ? p.E_pub : 0;
        float *lv = reinterpret_cast<float *>(dsmem + (sbase - smem_u32(dsmem)));  // [128][4][k] values
        int *li = reinterpret_cast<int *>(lv + kTileRows * 4 * p.k);               // [128][4][k] ids
        float *lmax = reinterpret_cast<float *>(li + kTileRows * 4 * p.k);          // [128][4]
        float *lsum = lmax + kTileRows * 4;                                          // [128][4]
        int *lcnt = reinterpret_cast<int *>(lsum + kTileRows * 4);                   // [128][4]
        if (ok) {
            __syncwarp();
            tc_fence_after();
            const uint32_t taddr = tmem + ((uint32_t)(q * 32) << 16);
            const int nch = (N + 31) / 32;
            const int my_cols = (sl < nch) ? min(P, N) : 0;  // any columns at all in this slice?
            int cnt = 0;
            float pv = 0.f, mx = -INFINITY;
            int pe = -1;
            const int slot = (r * 4 + sl) * p.k;
            for (int j = 0; j < p.k; ++j) {
                float bv = -INFINITY;
                int be = 0x7fffffff;
                for (int ch = sl; ch < nch; ch += 4) {
                    const int c0 = ch * 32;
                    float v[32];
                    tmem_ld32(taddr + c0, v);
                    tmem_ld_wait();
                    float cb[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                    int ce[4] = {0x7fffffff, 0x7fffffff, 0x7fffffff, 0x7fffffff};
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int e = c0 + i, u = i & 3;
                        float x = v[i];
                        if (x != x) x = -INFINITY;  // NaN never outranks a number
                        const bool after = (j == 0) || (x < pv) || (x == pv && e > pe);
                        if (e < P && after && (ce[u] == 0x7fffffff || x > cb[u])) { cb[u] = x; ce[u] = e; }
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (ce[u] != 0x7fffffff && (be == 0x7fffffff || ranks_above(cb[u], ce[u], bv, be))) {
                            bv = cb[u];
                            be = ce[u];
                        }
                }
                if (be == 0x7fffffff) break;  // this slice has no further column
                lv[slot + j] = bv;
                li[slot + j] = be;
                pv = bv;
                pe = be;
                if (cnt == 0) mx = bv;
                ++cnt;
            }
            // pool-softmax partial of this slice: sum of exp(x - slice max)
            float ssum = 0.f;
            if (!p.renorm && cnt > 0) {
                for (int ch = sl; ch < nch; ch += 4) {
                    const int c0 = ch * 32;
                    float v[32];
                    tmem_ld32(taddr + c0, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        float x = v[i];
                        if (x != x) x = -INFINITY;
                        if (c0 + i < P) ssum += expf(x - mx);
                    }
                }
            }
            (void)my_cols;
            lcnt[r * 4 + sl] = cnt;
            lmax[r * 4 + sl] = mx;
            lsum[r * 4 + sl] = ssum;
        }
        // all 16 epilogue warps: slice lists complete before the merge
        asm volatile("bar.sync 1, %0;\n" ::"r"(32 * kEpiWarps) : "memory");
        if (ok && sl == 0) {
            const bool valid = r < rows;
            const int t = s_tok[r];
            int head[4], n[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) { head[u] = 0; n[u] = lcnt[r * 4 + u]; }
            float sel_v[kMaxTopK];
            float top = 0.f;
            int npriv = 0;
            for (int j = 0; j < p.k; ++j) {
                int bu = -1;
                float bv = 0.f;
                int be = 0;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    if (head[u] < n[u]) {
                        const float x = lv[(r * 4 + u) * p.k + head[u]];
                        const int e = li[(r * 4 + u) * p.k + head[u]];
                        if (bu < 0 || ranks_above(x, e, bv, be)) { bu = u; bv = x; be = e; }
                    }
                }
                if (bu < 0) break;  // unreachable for k <= pool size
                head[bu] += 1;
                sel_v[j] = bv;
                if (j == 0) top = bv;
                const int gid = base + be;
                npriv += gid >= p.E_pub;
                if (valid) {
                    p.idx[(size_t)t * p.k + j] = gid;
                    // this row's position among the expert's rows (the dispatch
                    // stage adds the expert's offset)
                    p.ticket[(size_t)t * p.k + j] = (int32_t)atomicAdd(&p.counts[gid], 1u);
                    if (p.route_count) atomicAdd(&p.route_count[gid], 1u);
                }
            }
            float S = 0.f;
            if (p.renorm) {
                for (int j = 0; j < p.k; ++j) S += expf(sel_v[j] - top);
            } else {
#pragma unroll
                for (int u = 0; u < 4; ++u)  // fixed order: deterministic
                    if (n[u] > 0) S += lsum[r * 4 + u] * expf(lmax[r * 4 + u] - top);
            }
            if (valid) {
                for (int j = 0; j < p.k; ++j) p.w[(size_t)t * p.k + j] = expf(sel_v[j] - top) / S;
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
        tmem_dealloc(tmem, p.tmem_cols);
    }
}

__global__ void resolve_kernel(const uint8_t *policy, int T, uint8_t *tau)
{
    for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T; t += gridDim.x * blockDim.x)
        tau[t] = (policy != nullptr && policy[t] == 0x01) ? 1 : 0;
}

}  // namespace

cudaError_t launch_route(const Ctx &c)
{
    const Shape &s = c.s;
    cudaError_t merr = cudaMemsetAsync(c.counts, 0, sizeof(uint32_t) * s.E(), c.stream);
    if (merr != cudaSuccess) return merr;
    RouterParams p;
    RouterMaps maps;
    memset(&maps, 0, sizeof(maps));
    p.T = s.T; p.H = s.H; p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.k = s.k; p.renorm = s.renorm;
    int nmax = 0;
    for (int q = 0; q < 2; ++q) {
        const int P = q ? s.E_priv : s.E_pub;
        p.n_pad[q] = ((P < 16 ? 16 : P) + 15) & ~15;
        p.idesc[q] = make_idesc(kTileRows, p.n_pad[q]);
        nmax = p.n_pad[q] > nmax ? p.n_pad[q] : nmax;
    }
    p.tmem_cols = 32;
    while ((int)p.tmem_cols < nmax) p.tmem_cols <<= 1;
    p.stage_bytes = (uint32_t)(kABytes + nmax * 128);
    p.stages = (int)((200u * 1024u) / p.stage_bytes);
    if (p.stages > kRMaxStages) p.stages = kRMaxStages;
    p.policy = c.policy;
    p.hidden = c.hidden;
    p.rows_ws = c.router_rows;
    p.tau = c.tau;
    p.idx = c.idx;
    p.w = c.w;
    p.counts = c.counts;
    p.ticket = c.ticket;
    p.route_count = c.audit.route_count;
    p.route_priv_rows = c.audit.route_priv_rows;
    p.status = c.audit.status;
    const int grid = (s.T + kTileRows - 1) / kTileRows + 1;
    bool ok = encode_2d(&maps.rows, c.router_rows, s.H, (uint64_t)grid * kTileRows, kTileRows);
    ok &= encode_2d(&maps.hidden, c.hidden, s.H, s.T, kTileRows);
    ok &= encode_2d(&maps.router[0], c.router_pub, s.H, s.E_pub, p.n_pad[0]);
    ok &= encode_2d(&maps.router[1], c.router_priv, s.H, s.E_priv, p.n_pad[1]);
    if (!ok) return cudaErrorInvalidValue;
    // at least 116 KB of shared memory keeps one router CTA per SM, so the
    // TMEM allocation never waits for another CTA
    int smem = p.stages * (int)p.stage_bytes + 1024;
    if (smem < 116 * 1024) smem = 116 * 1024;
    const int lists = kTileRows * 4 * (s.k * 8 + 12) + 1024;  // top-k slice lists, reused after the MMAs
    if (smem < lists) smem = lists;
    cudaError_t err = cudaFuncSetAttribute(router_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (err != cudaSuccess) return err;
    return launch_pdl(router_tc_kernel, dim3(grid), dim3(kRThreads), smem, c.stream, p, maps);
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
