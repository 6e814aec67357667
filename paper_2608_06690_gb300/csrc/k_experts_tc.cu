// Stages 3 and 4 of the layer on the 5th-generation tensor cores: grouped
// BF16 expert GEMMs with tcgen05.mma accumulating in tensor memory (TMEM),
// operands staged into 128-byte-swizzled shared memory.
//
//   gate/up:  act = bf16(silu(A_e W_gate,e^T) * (A_e W_up,e^T))    (SwiGLU fused)
//   down:     y   = bf16(w_row * (act_e W_down,e^T))
//
// Groups are the routed experts (rows of the dispatch order) plus, with
// shared experts, one dense group over all T tokens (gate/up weights of the
// E_sh experts side by side; the down projection sums the E_sh experts in
// one accumulator).  A persistent grid (one CTA per SM) walks a tile list
// built on the device from the dispatch offsets: no host sync, and empty
// experts contribute no tile.  The list holds every gate/up tile, then every
// down tile, group by group, n-tile major inside a group.  The CTAs take the
// tiles in list order: in waves (CTA c: tiles c, c + grid, ...) when a group
// has several 128-row blocks, so that the m-tiles sharing weights run
// together, and otherwise dynamically, each CTA the next tile when its loader
// is ready for one (an atomic counter), which evens out tiles of unequal
// cost.  Warp 0 hands each tile index to the CTA's other roles through a
// small queue in shared memory.  A down tile waits (bounded) until the
// gate/up tiles of its activation rows have stored them; every one of those
// was handed out earlier to a running CTA, and no gate/up tile ever waits,
// so the wait ends.
//
// The routed gate/up tiles read their A rows straight from the hidden states:
// the row of dispatch slot r is hidden[tok_of_slot[r]], gathered into shared
// memory by four warps with 16-byte cp.async copies (the hidden states, read
// by every expert a token routes to, stay in L2), so the dispatched rows are
// never written out.  The gather warps never wait for their own copies: each
// thread's copies of a stage arrive on the stage's full barrier when they
// complete (cp.async.mbarrier.arrive), and the MMA thread fences the async
// proxy after that barrier, before the tensor cores read the rows.
//
// CTA roles (320 threads):
//   warp 0       three lanes issue the TMA loads of a 4-stage ring, one
//                operand box each (A: 128 rows x 64 K of the activations or,
//                for the shared group, of the hidden states; B: 256 rows x
//                64 K, i.e. 128 gate + 128 up rows, or 256 / 128 output
//                columns of the down projection in two halves)
//   warp 1       allocates 512 TMEM columns (two 128 x 256 FP32
//                accumulators, so the epilogue of one tile overlaps the MMAs
//                of the next) and one thread issues tcgen05.mma M=128 N=256
//                K=16, committing stage releases and accumulator-full events
//   warps 2..5   epilogue: tcgen05.ld of the warp's 32 TMEM lanes (= 32 tile
//                rows), SwiGLU or weight scaling, BF16 stores; in gate/up mode
//                the tiles of N-tile 0 also write the execution audit, each
//                row checked against the route log of its token
//   warps 6..9   the A-row gather of the routed gate/up tiles (cp.async into
//                the ring)
// Expert weights stream through L2 once and are loaded with an evict-first
// policy; the hidden states and activations, read again by other tiles of
// the launch, with evict-last.
// Every wait is bounded in time: on expiry the CTA records
// PMPE_STATUS_PIPELINE_TIMEOUT, stops issuing work, waits (bounded) for its
// own copies and MMAs in flight, frees its TMEM and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>

#include "pmpe_internal.cuh"
#include "tc_ptx.cuh"

namespace pmpe {
namespace {

constexpr int BM = 128;                       // rows per tile (MMA M)
constexpr int BK = 64;                        // K per stage: one 128-byte swizzle row
constexpr int kStages = 4;
constexpr int kABytes = BM * BK * 2;          // 16 KB
constexpr int kBBytes = 256 * BK * 2;         // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kAccCols = 256;                 // FP32 TMEM columns per accumulator
constexpr int kTmemCols = 2 * kAccCols;
constexpr int kGatherWarps = 4;               // warps 6..9
constexpr int kThreads = 192 + 32 * kGatherWarps;
constexpr int kLoaders = 3;                   // TMA-issuing lanes of warp 0
constexpr int kGatherThreads = 32 * kGatherWarps;
constexpr int kFullArrivals = kLoaders + kGatherThreads;  // per ring stage
constexpr int kMaxGroups = 2 * kMaxPool + 1;
constexpr int kPrefetchTiles = 96;            // gate/up tiles (1 MB of weights each) prefetched into L2 at small batches
// Large batches, the launch following the router: the gate and up weights of
// the list's first experts (at most 96 MiB, at most 16 experts) prefetched
// into L2 while the router runs, by the CTAs that start early, after a delay
// that lets the router's own reads of the token rows go first.
constexpr size_t kPrefillPrefetchBytes = 96ull << 20;
constexpr int kPrefillPrefetchExperts = 16;
constexpr unsigned long long kPrefillPrefetchDelayNs = 14000;
constexpr int kTQ = 8;                        // tile queue entries (tile indices handed to the CTA's roles)
constexpr int kTailWaves = 2;                 // waves of tiles at the list's end handed out dynamically
constexpr int kTQConsumers = 1 + 4 + kGatherWarps;  // MMA thread, epilogue warps, gather warps (one lane each)
constexpr int kOutBox = 32;                   // output staged and stored as 32 x 32 BF16 boxes (2 KB)
constexpr int kOutBufBytes = kOutBox * kOutBox * 2;
constexpr int kOutBytes = 4 * 2 * kOutBufBytes;  // 4 epilogue warps x 2 buffers
constexpr int kDynSmem = kStages * kStageBytes + kOutBytes + 1024 /* alignment slack */;

enum { kGateUp = 0, kDown = 1 };
enum { kTileGU = 0, kTileDown = 1 };

// One GEMM of the layer: gate/up (SwiGLU fused) or down (routing weight fused).
struct TcPhase {
    int bn;           // output columns per tile (gate/up: 128 activation columns; down: 256 or 128)
    uint32_t idesc;   // tcgen05 instruction descriptor (BF16 x BF16 -> FP32, M = 128, N = MMA width)
    bf16 *C_routed, *C_shared;
};

struct TcParams {
    // which GEMMs this launch runs: the gate/up tiles, the down tiles
    int has_gu, has_down;
    TcPhase ph[2];    // [kGateUp], [kDown]
    int E, E_pub, E_sh, T, H, I, R, k;
    const uint32_t *offsets;
    const float *w_of_slot;
    const int32_t *tok_of_slot;
    const int32_t *topk_idx;  // [T, k] the route log, read back by the execution audit
    const bf16 *hidden;       // the gather source of the routed gate/up tiles
    // has_gu && has_down: per (group, 128-row block), the gate/up epilogue
    // warps whose activations are stored (zeroed before the launch)
    uint32_t *ready;
    // the next tile of the list to hand out (zeroed before the launch): CTAs
    // take tiles in list order, each when it is ready for one
    uint32_t *tile_ctr;
    uint32_t *exec_rows, *exec_tiles, *exec_priv_rows, *shared_rows, *status;
    // fused dispatch (the launch follows the router directly): the CTAs first
    // derive the dispatch order from the router's per-tile counts and route
    // log, write the slot maps, clear the counters above, and meet at a grid
    // barrier (grid_bar, zeroed by the router) before the first tile
    int fuse_dispatch;
    const int32_t *ticket;      // [T, k] 128 * router tile + position among the tile's rows of its expert
    const float *w_route;       // [T, k] routing weights
    const uint32_t *tile_counts;  // [E][slots4] rows of each expert per router tile
    int slots, slots4;
    uint32_t *counts_w, *offsets_w;  // written: rows and first slot of each expert
    int32_t *slot_of_w, *tok_of_slot_w;
    float *w_of_slot_w;
    uint32_t *grid_bar;
    int clear_words;            // readiness counters and the tile counter, from `ready`
    // routing in the launch (T <= 128, nothing launched before this kernel
    // but the clearing of `ready`, the tile counter and the barriers): the
    // CTAs compute the masked router's logits, the top k, the routing weights
    // and the route log, then the dispatch order (route_in_launch)
    int fuse_route;
    int renorm;
    const uint8_t *policy;           // [T] policy bytes, or NULL (every token DENY)
    const bf16 *router_w[2];         // [E_pub, H] public, [E_priv, H] private router
    float *z;                        // [T][zpitch] logits of each token's pool (scratch)
    int zpitch;
    int32_t *idx_w, *ticket_w;       // [T, k] route log written
    float *w_w;                      // [T, k] routing weights written
    uint8_t *tau_w;                  // [T]
    uint32_t *tile_counts_w;         // [E][slots4]
    uint32_t *route_count, *route_priv_rows;
    uint32_t *bar_a, *bar_b;         // grid barriers after the logits and after the selection
    // with fuse_route: the weighted combine too, after a last grid barrier
    // (bar_d) once every CTA's down tiles are stored
    int fuse_combine;
    uint32_t *bar_d;
    bf16 *out;                       // [T, H]
    // small batches (every expert at most one 128-row block): the first
    // `prefetch_tiles` gate/up tiles of the list of all experts have their
    // weights prefetched into L2 by the CTA of the same index, before the
    // launch waits for the routing (the weights are inputs, not results of
    // the kernels before); 0 = off
    int prefetch_tiles;
    int prefetch_experts;      // large batches: CTA e < this prefetches expert e's gate and up rows
    const bf16 *gate_w[2], *up_w[2];  // [E_pool * I, H] public / private
    // optional FP32: the gate and up accumulators saved for the backward,
    // [R][2I] G | U of the routed rows, then [T][2 E_sh I] of the shared
    // experts (gu_save / gu_save_sh maps for whole 32-row blocks)
    float *saved_gu;
};

struct TcMaps {  // [phase]
    CUtensorMap c_routed[2], c_shared[2];  // outputs, 32 x 32 boxes, 64-byte swizzle
    CUtensorMap a_routed[2], a_shared[2];
    CUtensorMap b0[2][3];  // per pool [pub, priv, shared]: gate (gate/up) or down
    CUtensorMap b1[2][3];  // up (gate/up)
    CUtensorMap gu_save;   // saved_gu, routed rows [R][2I], 16 x 32 FP32 boxes, 64-byte swizzle
    CUtensorMap gu_save_sh;  // saved_gu's shared part [T][2 E_sh I], the same boxes
};

// ------------------------------------------------------------- tile list

struct Tile {
    int kind, ph, bn, g, m_tile, m0, n0, rows, row_base, nkb, cb;
    bool shared;
};

struct TileTable {
    int prefix[2][kMaxGroups + 1];  // tiles of the groups before g, per GEMM
    int mpre[kMaxGroups + 1];       // 128-row blocks of the groups before g
    int rows[kMaxGroups];
    int base[kMaxGroups];
};

__device__ __forceinline__ int group_n(const TcParams &p, int mode, bool shared)
{
    return mode == kGateUp ? (shared ? p.E_sh * p.I : p.I) : p.H;
}
__device__ __forceinline__ int group_k(const TcParams &p, int mode, bool shared)
{
    return mode == kGateUp ? p.H : (shared ? p.E_sh * p.I : p.I);
}

__device__ __forceinline__ int total_tiles(const TcParams &p, const TileTable &tt, int G)
{
    return (p.has_gu ? tt.prefix[kGateUp][G] : 0) + (p.has_down ? tt.prefix[kDown][G] : 0);
}

// The down GEMM's order of the groups: with shared experts their group sits
// after the first half of the routed experts, so that the list ends with
// routed down tiles (K = I) instead of the shared group's (K = E_sh I, the
// launch's longest tiles), which otherwise made the last wave uneven; there
// the shared group's gate/up tiles, the last of the gate/up list, are long
// finished.  The gate/up GEMM keeps the groups in id order (the copy warps
// fill no stage after one whose A comes through TMA).  down_place inverts it.
__device__ __forceinline__ int down_group(const TcParams &p, int L)
{
    if (p.E_sh == 0) return L;
    const int h = p.E / 2;
    return L < h ? L : (L == h ? p.E : L - 1);
}
__device__ __forceinline__ int down_place(const TcParams &p, int g)
{
    if (p.E_sh == 0) return g;
    const int h = p.E / 2;
    return g < h ? g : (g == p.E ? h : g + 1);
}

// Tile `tile` of the list: the gate/up tiles (when this launch runs them),
// then the down tiles; inside a GEMM, group by group (the down GEMM in
// down_group order), n-tile major.
__device__ __forceinline__ Tile decode_tile(const TcParams &p, const TileTable &tt, int G, int tile)
{
    Tile t;
    const int n_gu = p.has_gu ? tt.prefix[kGateUp][G] : 0;
    t.ph = tile < n_gu ? kGateUp : kDown;
    t.kind = t.ph == kGateUp ? kTileGU : kTileDown;
    const int local_all = tile - (t.ph == kDown ? n_gu : 0);
    const int *pre = tt.prefix[t.ph];
    int lo = 0, hi = G - 1;  // last group with prefix <= local_all
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (pre[mid] <= local_all) lo = mid; else hi = mid - 1;
    }
    t.bn = p.ph[t.ph].bn;
    const int g = t.ph == kDown ? down_group(p, lo) : lo;
    t.g = g;
    t.shared = g >= p.E;
    const int rows = tt.rows[g];
    const int mt = (rows + BM - 1) / BM;
    const int local = local_all - pre[lo];
    const int n_tile = local / mt;
    t.m_tile = local - n_tile * mt;
    t.m0 = t.m_tile * BM;
    t.n0 = n_tile * t.bn;
    t.cb = n_tile;
    t.rows = min(BM, rows - t.m0);
    t.row_base = tt.base[g];
    t.nkb = group_k(p, t.ph == kGateUp ? kGateUp : kDown, t.shared) / BK;
    return t;
}

// ---------------------------------------------------------------- kernel

// Weights of gate/up tile blockIdx.x of the list of all experts (the first
// wave when every expert has at most one 128-row block): 128 gate rows and
// 128 up rows, each block contiguous, prefetched into L2 by one thread.
__device__ __forceinline__ void prefetch_first_wave(const TcParams &p)
{
    const int nt = p.I / 128;
    const int e = (int)blockIdx.x / nt, n = (int)blockIdx.x - e * nt;
    if (e < p.E) {
        const int q = e < p.E_pub ? 0 : 1;
        const size_t row0 = (size_t)(q ? e - p.E_pub : e) * p.I + (size_t)n * 128;
        const uint32_t bytes = (uint32_t)(128u * (uint32_t)p.H * 2u);
        bulk_prefetch_l2(p.gate_w[q] + row0 * p.H, bytes);
        bulk_prefetch_l2(p.up_w[q] + row0 * p.H, bytes);
    }
}

// Arrival at a grid barrier: a release add, so that the writes the CTA
// barrier before it ordered (every thread's) are visible to whoever
// acquires the count.
__device__ __forceinline__ void grid_arrive(uint32_t *ctr)
{
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;\n" ::"l"(ctr) : "memory");
}

// Every CTA of the grid arrives (after all of its threads' writes), then
// waits, bounded, until `target` arrivals are counted (acquire loads; the CTA
// barrier after them orders the other threads); writes before the barrier,
// by any thread of any CTA, are visible after it.  The grid is resident all
// at once (checked before the launch).  False after a timeout or an abort.
// (A release add and a tight acquire spin measured 0.5 us faster a decode
// step than a full fence, a relaxed add and a spin with back-off.)
__device__ bool grid_barrier(uint32_t *ctr, uint32_t target, volatile int *abort_flag, uint32_t *status)
{
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        int ok = 1;
        grid_arrive(ctr);
        const unsigned long long t0 = globaltimer_ns();
        while (ld_acquire_gpu(ctr) < target) {
            if (*abort_flag) { ok = 0; break; }
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                *abort_flag = 1;
                if (status) atomicOr(status, PMPE_STATUS_PIPELINE_TIMEOUT);
                ok = 0;
                break;
            }
        }
        s_ok = ok;
    }
    __syncthreads();
    return s_ok != 0;
}

constexpr int kRouteMaxTokens = 128;   // routing in the launch: one selection CTA per token
constexpr int kRouteMaxH = 2048;       // the logits hold a row's 16-byte pieces in registers, 8 a lane at most
constexpr int kRouteXChunks = kRouteMaxH / 256;  // 16-byte pieces of the token row per lane

__device__ __forceinline__ float dot8_bf16(const uint4 &a, const uint4 &b, float acc)
{
    const __nv_bfloat162 *x = reinterpret_cast<const __nv_bfloat162 *>(&a);
    const __nv_bfloat162 *y = reinterpret_cast<const __nv_bfloat162 *>(&b);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 u = __bfloat1622float2(x[i]), v = __bfloat1622float2(y[i]);
        acc = fmaf(u.x, v.x, acc);
        acc = fmaf(u.y, v.y, acc);
    }
    return acc;
}

// Exact ranking of two candidates (logit, pool-local id): the larger logit,
// at equal logits the lower id (NaN was cleaned to -inf before).
__device__ __forceinline__ bool route_above(float x, int e, float bx, int be)
{
    return (x > bx) | ((x == bx) & (e < be));
}

// Routing inside the persistent launch, for T <= 128 tokens (Sec. 3.1 Eq. 4
// and App. B.1), in three steps separated by grid barriers:
//   1. logits: work items (token t, block c of t's pool), spread over the
//      CTAs, at most one each; each warp of a CTA forms the dot products of its
//      experts with the token row (FP32: a lane's 16-byte pieces in order,
//      then a butterfly), into z[t][e].  A token meets only its own pool's
//      router rows.
//   2. selection: CTA t < T, one warp: the top k of z[t] by k passes of an
//      exact (logit, id) maximum, ties to the lower id; the weights (softmax
//      over the k, or over the pool); the route log.
//   3. dispatch: every CTA forms per expert the mask of the tokens that
//      picked it, the counts and first slots (experts in id order, tokens in
//      order), and resolves its share of the routed rows (slot = first slot
//      + rank of the token among the expert's tokens).  The tile table takes
//      the counts and first slots; the caller then arrives at grid_bar.
// Returns false after an abort (a barrier timed out).
__device__ bool route_in_launch(const TcParams &p, uint8_t *ring, TileTable &tt, volatile int *s_abort)
{
    __shared__ int s_item[kRouteMaxTokens + 1];  // items of the tokens before t
    __shared__ uint8_t s_tau[kRouteMaxTokens];
    __shared__ int s_nd;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    constexpr int kWarps = kThreads / 32;
    const int T = p.T, K = p.k, E = p.E, E_priv = p.E - p.E_pub, R = p.R;
    // ---- tau per token (Sec. 2.1) and the logit work items: (token, block
    // of bs experts of its pool), bs the least size from 32 up that gives
    // every CTA at most one item (a CTA's item is a chain of dependent load
    // rounds, so two items on one CTA would double the step)
    __shared__ int s_bs;
    if (warp == 0) {
        int nd = 0;
        for (int b0 = 0; b0 < T; b0 += 32) {
            const int t = b0 + lane;
            const int tau = (t < T && p.policy) ? (p.policy[t] == 0x01 ? 1 : 0) : 0;
            if (t < T) s_tau[t] = (uint8_t)tau;
            nd += __popc(__ballot_sync(~0u, t < T && tau == 0));
        }
        const int na = T - nd;
        int bs = 256;  // one item per token always fits (T <= the grid)
        for (int b1 = 32; b1 < 256; b1 += 32) {  // the lanes test 32 sizes at a time
            const int c = b1 + lane;
            const bool fits = nd * ((p.E_pub + c - 1) / c) + na * ((E_priv + c - 1) / c) <= (int)gridDim.x;
            const unsigned m = __ballot_sync(~0u, fits);
            if (m) {
                bs = b1 + __ffs(m) - 1;
                break;
            }
        }
        int carry = 0;
        for (int b0 = 0; b0 < T; b0 += 32) {
            const int t = b0 + lane;
            const int v0 = t < T ? ((s_tau[t] ? E_priv : p.E_pub) + bs - 1) / bs : 0;
            int v = v0;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(~0u, v, off);
                if (lane >= off) v += y;
            }
            if (t < T) s_item[t] = carry + v - v0;
            carry += __shfl_sync(~0u, v, 31);
        }
        if (lane == 0) {
            s_item[T] = carry;
            s_nd = nd;
            s_bs = bs;
        }
    }
    __syncthreads();
    const int nitems = s_item[T], nd = s_nd, bs = s_bs;
    const int nch = p.H / 8;  // 16-byte pieces of a row
    // ---- 1. logits (loads straight into registers: each warp takes its
    // experts two at a time, so that a lane has 16 loads of 16 bytes in
    // flight; bulk copies of the block into shared memory were slower)
    for (int i = (int)blockIdx.x; i < nitems; i += (int)gridDim.x) {
        int lo = 0, hi = T - 1;  // the token of item i: the last t with s_item[t] <= i
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_item[mid] <= i) lo = mid; else hi = mid - 1;
        }
        const int t = lo, tau = s_tau[t];
        const int e0 = (i - s_item[t]) * bs;
        const int ne = min(bs, (tau ? E_priv : p.E_pub) - e0);
        const uint4 *xrow = reinterpret_cast<const uint4 *>(p.hidden + (size_t)t * p.H);
        const uint4 *wblk = reinterpret_cast<const uint4 *>(p.router_w[tau] + (size_t)e0 * p.H);
        uint4 xr[kRouteXChunks];
#pragma unroll
        for (int q = 0; q < kRouteXChunks; ++q) {
            const int ch = lane + 32 * q;
            xr[q] = ch < nch ? __ldg(xrow + ch) : make_uint4(0u, 0u, 0u, 0u);
        }
        for (int e = warp; e < ne; e += 2 * kWarps) {
            const int e2 = e + kWarps;  // the second expert of the pair (absent past the block)
            uint4 wa[kRouteXChunks], wb[kRouteXChunks];
#pragma unroll
            for (int q = 0; q < kRouteXChunks; ++q) {
                const int ch = lane + 32 * q;
                wa[q] = ch < nch ? __ldg(wblk + (size_t)e * nch + ch) : make_uint4(0u, 0u, 0u, 0u);
                wb[q] = (ch < nch && e2 < ne) ? __ldg(wblk + (size_t)e2 * nch + ch) : make_uint4(0u, 0u, 0u, 0u);
            }
            float acc_a = 0.f, acc_b = 0.f;
#pragma unroll
            for (int q = 0; q < kRouteXChunks; ++q) {
                if (lane + 32 * q < nch) {
                    acc_a = dot8_bf16(wa[q], xr[q], acc_a);
                    acc_b = dot8_bf16(wb[q], xr[q], acc_b);
                }
            }
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) {
                acc_a += __shfl_xor_sync(~0u, acc_a, off);
                acc_b += __shfl_xor_sync(~0u, acc_b, off);
            }
            if (lane == 0) {
                p.z[(size_t)t * p.zpitch + e0 + e] = acc_a;
                if (e2 < ne) p.z[(size_t)t * p.zpitch + e0 + e2] = acc_b;
            }
        }
    }
    if (!grid_barrier(p.bar_a, gridDim.x, s_abort, p.status)) return false;
    // the first wave's weights into L2 while the selection and the dispatch
    // run (not earlier: the prefetch would delay the router rows)
    if (warp == 2 && lane == 0 && (int)blockIdx.x < p.prefetch_tiles) prefetch_first_wave(p);
    // ---- 2. selection, one warp per token
    if ((int)blockIdx.x < T && warp == 0) {
        const int t = (int)blockIdx.x, tau = s_tau[t];
        const int P = tau ? E_priv : p.E_pub, base = tau ? p.E_pub : 0;
        const float *zt = p.z + (size_t)t * p.zpitch;
        float v[8], vo[8];
        int id[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int e = lane + 32 * q;
            const float x = e < P ? zt[e] : -INFINITY;
            vo[q] = v[q] = x != x ? -INFINITY : x;  // NaN never outranks a number
            id[q] = e < P ? e : 0x7fffffff;
        }
        float my_v = 0.f, top = 0.f;
        int my_e = 0;
        for (int j = 0; j < K; ++j) {
            float bv = v[0];
            int be = id[0];
#pragma unroll
            for (int q = 1; q < 8; ++q)
                if (route_above(v[q], id[q], bv, be)) {
                    bv = v[q];
                    be = id[q];
                }
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) {
                const float ov = __shfl_xor_sync(~0u, bv, off);
                const int oe = __shfl_xor_sync(~0u, be, off);
                if (route_above(ov, oe, bv, be)) {
                    bv = ov;
                    be = oe;
                }
            }
#pragma unroll
            for (int q = 0; q < 8; ++q)
                if (id[q] == be) {
                    v[q] = -INFINITY;
                    id[q] = 0x7fffffff;
                }
            if (lane == j) {
                my_v = bv;
                my_e = be;
            }
            if (j == 0) top = bv;
        }
        float den = 0.f;
        if (p.renorm) {  // softmax over the k selected logits, in rank order
            for (int j = 0; j < K; ++j) den += expf(__shfl_sync(~0u, my_v, j) - top);
        } else {         // softmax over the pool
#pragma unroll
            for (int q = 0; q < 8; ++q)
                if (lane + 32 * q < P) den += expf(vo[q] - top);
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) den += __shfl_xor_sync(~0u, den, off);
        }
        if (lane < K) {
            p.idx_w[(size_t)t * K + lane] = base + my_e;
            p.w_w[(size_t)t * K + lane] = expf(my_v - top) / den;
            if (p.route_count) atomicAdd(&p.route_count[base + my_e], 1u);
        }
        if (lane == 0) {
            p.tau_w[t] = (uint8_t)tau;
            if (p.route_priv_rows) atomicAdd(&p.route_priv_rows[t], tau ? (unsigned)K : 0u);
        }
    }
    if (!grid_barrier(p.bar_b, gridDim.x, s_abort, p.status)) return false;
    // ---- 3. dispatch order: per expert the mask of its tokens (4 x 32 bits)
    uint32_t *smask = reinterpret_cast<uint32_t *>(ring);
    int *sfirst = reinterpret_cast<int *>(smask + (size_t)E * 4);
    int *scount = sfirst + E;
    for (int i = tid; i < E * 4; i += kThreads) smask[i] = 0u;
    __syncthreads();
    for (int r = tid; r < R; r += kThreads) {
        const int e = p.idx_w[r], t = r / K;
        if ((unsigned)e < (unsigned)E) atomicOr(&smask[e * 4 + (t >> 5)], 1u << (t & 31));
    }
    __syncthreads();
    if (warp == 0) {  // rows per expert and their exclusive prefix: the first slots
        int carry = 0;
        for (int b0 = 0; b0 < E; b0 += 32) {
            const int g = b0 + lane;
            const int v0 = g < E ? __popc(smask[g * 4]) + __popc(smask[g * 4 + 1]) + __popc(smask[g * 4 + 2]) +
                                       __popc(smask[g * 4 + 3])
                                 : 0;
            int v = v0;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(~0u, v, off);
                if (lane >= off) v += y;
            }
            if (g < E) {
                sfirst[g] = carry + v - v0;
                scount[g] = v0;
            }
            carry += __shfl_sync(~0u, v, 31);
        }
    }
    __syncthreads();
    // the router tile of a pool's tokens (the cluster router's numbering:
    // the DENY tile first when there are DENY tokens)
    auto tile_of = [&](int g) { return g < p.E_pub ? 0 : (nd > 0 ? 1 : 0); };
    if (blockIdx.x == 0) {
        for (int g = tid; g < E; g += kThreads) {
            p.offsets_w[g] = (uint32_t)sfirst[g];
            p.counts_w[g] = (uint32_t)scount[g];
            for (int sl = 0; sl < p.slots; ++sl)
                p.tile_counts_w[(size_t)g * p.slots4 + sl] = sl == tile_of(g) ? (uint32_t)scount[g] : 0u;
        }
        if (tid == 0) p.offsets_w[E] = (uint32_t)R;
    }
    for (int r = (int)blockIdx.x * kThreads + tid; r < R; r += (int)gridDim.x * kThreads) {
        const int e = p.idx_w[r], t = r / K;
        if ((unsigned)e >= (unsigned)E) {  // never produced by the selection
            if (p.status) atomicOr(p.status, PMPE_STATUS_BAD_EXPERT_ID);
            continue;
        }
        const int wd = t >> 5;
        int rank = __popc(smask[e * 4 + wd] & ((1u << (t & 31)) - 1u));
        for (int w2 = 0; w2 < wd; ++w2) rank += __popc(smask[e * 4 + w2]);
        const int slot = sfirst[e] + rank;
        if ((unsigned)slot >= (unsigned)R) continue;
        p.slot_of_w[r] = slot;
        p.tok_of_slot_w[slot] = t;
        p.w_of_slot_w[slot] = p.w_w[r];
        p.ticket_w[r] = tile_of(e) * 128 + rank;
    }
    for (int g = tid; g < E; g += kThreads) {
        tt.rows[g] = scount[g];
        tt.base[g] = sfirst[g];
    }
    fence_proxy_async_smem();  // this thread's use of the ring, before the GEMM's copies land there
    return true;
}

// Shared-memory bytes the fused dispatch needs for its per-expert prefix of
// the router tiles' counts ([E][slots + 1] words, inside the ring).
constexpr size_t fused_dispatch_smem(int E, int slots) { return (size_t)E * (size_t)(slots + 1) * 4u; }

// kRoute: the instantiation that can route the tokens itself (p.fuse_route);
// the other one carries none of that code (fewer registers, a smaller body).
template <bool kRoute>
__global__ void __launch_bounds__(kThreads, 1) expert_gemm_tc_kernel(const TcParams p, const __grid_constant__ TcMaps maps)
{
    extern __shared__ uint8_t dsmem[];
    __shared__ TileTable tt;
    __shared__ __align__(8) uint64_t bars[2 * kStages + 5 + 2 * kTQ];
    __shared__ uint32_t s_tmem;
    __shared__ volatile int s_abort;
    __shared__ volatile int s_tq[kTQ];
    __shared__ volatile int s_pdl_done;  // thread 0 has passed griddepcontrol.wait

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t sbase = (smem_u32(dsmem) + 1023u) & ~1023u;
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (kStages + s); };
    auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * kStages + b); };
    auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * kStages + 2 + b); };
    const uint32_t done_bar = bar0 + 8u * (2 * kStages + 4);
    auto tq_full_bar = [&](int i) { return bar0 + 8u * (2 * kStages + 5 + i); };
    auto tq_empty_bar = [&](int i) { return bar0 + 8u * (2 * kStages + 5 + kTQ + i); };
    // Entry i of the CTA's tile sequence, for a consumer role (one thread):
    // -1 at the end of the list or after an abort.  In wave order every role
    // computes it; dynamically, warp 0 hands it out through the tile queue.
    // The list's tiles [0, tail) go out in waves (CTA c: c, c + grid, ...,
    // n_wave of them), the rest [tail, total) dynamically, through the queue.
    int total = 0, tail = 0, n_wave = 0;
    auto next_tile = [&](int i) -> int {
        if (i < n_wave) return s_abort ? -1 : (int)blockIdx.x + i * (int)gridDim.x;
        const int d = i - n_wave, slot = d % kTQ;
        if (!mbar_wait(tq_full_bar(slot), (uint32_t)(d / kTQ) & 1u, &s_abort, p.status)) return -1;
        const int t = s_tq[slot];
        mbar_arrive(tq_empty_bar(slot));
        return t;
    };

    const int G = p.E + (p.E_sh > 0 ? 1 : 0);
    // expert weights stream through L2 once (evict first); the hidden states,
    // activations and per-row outputs are read again by other tiles of this
    // launch (evict last)
    const uint64_t pol_stream = l2_policy_evict_first(), pol_keep = l2_policy_evict_last();
    if (warp == 0 && lane < 2) {  // the weight maps of this launch's GEMMs, ahead of their first loads
        const int ph = lane == 0 ? kGateUp : kDown;
        if (ph == kGateUp ? p.has_gu : p.has_down)
            for (int q = 0; q < (p.E_sh > 0 ? 3 : 2); ++q) {
                prefetch_tmap(&maps.b0[ph][q]);
                if (ph == kGateUp) prefetch_tmap(&maps.b1[ph][q]);
            }
    }
    pdl_trigger();

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) { mbar_init(full_bar(s), kFullArrivals); mbar_init(empty_bar(s), 1); }
        for (int b = 0; b < 2; ++b) { mbar_init(tfull_bar(b), 1); mbar_init(tempty_bar(b), 4); }
        mbar_init(done_bar, 1);
        for (int i = 0; i < kTQ; ++i) { mbar_init(tq_full_bar(i), 1); mbar_init(tq_empty_bar(i), kTQConsumers); }
        s_abort = 0;
        s_pdl_done = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(&s_tmem)),
                     "r"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::);
    }
    __syncthreads();  // s_pdl_done and s_abort are initialised
    // weights of the first wave into L2 while the routing is computed (in
    // this launch: after this CTA's router rows have landed, which the
    // prefetch would otherwise delay)
    if (warp == 2 && lane == 0 && (int)blockIdx.x < p.prefetch_tiles && !p.fuse_route) prefetch_first_wave(p);
    if (warp == 2 && lane == 0 && (int)blockIdx.x < p.prefetch_experts) {
        // the list starts with expert 0's tiles, then expert 1's, ...: the
        // first wave's weights, after the delay, or at once when the router
        // has already finished (thread 0 passed its wait; bounded spin)
        const unsigned long long t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < kPrefillPrefetchDelayNs && !s_pdl_done) {
        }
        const int e = (int)blockIdx.x;
        const int q = e < p.E_pub ? 0 : 1;
        const size_t row0 = (size_t)(q ? e - p.E_pub : e) * p.I;
        for (int r = 0; r < p.I; r += 128) {
            const uint32_t bytes = (uint32_t)min(128, p.I - r) * (uint32_t)p.H * 2u;
            bulk_prefetch_l2(p.gate_w[q] + (row0 + r) * p.H, bytes);
            bulk_prefetch_l2(p.up_w[q] + (row0 + r) * p.H, bytes);
        }
    }
    pdl_wait();  // the dispatch offsets and slot maps (or the route log, or cleared counters) come from the previous kernel
    if (tid == 0) s_pdl_done = 1;
    if (kRoute && p.fuse_route) {
        const bool ok = route_in_launch(p, dsmem + (sbase - smem_u32(dsmem)), tt, &s_abort);
        if (!ok && tid == 0) s_abort = 1;
        __syncthreads();
        if (tid == 0) grid_arrive(p.grid_bar);  // the roles wait for it (wait_dispatch)
    }
    if (p.fuse_dispatch) {
        // ---- the dispatch order, as dispatch_kernel derives it.  pre[e][s]:
        // rows of expert e in the router tiles before tile s (in the ring,
        // which no load has touched yet), its total = the expert's rows
        uint32_t *pre = reinterpret_cast<uint32_t *>(dsmem + (sbase - smem_u32(dsmem)));
        const int sp = p.slots + 1;
        for (int g = tid; g < p.E; g += kThreads) {
            const uint32_t *tc = p.tile_counts + (size_t)g * p.slots4;
            uint32_t acc = 0;
            int s2 = 0;
            for (; s2 + 4 <= p.slots; s2 += 4) {
                const uint4 v = *reinterpret_cast<const uint4 *>(tc + s2);  // slots4: rows 16-byte aligned
                pre[g * sp + s2] = acc; acc += v.x;
                pre[g * sp + s2 + 1] = acc; acc += v.y;
                pre[g * sp + s2 + 2] = acc; acc += v.z;
                pre[g * sp + s2 + 3] = acc; acc += v.w;
            }
            for (; s2 < p.slots; ++s2) { pre[g * sp + s2] = acc; acc += tc[s2]; }
            pre[g * sp + p.slots] = acc;
            tt.rows[g] = (int)acc;
        }
        __syncthreads();
        if (warp == 0) {  // exclusive prefix over the experts: their first slots
            int carry = 0;
            for (int b = 0; b < p.E; b += 32) {
                const int v0 = b + lane < p.E ? tt.rows[b + lane] : 0;
                int v = v0;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const int y = __shfl_up_sync(~0u, v, off);
                    if (lane >= off) v += y;
                }
                if (b + lane < p.E) tt.base[b + lane] = carry + v - v0;
                carry += __shfl_sync(~0u, v, 31);
            }
        }
        __syncthreads();
        if (blockIdx.x == 0) {
            for (int g = tid; g < p.E; g += kThreads) {
                p.offsets_w[g] = (uint32_t)tt.base[g];
                p.counts_w[g] = (uint32_t)tt.rows[g];
            }
            if (tid == 0) p.offsets_w[p.E] = (uint32_t)(tt.base[p.E - 1] + tt.rows[p.E - 1]);
            for (int i = tid; i < p.clear_words; i += kThreads) p.ready[i] = 0u;
        }
        // this CTA's share of the routed rows r = (t, j): slot = first slot of
        // its expert + the expert's rows in earlier router tiles + its
        // position in its tile (ticket = 128 * tile + position)
        for (int r = blockIdx.x * kThreads + tid; r < p.R; r += gridDim.x * kThreads) {
            const int e = p.topk_idx[r];
            if ((unsigned)e >= (unsigned)p.E) {  // never produced by the router
                if (p.status) atomicOr(p.status, PMPE_STATUS_BAD_EXPERT_ID);
                continue;
            }
            const int tk = p.ticket[r];
            const int ts = min(tk >> 7, p.slots);
            const int slot = tt.base[e] + (int)pre[e * sp + ts] + (tk & 127);
            if ((unsigned)slot >= (unsigned)p.R) continue;  // only a corrupt ticket could fail this
            p.slot_of_w[r] = slot;
            p.tok_of_slot_w[slot] = r / p.k;
            p.w_of_slot_w[slot] = p.w_route[r];
        }
        // arrive at the grid barrier (an arrival counter the router zeroed);
        // each role waits for every CTA's arrival (wait_dispatch) only before
        // it first reads what other CTAs wrote here, so that the tile table,
        // the first weight loads and the other CTAs' arrivals overlap
        __syncthreads();
        if (tid == 0) grid_arrive(p.grid_bar);
    }
    // Until every CTA has arrived: the slot maps (tok_of_slot, w_of_slot) and
    // the readiness and tile counters (cleared by CTA 0) are not yet final.
    // Every lane that calls this acquires the arrivals itself (bounded wait;
    // the grid is resident all at once, checked before the launch).
    auto wait_dispatch = [&]() -> bool {
        if (!p.fuse_dispatch && !p.fuse_route) return true;
        const unsigned long long t0 = globaltimer_ns();
        while (ld_acquire_gpu(p.grid_bar) < gridDim.x) {
            if (s_abort) return false;
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                s_abort = 1;
                if (p.status) atomicOr(p.status, PMPE_STATUS_PIPELINE_TIMEOUT);
                return false;
            }
            __nanosleep(32);
        }
        return true;
    };
    // tile list: rows and tiles per group, prefixes over groups
    int multi = 0;  // some group has more than one 128-row block
    for (int g = tid; g < G; g += kThreads) {
        const bool shared = g >= p.E;
        int rows, base;
        if (shared) {
            rows = p.T;
            base = 0;
        } else if (p.fuse_dispatch || p.fuse_route) {  // derived above
            rows = min(tt.rows[g], p.R);
            base = min(tt.base[g], p.R - rows);
        } else {  // clamped to [0, R): only a corrupt workspace could make this matter
            const int b = min((int)p.offsets[g], p.R), e = min(max((int)p.offsets[g + 1], b), p.R);
            rows = e - b;
            base = b;
        }
        const int mt = (rows + BM - 1) / BM;
        multi |= mt > 1 ? 1 : 0;
        tt.rows[g] = rows;
        tt.base[g] = base;
        tt.mpre[g + 1] = mt;
        tt.prefix[kGateUp][g + 1] = mt * (group_n(p, kGateUp, shared) / p.ph[kGateUp].bn);
        tt.prefix[kDown][down_place(p, g) + 1] = mt * (group_n(p, kDown, shared) / p.ph[kDown].bn);
    }
    // the same value in every thread of every CTA (all read the same offsets)
    multi = __syncthreads_or(multi);
    if (warp < 3) {  // three inclusive scans, one per warp: tiles of each GEMM, row blocks
        int *arr = warp == 2 ? tt.mpre : tt.prefix[warp];
        int carry = 0;
        for (int b = 0; b < G; b += 32) {
            int v = b + lane < G ? arr[b + lane + 1] : 0;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(~0u, v, off);
                if (lane >= off) v += y;
            }
            __syncwarp();
            if (b + lane < G) arr[b + lane + 1] = carry + v;
            carry += __shfl_sync(~0u, v, 31);
        }
        if (lane == 0) arr[0] = 0;
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = s_tmem;
    total = total_tiles(p, tt, G);
    // waves keep an expert's m-tiles (which share weights) running together;
    // the last kTailWaves waves, and every tile when no group has a second
    // 128-row block (nothing to share), go out dynamically, so that the CTAs
    // finish together
    tail = multi == 0 ? 0 : max(0, total - kTailWaves * (int)gridDim.x);
    n_wave = (int)blockIdx.x < tail ? (tail - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;

    if (warp == 0 && lane < kLoaders) {
        // ------------------------------------------------ TMA producers
        // Three lanes, one operand box each: a single thread's TMA boxes are
        // processed one after another, so spreading a stage's boxes over
        // three issuing threads triples the ring's fill rate.
        //   lane 0: the A tile (128 rows x 64 K) when A comes through TMA (the
        //           activations, or the hidden states of the shared group), and
        //           then also the arrivals of the gather warps, which have
        //           nothing to copy; in a routed gate/up tile the gather warps
        //           fill A and lane 0 only arrives
        //   lane 1: gate rows (gate/up) or B rows [0, bn/2) (down)
        //   lane 2: up rows (gate/up)   or B rows [bn/2, bn) (down)
        int stage = 0;
        uint32_t phase = 0;
        uint32_t filled = 0, last_parity = 0;  // per-stage bits, for the drain below
        // Lane 0 picks the tiles and hands each to the CTA's other roles
        // through the tile queue.  When a group has several 128-row blocks,
        // its m-tiles share weights: they sit next to each other in the list
        // and the CTAs take the list in waves (CTA c: tiles c, c + grid, ...),
        // so those m-tiles run at the same moment and one DRAM read of the
        // weights serves them all.  When no group has (decode), nothing is
        // shared, and the tiles go out dynamically, the next one to whichever
        // CTA is ready (an atomic counter, taken one tile ahead), which
        // evens out tiles of unequal cost.
        uint32_t ahead = 0u;  // lane 0: the next dynamic tile, taken one ahead
        bool synced = false;  // lane 0: wait_dispatch has returned
        for (int qi = 0;; ++qi) {
            int tile = -1;
            if (qi < n_wave) {
                tile = next_tile(qi);
            } else {
                if (lane == 0) {
                    const int d = qi - n_wave, slot = d % kTQ;
                    if (d == 0) {
                        if (!synced) synced = wait_dispatch();
                        ahead = synced ? (uint32_t)tail + atomicAdd(p.tile_ctr, 1u) : (uint32_t)total;
                    }
                    if (mbar_wait(tq_empty_bar(slot), ((uint32_t)(d / kTQ) & 1u) ^ 1u, &s_abort, p.status) &&
                        !s_abort && ahead < (uint32_t)total) {
                        tile = (int)ahead;
                        ahead = (uint32_t)tail + atomicAdd(p.tile_ctr, 1u);
                    }
                    s_tq[slot] = tile;
                    mbar_arrive(tq_full_bar(slot));
                }
                tile = __shfl_sync((1u << kLoaders) - 1u, tile, 0);
            }
            if (tile < 0) break;
            const Tile t = decode_tile(p, tt, G, tile);
            const bool gather = t.kind == kTileGU && !t.shared;
            const int q = t.shared ? 2 : (t.g < p.E_pub ? 0 : 1);
            const int ei = t.shared ? 0 : (q == 0 ? t.g : t.g - p.E_pub);
            const CUtensorMap *amap = t.shared ? &maps.a_shared[t.ph] : &maps.a_routed[t.ph];
            const int arow = t.row_base + t.m0;
            const uint32_t my_tx = lane == 0 ? (gather ? 0u : (uint32_t)kABytes)
                                             : (t.ph == kGateUp ? (uint32_t)(BM * 128) : (uint32_t)(t.bn / 2 * 128));
            bool ok = true;
            if (t.kind == kTileDown && p.has_gu && lane == 0) {
                // a down tile after the gate/up tiles of the same launch: its
                // activation rows are complete once every gate/up epilogue
                // warp of their row block has stored its part (bounded wait;
                // the weights are loaded meanwhile)
                const uint32_t need = 4u * (uint32_t)(group_n(p, kGateUp, t.shared) / p.ph[kGateUp].bn);
                const uint32_t *rp = p.ready + tt.mpre[t.g] + t.m_tile;
                if (!synced) synced = wait_dispatch();
                if (!synced) ok = false;
                const unsigned long long t0 = globaltimer_ns();
                while (ok && ld_acquire_gpu(rp) < need) {
                    if (s_abort) { ok = false; break; }
                    if (globaltimer_ns() - t0 > kWaitLimitNs) {
                        s_abort = 1;
                        if (p.status) atomicOr(p.status, PMPE_STATUS_PIPELINE_TIMEOUT);
                        ok = false;
                        break;
                    }
                    __nanosleep(128);
                }
                // the async proxy (TMA) reads what the generic acquire observed
                asm volatile("fence.proxy.async.global;\n" ::: "memory");
            }
            for (int kb = 0; kb < t.nkb && ok; ++kb) {
                if (!mbar_wait(empty_bar(stage), phase ^ 1u, &s_abort, p.status)) { ok = false; break; }
                const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
                mbar_expect_tx(full_bar(stage), my_tx);
                const int kx = kb * BK;
                if (lane == 0) {
                    if (!gather) {
                        tma_load_2d_hint(sA, amap, full_bar(stage), kx, arow, pol_keep);
                        mbar_arrive_count(full_bar(stage), kGatherThreads);
                    }
                } else if (t.ph == kGateUp) {
                    const int brow = ei * p.I + t.n0;  // shared: n0 spans E_sh * I rows
                    tma_load_2d_hint(sB + (lane - 1) * BM * 128, lane == 1 ? &maps.b0[t.ph][q] : &maps.b1[t.ph][q],
                                     full_bar(stage), kx, brow, pol_stream);
                } else {
                    const int half = (lane - 1) * (t.bn / 2);
                    if (t.shared) {
                        const int sidx = kx / p.I;
                        tma_load_2d_hint(sB + half * 128, &maps.b0[t.ph][2], full_bar(stage), kx - sidx * p.I,
                                         sidx * p.H + t.n0 + half, pol_stream);
                    } else {
                        tma_load_2d_hint(sB + half * 128, &maps.b0[t.ph][q], full_bar(stage), kx,
                                         ei * p.H + t.n0 + half, pol_stream);
                    }
                }
                filled |= 1u << stage;
                last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
                if (++stage == kStages) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
        }
        // drain: every copy this thread issued has landed before the CTA exits
        for (int s = 0; s < kStages; ++s)
            if ((filled >> s) & 1u) {
                const unsigned long long t0 = globaltimer_ns();
                while (!mbar_try_wait(full_bar(s), (last_parity >> s) & 1u))
                    if (globaltimer_ns() - t0 > kWaitLimitNs) break;
            }
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------ MMA issuer
        int stage = 0, it = 0;
        uint32_t phase = 0;
        for (int qi = 0;; ++qi) {
            const int tile = next_tile(qi);
            if (tile < 0) break;
            const Tile t = decode_tile(p, tt, G, tile);
            const uint32_t idesc = p.ph[t.ph].idesc;
            const int buf = it & 1;
            const uint32_t use = (uint32_t)(it >> 1) & 1u;
            ++it;
            if (!mbar_wait(tempty_bar(buf), use ^ 1u, &s_abort, p.status)) break;
            tc_fence_after();
            const uint32_t d_tmem = tmem_base + (uint32_t)(buf * kAccCols);
            bool ok = true;
            for (int kb = 0; kb < t.nkb; ++kb) {
                if (!mbar_wait(full_bar(stage), phase, &s_abort, p.status)) { ok = false; break; }
                tc_fence_after();
                // rows the gather warps copied (generic proxy, complete when
                // the barrier's phase completed) are read by the tensor cores
                // through the async proxy
                fence_proxy_async_smem();
                const uint32_t sA = sbase + stage * kStageBytes, sB = sA + kABytes;
                const uint64_t ad = sw128_desc(sA), bd = sw128_desc(sB);
#pragma unroll
                for (int k = 0; k < BK / 16; ++k)  // +32 bytes of K per step inside the swizzle row
                    tc_mma(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kb | k) != 0);
                tc_commit(empty_bar(stage));
                if (++stage == kStages) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
            tc_commit(tfull_bar(buf));
        }
        // every MMA this thread issued has completed before TMEM is freed
        tc_commit(done_bar);
        {
            const unsigned long long t0 = globaltimer_ns();
            while (!mbar_try_wait(done_bar, 0))
                if (globaltimer_ns() - t0 > kWaitLimitNs) break;
        }
    } else if (warp >= 2 && warp < 6) {
        // ------------------------------------------------ epilogue
        const int quarter = warp & 3;  // TMEM lanes this warp may access
        const uint32_t out_base = sbase + kStages * kStageBytes + (uint32_t)((warp - 2) * 2 * kOutBufBytes);
        int out_parity = 0;
        int it = 0;
        bool synced = false;  // wait_dispatch has returned (every lane acquires)
        for (int qi = 0;; ++qi) {
            int tile = 0;
            if (lane == 0) tile = next_tile(qi);
            tile = __shfl_sync(~0u, tile, 0);
            if (tile < 0) break;
            const Tile t = decode_tile(p, tt, G, tile);
            const int buf = it & 1;
            const uint32_t use = (uint32_t)(it >> 1) & 1u;
            ++it;
            // one lane waits, the warp follows: tcgen05.ld below is warp-collective
            int ok = 1;
            if (lane == 0) ok = mbar_wait(tfull_bar(buf), use, &s_abort, p.status) ? 1 : 0;
            ok = __shfl_sync(~0u, ok, 0);
            if (!ok) break;
            if (!synced && !(synced = wait_dispatch())) break;
            __syncwarp();
            tc_fence_after();
            const TcPhase &ph = p.ph[t.ph];
            const bool gu = t.kind == kTileGU;
            const int r = quarter * 32 + lane;  // tile row of this thread
            const bool valid = r < t.rows;
            const int grow = t.row_base + t.m0 + r;
            const uint32_t taddr = tmem_base + (uint32_t)(buf * kAccCols) + ((uint32_t)(quarter * 32) << 16);
            if (gu) {
                // Whole 32-row blocks go out through shared memory and TMA
                // stores; the block holding a tile's last rows is written row
                // by row so that it never touches the next expert's rows.
                const bool full_block = (t.rows - quarter * 32) >= 32;
                const int ldc = t.shared ? p.E_sh * p.I : p.I;
                bf16 *crow = (t.shared ? ph.C_shared : ph.C_routed) + (size_t)grow * ldc + t.n0;
                const CUtensorMap *cmap = t.shared ? &maps.c_shared[t.ph] : &maps.c_routed[t.ph];
#pragma unroll 1
                for (int c = 0; c < BM / 32; ++c) {
                    uint32_t pk[16];
                    float gv[32], uv[32];
                    tmem_ld32(taddr + c * 32, gv);
                    tmem_ld32(taddr + 128 + c * 32, uv);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 16; ++i)
                        pk[i] = pack_bf16x2(silu_mul(gv[2 * i], uv[2 * i]), silu_mul(gv[2 * i + 1], uv[2 * i + 1]));
                    if (p.saved_gu) {
                        // G and U of these 32 columns, as FP32, for the backward
                        const int y0 = t.row_base + t.m0 + quarter * 32;
                        const int ld2 = t.shared ? 2 * p.E_sh * p.I : 2 * p.I;  // floats per saved row
                        const int uoff = ld2 / 2;                                // U follows G
                        const CUtensorMap *smap = t.shared ? &maps.gu_save_sh : &maps.gu_save;
                        if (full_block) {
#pragma unroll
                            for (int b = 0; b < 4; ++b) {  // G lo, G hi, U lo, U hi: 16 columns each
                                const float *src = (b < 2 ? gv : uv) + (b & 1) * 16;
                                const uint32_t sbuf = out_base + (uint32_t)(out_parity * kOutBufBytes);
                                if (lane == 0) bulk_wait_read<1>();
                                __syncwarp();
#pragma unroll
                                for (int j = 0; j < 4; ++j) {
                                    const uint32_t addr = sbuf + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4);
                                    asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr),
                                                 "f"(src[4 * j]), "f"(src[4 * j + 1]), "f"(src[4 * j + 2]),
                                                 "f"(src[4 * j + 3])
                                                 : "memory");
                                }
                                fence_proxy_async_smem();
                                __syncwarp();
                                if (lane == 0) {
                                    tma_store_2d(smap, sbuf, (b < 2 ? 0 : uoff) + t.n0 + c * 32 + (b & 1) * 16, y0);
                                    bulk_commit();
                                }
                                out_parity ^= 1;
                            }
                        } else if (valid) {
                            float *sbase = t.shared ? p.saved_gu + (size_t)p.R * 2 * p.I : p.saved_gu;
                            float4 *gd = reinterpret_cast<float4 *>(sbase + (size_t)grow * ld2 + t.n0 + c * 32);
                            float4 *ud = gd + uoff / 4;
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                gd[i] = make_float4(gv[4 * i], gv[4 * i + 1], gv[4 * i + 2], gv[4 * i + 3]);
                                ud[i] = make_float4(uv[4 * i], uv[4 * i + 1], uv[4 * i + 2], uv[4 * i + 3]);
                            }
                        }
                    }
                    if (full_block) {
                        const uint32_t sbuf = out_base + (uint32_t)(out_parity * kOutBufBytes);
                        if (lane == 0) bulk_wait_read<1>();  // the store that used this buffer has read it
                        __syncwarp();
                        // 64-byte rows, 16-byte chunk j of row r at chunk j ^ ((r >> 1) & 3): the
                        // TMA 64-byte swizzle, and conflict-free for these 16-byte writes
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const uint32_t addr = sbuf + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4);
                            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(pk[4 * j]),
                                         "r"(pk[4 * j + 1]), "r"(pk[4 * j + 2]), "r"(pk[4 * j + 3])
                                         : "memory");
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d_hint(cmap, sbuf, t.n0 + c * 32, t.row_base + t.m0 + quarter * 32, pol_keep);
                            bulk_commit();
                        }
                        out_parity ^= 1;
                    } else if (valid) {
                        uint4 *dst = reinterpret_cast<uint4 *>(crow + c * 32);
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
                    }
                }
            } else {
                // ---- down: y = w * (act W_down^T), BF16, one row per thread;
                // whole 32-row blocks through shared memory and TMA stores, a
                // tile's last partial block row by row
                const bool full_block = (t.rows - quarter * 32) >= 32;
                bf16 *crow = (t.shared ? ph.C_shared : ph.C_routed) + (size_t)grow * p.H + t.n0;
                const CUtensorMap *cmap = t.shared ? &maps.c_shared[t.ph] : &maps.c_routed[t.ph];
                const float sc = t.shared ? 1.f : (valid ? p.w_of_slot[grow] : 0.f);
#pragma unroll 1
                for (int c = 0; c < t.bn / 32; ++c) {
                    uint32_t pk[16];
                    float v[32];
                    tmem_ld32(taddr + c * 32, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 16; ++i) pk[i] = pack_bf16x2(v[2 * i] * sc, v[2 * i + 1] * sc);
                    if (full_block) {
                        const uint32_t sbuf = out_base + (uint32_t)(out_parity * kOutBufBytes);
                        if (lane == 0) bulk_wait_read<1>();  // the store that used this buffer has read it
                        __syncwarp();
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const uint32_t addr = sbuf + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4);
                            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(pk[4 * j]),
                                         "r"(pk[4 * j + 1]), "r"(pk[4 * j + 2]), "r"(pk[4 * j + 3])
                                         : "memory");
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(cmap, sbuf, t.n0 + c * 32, t.row_base + t.m0 + quarter * 32);
                            bulk_commit();
                        }
                        out_parity ^= 1;
                    } else if (valid) {
                        uint4 *dst = reinterpret_cast<uint4 *>(crow + c * 32);
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty_bar(buf));
            // execution audit: rows this tile processed, counted where they
            // ran.  A row counts for its expert only if its token's route
            // names this expert (the route log is read back and checked, row
            // by row); a row that fails the check is a dispatch mismatch.
            // The per-token private count follows the rows physically run.
            if (gu) {
                const unsigned vm = __ballot_sync(~0u, valid);
                if (!t.shared && t.n0 == 0) {
                    const int tok = valid ? p.tok_of_slot[grow] : -1;
                    bool routed = false;
                    if ((unsigned)tok < (unsigned)p.T) {
                        const int32_t *ti = p.topk_idx + (size_t)tok * p.k;
                        for (int j = 0; j < p.k; ++j) routed |= ti[j] == t.g;
                    }
                    if (valid && !routed && p.status) atomicOr(p.status, PMPE_STATUS_DISPATCH_MISMATCH);
                    const unsigned ok_rows = __ballot_sync(~0u, valid && routed);
                    if (lane == 0 && p.exec_rows && ok_rows) atomicAdd(&p.exec_rows[t.g], (unsigned)__popc(ok_rows));
                    if (lane == 0 && quarter == 0 && p.exec_tiles) atomicAdd(&p.exec_tiles[t.g], 1u);
                    if ((unsigned)tok < (unsigned)p.T && t.g >= p.E_pub && p.exec_priv_rows)
                        atomicAdd(&p.exec_priv_rows[tok], 1u);
                }
                if (t.shared && p.shared_rows && lane == 0 && vm && (t.n0 % p.I) == 0)
                    atomicAdd(p.shared_rows, (unsigned)__popc(vm));
            }
            if (gu && p.has_down) {
                // release this warp's activation rows to the down tiles that
                // read them: the row stores (generic) and the TMA stores (async
                // proxy, complete after wait_group 0) are ordered before the count
                __threadfence();
                __syncwarp();
                if (lane == 0) {
                    bulk_wait_all();
                    asm volatile("fence.proxy.async.global;\n" ::: "memory");
                    __threadfence();
                    atomicAdd(p.ready + tt.mpre[t.g] + t.m_tile, 1u);
                }
                __syncwarp();
            }
        }
        if (lane == 0) bulk_wait_all();  // this warp's TMA stores are complete before the CTA exits
    } else if (warp >= 6) {
        // ------------------------------------------------ A-row gather
        // Gather: thread i of the 128 copies 16-byte chunk (i & 7) of tile rows
        // (i >> 3) + 16 j, j = 0..7, every stage, into the 128-byte-swizzled A
        // slot of the stage (chunk c of row r at chunk c ^ (r & 7)); a warp
        // instruction covers four whole 128-byte rows.  Rows past the tile's
        // rows are zero-filled.  Each thread's copies of a stage arrive on the
        // stage's full barrier when they complete (cp.async.mbarrier.arrive),
        // so the threads never wait for their own copies: up to the whole ring
        // is in flight.  The MMA thread fences the async proxy after the
        // barrier before the tensor cores read the rows.
        const int gi = tid - 192;            // 0 .. 127
        const int chunk = gi & 7, row0 = gi >> 3;
        uint32_t sc = 0;                     // ring stages passed so far (the ring position)
        bool ok = true;
        bool synced = false;                 // wait_dispatch has returned (every lane acquires)
        auto drain = [&]() { cp_async_wait<0>(); };
        for (int qi = 0; ok; ++qi) {
            int tile = 0;
            if (lane == 0) tile = next_tile(qi);
            tile = __shfl_sync(~0u, tile, 0);
            if (tile < 0) break;
            const Tile t = decode_tile(p, tt, G, tile);
            if (t.kind != kTileGU || t.shared) {  // A comes through TMA: only follow the ring
                sc += (uint32_t)t.nkb;
                continue;
            }
            if (!synced && !(synced = wait_dispatch())) break;
            // this thread's 8 rows: their token rows in the hidden states
            const bf16 *src[8];
            uint32_t nbytes[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int r = row0 + 16 * j;
                const int tok = r < t.rows ? p.tok_of_slot[t.row_base + t.m0 + r] : -1;
                const bool in = (unsigned)tok < (unsigned)p.T;
                src[j] = p.hidden + (in ? (size_t)tok * p.H : 0) + chunk * 8;
                nbytes[j] = in ? 16u : 0u;
            }
            for (int kb = 0; kb < t.nkb; ++kb, ++sc) {
                const int stage = (int)(sc % kStages);
                const uint32_t phase = (sc / kStages) & 1u;
                int free_ = 1;
                if (lane == 0) free_ = mbar_wait(empty_bar(stage), phase ^ 1u, &s_abort, p.status) ? 1 : 0;
                free_ = __shfl_sync(~0u, free_, 0);
                if (!free_) { ok = false; break; }
                const uint32_t sA = sbase + stage * kStageBytes;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int r = row0 + 16 * j;
                    cp_async16_zfill(sA + r * 128 + ((chunk ^ (r & 7)) << 4), src[j] + kb * BK, nbytes[j], pol_keep);
                }
                cp_async_arrive_noinc(full_bar(stage));
            }
        }
        drain();
    }

    // every warp reconverges before the block barrier: __syncthreads is a
    // warp-aligned barrier, and the single-thread roles above diverge from
    // their warps; TMEM is freed only after all epilogue reads completed
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(kTmemCols));
    }
    if (kRoute && p.fuse_combine) {
        // ---- the weighted combine (Sec. 3.1), as combine_kernel sums it:
        // j ascending, then the shared experts, in FP32.  Every epilogue
        // warp's stores are complete (wait_group 0 above); they are made
        // visible, then every CTA meets at the last grid barrier.
        if (warp >= 2 && warp < 6 && lane == 0) {
            asm volatile("fence.proxy.async.global;\n" ::: "memory");
            __threadfence();
        }
        if (grid_barrier(p.bar_d, gridDim.x, &s_abort, p.status)) {
            const bf16 *y = p.ph[kDown].C_routed;
            const bf16 *y_sh = p.E_sh > 0 ? p.ph[kDown].C_shared : nullptr;
            const int nv = p.H / 8;
            for (int t = (int)blockIdx.x; t < p.T; t += (int)gridDim.x) {
                for (int c = tid; c < nv; c += kThreads) {
                    float acc[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
                    for (int j = 0; j < p.k; ++j) {
                        int slot = p.slot_of_w[(size_t)t * p.k + j];
                        if ((unsigned)slot >= (unsigned)p.R) slot = 0;  // only after a dispatch mismatch (status set)
                        const uint4 v = *reinterpret_cast<const uint4 *>(y + (size_t)slot * p.H + (size_t)c * 8);
                        const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float2 f = __bfloat1622float2(b[q]);
                            acc[2 * q] += f.x;
                            acc[2 * q + 1] += f.y;
                        }
                    }
                    if (y_sh) {
                        const uint4 v = *reinterpret_cast<const uint4 *>(y_sh + (size_t)t * p.H + (size_t)c * 8);
                        const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float2 f = __bfloat1622float2(b[q]);
                            acc[2 * q] += f.x;
                            acc[2 * q + 1] += f.y;
                        }
                    }
                    uint4 o;
                    o.x = pack_bf16x2(acc[0], acc[1]);
                    o.y = pack_bf16x2(acc[2], acc[3]);
                    o.z = pack_bf16x2(acc[4], acc[5]);
                    o.w = pack_bf16x2(acc[6], acc[7]);
                    reinterpret_cast<uint4 *>(p.out + (size_t)t * p.H)[c] = o;
                }
            }
        }
    }
}

// ------------------------------------------------------------ host side

// Parameters and tensor maps of one GEMM (`mode`) of a launch.
bool fill_phase(const Ctx &c, int mode, TcParams &p, TcMaps &maps)
{
    const Shape &s = c.s;
    const uint64_t R = (uint64_t)s.T * s.k, T = (uint64_t)s.T;
    bool ok = true;
    if (mode == kGateUp) {
        TcPhase &f = p.ph[mode];
        f.C_routed = c.act;
        f.C_shared = c.act_sh;
        ok &= encode_2d_box(&maps.c_routed[mode], c.act, s.I, R, kOutBox, kOutBox, CU_TENSOR_MAP_SWIZZLE_64B);
        if (s.E_sh > 0)
            ok &= encode_2d_box(&maps.c_shared[mode], c.act_sh, (uint64_t)s.E_sh * s.I, T, kOutBox, kOutBox,
                                CU_TENSOR_MAP_SWIZZLE_64B);
        for (int q = 0; q < 2; ++q) {
            const uint64_t n = (uint64_t)(q ? s.E_priv : s.E_pub) * s.I;
            ok &= encode_2d(&maps.b0[mode][q], c.gate[q], s.H, n, 128);
            ok &= encode_2d(&maps.b1[mode][q], c.up[q], s.H, n, 128);
        }
        if (s.E_sh > 0) {
            ok &= encode_2d(&maps.a_shared[mode], c.hidden, s.H, T, BM);
            ok &= encode_2d(&maps.b0[mode][2], c.gate[2], s.H, (uint64_t)s.E_sh * s.I, 128);
            ok &= encode_2d(&maps.b1[mode][2], c.up[2], s.H, (uint64_t)s.E_sh * s.I, 128);
        }
    } else {
        const int bn = p.ph[mode].bn;
        TcPhase &f = p.ph[mode];
        f.C_routed = c.y;
        f.C_shared = c.y_sh;
        ok &= encode_2d_box(&maps.c_routed[mode], c.y, s.H, R, kOutBox, kOutBox, CU_TENSOR_MAP_SWIZZLE_64B);
        if (s.E_sh > 0)
            ok &= encode_2d_box(&maps.c_shared[mode], c.y_sh, s.H, T, kOutBox, kOutBox, CU_TENSOR_MAP_SWIZZLE_64B);
        ok &= encode_2d(&maps.a_routed[mode], c.act, s.I, R, BM);
        for (int q = 0; q < 2; ++q) {
            const uint64_t n = (uint64_t)(q ? s.E_priv : s.E_pub) * s.H;
            ok &= encode_2d(&maps.b0[mode][q], c.down[q], s.I, n, bn / 2);
        }
        if (s.E_sh > 0) {
            ok &= encode_2d(&maps.a_shared[mode], c.act_sh, (uint64_t)s.E_sh * s.I, T, BM);
            ok &= encode_2d(&maps.b0[mode][2], c.down[2], s.I, (uint64_t)s.E_sh * s.H, bn / 2);
        }
    }
    return ok;
}

// The dynamic shared-memory limit of one instantiation, raised once per device.
template <bool kRoute>
cudaError_t ensure_tc_smem()
{
    static std::atomic<int> smem_limit[64];
    return ensure_dynamic_smem(expert_gemm_tc_kernel<kRoute>, kDynSmem, smem_limit);
}

// One persistent launch of the gate/up tiles, the down tiles, or both (and,
// with fuse_dispatch, the dispatch before them).
cudaError_t launch_tc(const Ctx &c, bool gu, bool down, bool fuse_dispatch = false, bool fuse_route = false,
                      bool fuse_combine = false)
{
    const Shape &s = c.s;
    TcParams p;
    TcMaps maps;
    memset(&p, 0, sizeof(p));
    memset(&maps, 0, sizeof(maps));
    p.has_gu = gu;
    p.has_down = down;
    p.E = s.E(); p.E_pub = s.E_pub; p.E_sh = s.E_sh; p.T = s.T; p.H = s.H; p.I = s.I; p.R = s.T * s.k; p.k = s.k;
    p.ph[kGateUp].bn = 128;
    p.ph[kGateUp].idesc = make_idesc(BM, 256);
    p.ph[kDown].bn = column_block(s.H);
    p.ph[kDown].idesc = make_idesc(BM, p.ph[kDown].bn);
    p.offsets = c.offsets;
    p.w_of_slot = c.w_of_slot;
    p.tok_of_slot = c.tok_of_slot;
    p.topk_idx = c.idx;
    p.hidden = c.hidden;
    p.ready = c.gemm_ready;
    if (gu && s.T <= BM && s.I % 128 == 0 && (long long)s.H * s.I >= (1ll << 20)) {
        // at most T rows per expert: no expert has a second 128-row block
        // (small experts, as in the tiny layer: the launch is too short to
        // gain from it)
        p.prefetch_tiles = std::min(s.E() * (s.I / 128), kPrefetchTiles);
        for (int q = 0; q < 2; ++q) {
            p.gate_w[q] = c.gate[q];
            p.up_w[q] = c.up[q];
        }
    }
    p.tile_ctr = c.gemm_ready + gemm_ready_words(s) - 2;
    p.exec_rows = c.audit.exec_rows;
    p.exec_tiles = c.audit.exec_tiles;
    p.exec_priv_rows = c.audit.exec_priv_rows;
    p.shared_rows = c.audit.shared_rows;
    p.status = c.audit.status;
    if (fuse_dispatch) {
        p.fuse_dispatch = 1;
        const size_t gu_bytes = (size_t)2 * s.I * s.H * 2;  // one expert's gate and up rows
        p.prefetch_experts = (int)std::min<size_t>(std::min<size_t>(kPrefillPrefetchBytes / gu_bytes,
                                                                    (size_t)kPrefillPrefetchExperts),
                                                   (size_t)s.E());
        for (int q = 0; q < 2; ++q) {
            p.gate_w[q] = c.gate[q];
            p.up_w[q] = c.up[q];
        }
        p.ticket = c.ticket;
        p.w_route = c.w;
        p.tile_counts = c.tile_counts;
        p.slots = router_slots(s.T);
        p.slots4 = router_slots4(s.T);
        p.counts_w = c.counts;
        p.offsets_w = c.offsets;
        p.slot_of_w = c.slot_of;
        p.tok_of_slot_w = c.tok_of_slot;
        p.w_of_slot_w = c.w_of_slot;
        p.grid_bar = c.gemm_ready + gemm_ready_words(s) - 1;
        p.clear_words = (int)gemm_ready_words(s) - 1;
    }
    if (fuse_route) {  // every counter cleared by clear_counters_kernel before this launch
        p.fuse_route = 1;
        p.renorm = s.renorm;
        p.policy = c.policy;
        p.router_w[0] = c.router_pub;
        p.router_w[1] = c.router_priv;
        p.z = reinterpret_cast<float *>(c.router_rows);  // the chunked router's scratch, unused here
        p.zpitch = std::max(s.E_pub, s.E_priv);
        p.idx_w = c.idx;
        p.ticket_w = c.ticket;
        p.w_w = c.w;
        p.tau_w = c.tau;
        p.tile_counts_w = c.tile_counts;
        p.route_count = c.audit.route_count;
        p.route_priv_rows = c.audit.route_priv_rows;
        p.slots = router_slots(s.T);
        p.slots4 = router_slots4(s.T);
        p.counts_w = c.counts;
        p.offsets_w = c.offsets;
        p.slot_of_w = c.slot_of;
        p.tok_of_slot_w = c.tok_of_slot;
        p.w_of_slot_w = c.w_of_slot;
        p.bar_a = c.gemm_ready + gemm_ready_words(s) - 4;
        p.bar_b = c.gemm_ready + gemm_ready_words(s) - 3;
        p.grid_bar = c.gemm_ready + gemm_ready_words(s) - 1;
        if (fuse_combine) {
            p.fuse_combine = 1;
            p.bar_d = c.gemm_ready + gemm_ready_words(s) - 5;
            p.out = c.out;
        }
    }
    bool ok = true;
    if (gu) ok &= fill_phase(c, kGateUp, p, maps);
    if (down) ok &= fill_phase(c, kDown, p, maps);
    if (c.saved_gu && gu) {
        p.saved_gu = c.saved_gu;
        ok &= encode_2d_f32(&maps.gu_save, c.saved_gu, 2 * (uint64_t)s.I, (uint64_t)s.T * s.k, 16, 32,
                            CU_TENSOR_MAP_SWIZZLE_64B);
        if (s.E_sh > 0)
            ok &= encode_2d_f32(&maps.gu_save_sh, c.saved_gu + (size_t)s.T * s.k * 2 * s.I,
                                2 * (uint64_t)s.E_sh * s.I, (uint64_t)s.T, 16, 32, CU_TENSOR_MAP_SWIZZLE_64B);
    }
    if (!ok) return cudaErrorInvalidValue;
    const cudaError_t err = fuse_route ? ensure_tc_smem<true>() : ensure_tc_smem<false>();
    if (err != cudaSuccess) return err;
    if (fuse_route)
        return launch_pdl(expert_gemm_tc_kernel<true>, dim3(c.num_sms), dim3(kThreads), kDynSmem, c.stream, p, maps);
    return launch_pdl(expert_gemm_tc_kernel<false>, dim3(c.num_sms), dim3(kThreads), kDynSmem, c.stream, p, maps);
}

// Whether the persistent grid (one CTA per SM) can be resident all at once:
// the down tiles of the gate/up + down launch wait for gate/up tiles that
// other CTAs own, so every CTA must run concurrently.  Cached per device.
static bool grid_fits(const Ctx &c)
{
    static std::atomic<int> fits[64];  // 0 unknown, 1 yes, 2 no
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (dev >= 0 && dev < 64 && fits[dev].load() != 0) return fits[dev].load() == 1;
    int per_sm = 0, per_sm_r = 0;
    const bool ok = ensure_tc_smem<false>() == cudaSuccess && ensure_tc_smem<true>() == cudaSuccess &&
                    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, expert_gemm_tc_kernel<false>, kThreads,
                                                                  kDynSmem) == cudaSuccess &&
                    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_r, expert_gemm_tc_kernel<true>, kThreads,
                                                                  kDynSmem) == cudaSuccess &&
                    per_sm >= 1 && per_sm_r >= 1;
    if (dev >= 0 && dev < 64) fits[dev].store(ok ? 1 : 2);
    return ok;
}

}  // namespace

// The two GEMMs in separate launches (diagnostics, and the fallback when the
// persistent grid cannot be resident at once): each starts from tile 0.
cudaError_t launch_gateup(const Ctx &c)
{
    const cudaError_t err = cudaMemsetAsync(c.gemm_ready + gemm_ready_words(c.s) - 2, 0, sizeof(uint32_t), c.stream);
    return err == cudaSuccess ? launch_tc(c, true, false) : err;
}

cudaError_t launch_down(const Ctx &c)
{
    const cudaError_t err = cudaMemsetAsync(c.gemm_ready + gemm_ready_words(c.s) - 2, 0, sizeof(uint32_t), c.stream);
    return err == cudaSuccess ? launch_tc(c, false, true) : err;
}

// The dispatch can run inside the persistent launch when that launch's grid
// is resident at once (its grid barrier) and the prefix table of the router
// tiles' counts fits its ring.  For small experts (fewer than 2^20 weights a
// projection: the tiny test layer) the launch is short and the grid barrier
// costs more than the dispatch kernel it saves (40.1 vs 38.2 us a step).
bool experts_fuse_dispatch(const Ctx &c)
{
    return (long long)c.s.H * c.s.I >= (1ll << 20) && grid_fits(c) &&
           fused_dispatch_smem(c.s.E(), router_slots(c.s.T)) <= (size_t)(kStages * kStageBytes);
}

// Routing in the expert launch: at most 128 tokens (one selection CTA each,
// all resident with the persistent grid), the masked router of the method
// (not the unmasked control), pools of at most 256 experts (8 logits a lane
// in the selection), H <= 2048 (a lane holds at most 8 16-byte pieces of a
// row in registers for the logits), and the dispatch's per-expert masks fit
// the ring.
bool experts_fuse_route(const Ctx &c)
{
    const Shape &s = c.s;
    return s.T >= 1 && s.T <= kRouteMaxTokens && s.T <= c.num_sms && !c.unmasked && s.H <= kRouteMaxH &&
           s.E_pub <= 256 && s.E_priv <= 256 && (size_t)s.E() * 24u <= (size_t)(kStages * kStageBytes) &&
           grid_fits(c);
}

__global__ void clear_counters_kernel(uint32_t *w, int n)
{
    pdl_trigger();
    pdl_wait();  // the previous forward on this workspace has finished with them
    for (int i = threadIdx.x; i < n; i += blockDim.x) w[i] = 0u;
}

// The forward's launches when the expert launch routes: the counters
// (readiness, tile, barriers) cleared by a one-block kernel, then the
// persistent launch (routing, dispatch order, gate/up and down).
cudaError_t launch_experts_routed(const Ctx &c, bool combine)
{
    const cudaError_t err =
        launch_pdl(clear_counters_kernel, dim3(1), dim3(256), 0, c.stream, c.gemm_ready, (int)gemm_ready_words(c.s));
    return err == cudaSuccess ? launch_tc(c, true, true, false, true, combine) : err;
}

cudaError_t launch_experts(const Ctx &c, bool zero_ready, bool fuse_dispatch)
{
    if (!grid_fits(c)) {  // the two GEMMs one after the other: no cross-CTA wait
        const cudaError_t err = launch_gateup(c);
        return err == cudaSuccess ? launch_down(c) : err;
    }
    if (zero_ready && !fuse_dispatch) {
        const cudaError_t err = cudaMemsetAsync(c.gemm_ready, 0, sizeof(uint32_t) * gemm_ready_words(c.s), c.stream);
        if (err != cudaSuccess) return err;
    }
    return launch_tc(c, true, true, fuse_dispatch);
}

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    return fn;
}

// 2-D tensor map over a row-major [rows, cols] matrix of `type` elements of
// `elem_bytes` bytes, box = box_cols x box_rows, zero fill out of bounds.
static bool encode_2d_typed(CUtensorMap *m, CUtensorMapDataType type, uint32_t elem_bytes, const void *ptr,
                            uint64_t cols, uint64_t rows, uint32_t box_cols, uint32_t box_rows,
                            CUtensorMapSwizzle swizzle)
{
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * elem_bytes};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, type, 2, const_cast<void *>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_3d_blocks(CUtensorMap *m, const void *ptr, uint64_t cols, uint64_t rows, uint32_t box_rows, uint32_t nblocks)
{
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[3] = {64, rows, cols / 64};
    const cuuint64_t strides[2] = {cols * 2, 128};  // row pitch; 64-column blocks 128 bytes apart
    const cuuint32_t box[3] = {64, box_rows, nblocks};
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_2d_box(CUtensorMap *m, const void *ptr, uint64_t cols, uint64_t rows, uint32_t box_cols,
                   uint32_t box_rows, CUtensorMapSwizzle swizzle)
{
    return encode_2d_typed(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, ptr, cols, rows, box_cols, box_rows, swizzle);
}

bool encode_2d_f32(CUtensorMap *m, const void *ptr, uint64_t cols, uint64_t rows, uint32_t box_cols,
                   uint32_t box_rows, CUtensorMapSwizzle swizzle)
{
    return encode_2d_typed(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, ptr, cols, rows, box_cols, box_rows, swizzle);
}

bool encode_2d(CUtensorMap *m, const void *ptr, uint64_t cols, uint64_t rows, uint32_t box_rows)
{
    return encode_2d_box(m, ptr, cols, rows, 64u, box_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}

uint32_t make_idesc(int M, int N)
{
    return (1u << 4)                    // D: FP32
           | (1u << 7)                  // A: BF16
           | (1u << 10)                 // B: BF16
           | ((uint32_t)(N >> 3) << 17) // N / 8
           | ((uint32_t)(M >> 4) << 24);// M / 16   (A and B K-major: transpose bits 15, 16 = 0)
}

uint32_t make_idesc_major(int M, int N, bool a_mn_major, bool b_mn_major)
{
    return make_idesc(M, N) | ((a_mn_major ? 1u : 0u) << 15) | ((b_mn_major ? 1u : 0u) << 16);
}


}  // namespace pmpe
