// Stages 2 and 5 of the layer: the dispatch order of the routed rows, and
// the weighted unpermute-combine.
//
// Dispatch (the grouping any grouped expert execution needs): the routed rows
// are grouped by expert id -- expert e owns slots [offset[e], offset[e+1]) --
// and, inside an expert, ordered by token: the router's ticket names the
// row's 128-token tile and its position among that tile's rows of its
// expert, and the rows of the earlier tiles (tile_counts) come first.  The
// tiles of a pool run in ascending token order, so every run gives the same
// order: the stable (t, j) order.  Only the slot maps are written (slot_of,
// tok_of_slot, w_of_slot): the expert kernel gathers each slot's token row
// from the hidden states itself.  An id outside [0, E) is recorded in the
// status word.  The backward, which reads the dispatched rows as one matrix,
// fills it with gather_dispatch_rows_kernel.
//
// Combine: out_t = bf16( sum_{j < k} y[slot(t, j)] + y_shared[t] ), summed in
// FP32 in a fixed order (j ascending, then shared), so the result of a token
// never depends on the other tokens of the batch.
#include <algorithm>

#include "pmpe_internal.cuh"
#include "tc_ptx.cuh"

namespace pmpe {
namespace {

constexpr int kDispThreads = 256;

struct DispatchParams {
    const int32_t *idx;
    const int32_t *ticket;
    const float *w;
    uint32_t *counts;             // [E] written: the rows of each expert
    const uint32_t *tile_counts;  // [E][slots4] rows of each expert per router tile
    int slots, slots4;            // router tile slots, and the row pitch of tile_counts
    int T, R, k, E;
    uint32_t *gemm_ready;         // the expert kernel's readiness counters, cleared here
    int gemm_ready_words;
    uint32_t *offsets;
    int32_t *slot_of, *tok_of_slot;
    float *w_of_slot;
    uint32_t *status;
};

// Slot of routed row r = (t, j): offset[e] + the rows of expert e in the
// router tiles before the row's tile + its position in that tile (ticket =
// 128 * tile + position).  Summing the earlier tiles' counts per row measured
// faster than building their prefix once, in the router's last CTA or in
// every dispatch CTA's shared memory.  Records the row in slot_of,
// tok_of_slot and w_of_slot (nothing for an id outside [0, E) or a slot
// outside [0, R)).
__device__ __forceinline__ void resolve_slot(const DispatchParams &p, const uint32_t *s_off, int r)
{
    const int t = r / p.k;
    const int e = p.idx[r];
    if ((unsigned)e >= (unsigned)p.E) {  // never produced by the router
        if (p.status) atomicOr(p.status, PMPE_STATUS_BAD_EXPERT_ID);
        return;
    }
    const int tk = p.ticket[r];
    const int ts = min(tk >> 7, p.slots4 - 1);
    const uint32_t *tc = p.tile_counts + (size_t)e * p.slots4;
    uint32_t before = 0;
    for (int s2 = 0; s2 < ts; ++s2) before += __ldg(tc + s2);
    const int slot = (int)(s_off[e] + before) + (tk & 127);
    if ((unsigned)slot >= (unsigned)p.R) return;  // only a corrupt ticket could fail this
    p.slot_of[r] = slot;
    p.tok_of_slot[slot] = t;
    p.w_of_slot[slot] = p.w[r];
}

// The dispatch order.  Every CTA forms the experts' row counts (the column
// sums of tile_counts) and offsets (their exclusive prefix sum) in shared
// memory; CTA 0 also writes both out and clears the expert kernel's
// readiness counters, which that kernel reads after this one; routed row
// r = (t, j) of expert e, in tile s at position q of the tile's rows of e,
// goes to slot offset[e] + sum_{s' < s} tile_counts[e][s'] + q.  One thread
// per routed row.
__global__ void __launch_bounds__(kDispThreads) dispatch_kernel(const DispatchParams p)
{
    __shared__ uint32_t s_off[2 * kMaxPool + 1];
    __shared__ uint32_t s_cnt[2 * kMaxPool];
    pdl_trigger();
    pdl_wait();
    // the rows of each expert: its column sums of tile_counts (every slot's
    // column is written by the router, zeros included)
    for (int e = threadIdx.x; e < p.E; e += kDispThreads) {
        const uint32_t *tc = p.tile_counts + (size_t)e * p.slots4;
        uint32_t tot = 0;
        for (int s2 = 0; s2 < p.slots; ++s2) tot += __ldg(tc + s2);
        s_cnt[e] = tot;
    }
    __syncthreads();
    if (threadIdx.x < 32) {
        uint32_t carry = 0;
        const int lane = threadIdx.x;
        for (int b = 0; b < p.E; b += 32) {
            uint32_t v = b + lane < p.E ? s_cnt[b + lane] : 0u;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const uint32_t y = __shfl_up_sync(~0u, v, off);
                if (lane >= off) v += y;
            }
            if (b + lane < p.E) s_off[b + lane + 1] = carry + v;
            carry += __shfl_sync(~0u, v, 31);
        }
        if (lane == 0) s_off[0] = 0;
    }
    __syncthreads();
    if (blockIdx.x == 0) {
        for (int e = threadIdx.x; e <= p.E; e += kDispThreads) p.offsets[e] = s_off[e];
        for (int e = threadIdx.x; e < p.E; e += kDispThreads) p.counts[e] = s_cnt[e];
        for (int i = threadIdx.x; i < p.gemm_ready_words; i += kDispThreads) p.gemm_ready[i] = 0u;
    }
    for (int r = blockIdx.x * kDispThreads + threadIdx.x; r < p.R; r += gridDim.x * kDispThreads)
        resolve_slot(p, s_off, r);
}

// The token rows of the dispatch slots [offsets[g0], offsets[g1]) copied into
// rows[slot] (the dispatched-row matrix the backward's GEMMs read): one warp
// per slot, eight 16-byte loads in flight per lane.
__global__ void __launch_bounds__(256) gather_dispatch_rows_kernel(const bf16 *hidden, const int32_t *tok_of_slot,
                                                                    const uint32_t *offsets, int g0, int g1, int R,
                                                                    int T, int H, bf16 *rows)
{
    const uint32_t p0 = min(offsets[g0], (uint32_t)R), p1 = min(max(offsets[g1], p0), (uint32_t)R);
    const int nv = H / 8;
    const int lane = threadIdx.x & 31;
    const int warps = gridDim.x * (blockDim.x >> 5);
    constexpr int kU = 8;
    for (uint32_t r = p0 + blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < p1; r += warps) {
        const int t = tok_of_slot[r];
        if ((unsigned)t >= (unsigned)T) continue;  // only a corrupt dispatch could fail this
        const uint4 *src = reinterpret_cast<const uint4 *>(hidden + (size_t)t * H);
        uint4 *dst = reinterpret_cast<uint4 *>(rows + (size_t)r * H);
        for (int c0 = 0; c0 < nv; c0 += 32 * kU) {
            uint4 v[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + u * 32 + lane;
                if (c < nv) v[u] = __ldg(src + c);
            }
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + u * 32 + lane;
                if (c < nv) dst[c] = v[u];
            }
        }
    }
}

__device__ __forceinline__ void add_bf16x8(float *acc, const uint4 &v)
{
    const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(b[i]);
        acc[2 * i] += f.x;
        acc[2 * i + 1] += f.y;
    }
}

// Combine: one thread per (token, 16-byte chunk of the output row).  The k
// routed rows are loaded in batches of 8 independent 16-byte loads before
// they are summed (in j order), so the loads overlap instead of forming a
// chain of dependent memory round trips.  Four resident CTAs per SM (at most
// 64 registers a thread) keep more of those loads in flight.
__global__ void __launch_bounds__(256, 4) combine_kernel(const bf16 *__restrict__ y, const bf16 *__restrict__ y_sh,
                                                      const int32_t *__restrict__ slot_of, int T, int H, int k,
                                                      bf16 *__restrict__ out)
{
    pdl_trigger();
    pdl_wait();
    const int nv = H / 8;
    const int R = T * k;
    const long long total = (long long)T * nv;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int t = (int)(i / nv), c = (int)(i - (long long)t * nv);
        const int32_t *slots = slot_of + (size_t)t * k;
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        for (int j0 = 0; j0 < k; j0 += 8) {
            uint4 v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                if (j0 + u < k) {
                    int slot = __ldg(slots + j0 + u);
                    if ((unsigned)slot >= (unsigned)R) slot = 0;  // only after a dispatch mismatch (status set)
                    v[u] = __ldg(reinterpret_cast<const uint4 *>(y + (size_t)slot * H) + c);
                }
            }
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (j0 + u < k) add_bf16x8(acc, v[u]);
        }
        if (y_sh) add_bf16x8(acc, __ldg(reinterpret_cast<const uint4 *>(y_sh + (size_t)t * H) + c));
        uint4 o;
        o.x = pack_bf16x2(acc[0], acc[1]);
        o.y = pack_bf16x2(acc[2], acc[3]);
        o.z = pack_bf16x2(acc[4], acc[5]);
        o.w = pack_bf16x2(acc[6], acc[7]);
        reinterpret_cast<uint4 *>(out + (size_t)t * H)[c] = o;
    }
}

// Combine through bulk copies (the form launch_combine takes when a ring of
// at least two tokens fits shared memory).  Two CTAs per SM take tokens
// blockIdx.x, blockIdx.x + grid, ...  All threads first stage the CTA's
// dispatch slots in shared memory (one round of independent loads); then
// lane j of warp 0 copies row j of a token (its k routed rows, then its
// shared-expert row) from y into a ring stage with one bulk copy, and the
// consumer warps sum the stage in combine_kernel's order (j ascending, then
// shared, FP32), so both forms give the same bits.  The rows in flight sit
// in shared memory, not in registers, where the thread-per-chunk form was
// bound by the loads its registers could hold (ncu: long-scoreboard stalls,
// 50 % occupancy).  Measured at Qwen3 prefill: the layer step 431 -> 424 us
// (the routed rows y, written just before, are partly still in L2); at
// DeepSeek-V2-Lite 979 -> 972 us.  One CTA per SM with a 200 KB ring was as
// fast inside the step but slower from DRAM alone (41 vs 33 us): a CTA's
// bulk copies in flight were too few to cover DRAM latency.
constexpr int kCombWarps = 8;                            // consumer warps; warp 0 issues the copies
constexpr int kCombTmaThreads = 32 * (kCombWarps + 1);
constexpr int kCombMaxStages = 8;
constexpr int kCombCtasPerSm = 2;
constexpr int kCombSmemBytes = 100 * 1024;               // ring + staged slots, per CTA

struct CombineTmaParams {
    const bf16 *y, *y_sh;
    const int32_t *slot_of;
    int T, H, k, R;
    int nrows;                       // rows per token: k, plus one with shared experts
    int stages;
    uint32_t row_bytes, stage_bytes;
    bf16 *out;
    uint32_t *status;
};

__global__ void __launch_bounds__(kCombTmaThreads, kCombCtasPerSm) combine_tma_kernel(const CombineTmaParams p)
{
    extern __shared__ uint8_t csm[];
    __shared__ __align__(8) uint64_t bars[2 * kCombMaxStages];
    __shared__ volatile int s_abort;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t sbase = (smem_u32(csm) + 127u) & ~127u;
    const uint8_t *sgen = csm + (sbase - smem_u32(csm));
    int *s_slots = reinterpret_cast<int *>(csm + (sbase - smem_u32(csm)) + (size_t)p.stages * p.stage_bytes);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int st) { return bar0 + 8u * (uint32_t)st; };
    auto empty_bar = [&](int st) { return bar0 + 8u * (uint32_t)(kCombMaxStages + st); };
    if (tid == 0) {
        for (int st = 0; st < p.stages; ++st) {
            mbar_init(full_bar(st), 1);
            mbar_init(empty_bar(st), kCombWarps);
        }
        s_abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    pdl_trigger();
    pdl_wait();
    const int grid = (int)gridDim.x, b = (int)blockIdx.x;
    const int ntok = b < p.T ? (p.T - 1 - b) / grid + 1 : 0;
    const int nslots = ntok * p.k;
#pragma unroll 4
    for (int x = tid; x < nslots; x += kCombTmaThreads) {
        const int tl = x / p.k, j = x - tl * p.k;
        int slot = __ldg(p.slot_of + (size_t)(b + tl * grid) * p.k + j);
        if ((unsigned)slot >= (unsigned)p.R) slot = 0;  // only after a dispatch mismatch (status set)
        s_slots[x] = slot;
    }
    __syncthreads();
    if (warp == 0) {
        const uint64_t pol = l2_policy_evict_first();
        uint32_t filled = 0u, last_parity = 0u;
        for (int i = 0; i < ntok; ++i) {
            const int st = i % p.stages;
            const uint32_t ph = (uint32_t)(i / p.stages) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(empty_bar(st), ph ^ 1u, &s_abort, p.status) ? 1 : 0;
            if (!__shfl_sync(~0u, ok, 0)) break;
            if (lane == 0) mbar_expect_tx(full_bar(st), (uint32_t)p.nrows * p.row_bytes);
            __syncwarp();
            if (lane < p.nrows) {
                const int t = b + i * grid;
                const bf16 *src = lane < p.k ? p.y + (size_t)s_slots[i * p.k + lane] * p.H : p.y_sh + (size_t)t * p.H;
                bulk_load_g2s(sbase + (uint32_t)st * p.stage_bytes + (uint32_t)lane * p.row_bytes, src, p.row_bytes,
                              full_bar(st), pol);
            }
            filled |= 1u << st;
            last_parity = (last_parity & ~(1u << st)) | (ph << st);
        }
        // no copy into this CTA's shared memory may still be in flight at its
        // exit (bounded: after an abort the consumers stopped early)
        if (lane == 0)
            for (int st = 0; st < p.stages; ++st)
                if ((filled >> st) & 1u) {
                    const unsigned long long w0 = globaltimer_ns();
                    while (!mbar_try_wait(full_bar(st), (last_parity >> st) & 1u))
                        if (globaltimer_ns() - w0 > kWaitLimitNs) break;
                }
    } else {
        const int ct = tid - 32;
        const int nv = p.H / 8;
        for (int i = 0; i < ntok; ++i) {
            const int st = i % p.stages;
            const uint32_t ph = (uint32_t)(i / p.stages) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(full_bar(st), ph, &s_abort, p.status) ? 1 : 0;
            if (!__shfl_sync(~0u, ok, 0)) break;
            mbar_try_wait(full_bar(st), ph);  // completed: this lane's acquire of the copied rows
            const int t = b + i * grid;
            const uint8_t *stage = sgen + (size_t)st * p.stage_bytes;
            for (int c = ct; c < nv; c += 32 * kCombWarps) {
                float acc[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) acc[q] = 0.f;
                for (int j = 0; j < p.nrows; ++j)
                    add_bf16x8(acc, *reinterpret_cast<const uint4 *>(stage + (size_t)j * p.row_bytes + (size_t)c * 16));
                uint4 o;
                o.x = pack_bf16x2(acc[0], acc[1]);
                o.y = pack_bf16x2(acc[2], acc[3]);
                o.z = pack_bf16x2(acc[4], acc[5]);
                o.w = pack_bf16x2(acc[6], acc[7]);
                reinterpret_cast<uint4 *>(p.out + (size_t)t * p.H)[c] = o;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(empty_bar(st));
        }
    }
}

// Grid for a grid-stride loop over `work` items of 256-thread blocks: enough
// blocks to cover the work once, capped at 8 resident blocks per SM.
int grid_for(long long work, int num_sms)
{
    const long long blocks = (work + 255) / 256;
    const long long cap = 8LL * num_sms;
    return (int)(blocks < cap ? (blocks > 0 ? blocks : 1) : cap);
}

}  // namespace

int column_block(int H) { return H % 256 == 0 ? 256 : 128; }

cudaError_t launch_permute(const Ctx &c)
{
    const Shape &s = c.s;
    const int R = s.T * s.k;
    DispatchParams p;
    p.idx = c.idx; p.ticket = c.ticket; p.w = c.w; p.counts = c.counts;
    p.tile_counts = c.tile_counts;
    p.slots = router_slots(c.s.T);
    p.slots4 = router_slots4(c.s.T);
    p.gemm_ready = c.gemm_ready;
    p.gemm_ready_words = (int)gemm_ready_words(s);
    p.T = s.T; p.R = R; p.k = s.k; p.E = s.E();
    p.offsets = c.offsets; p.slot_of = c.slot_of; p.tok_of_slot = c.tok_of_slot; p.w_of_slot = c.w_of_slot;
    p.status = c.audit.status;
    const int grid = std::max(1, std::min((R + kDispThreads - 1) / kDispThreads, 4 * c.num_sms));
    return launch_pdl(dispatch_kernel, dim3(grid), dim3(kDispThreads), 0, c.stream, p);
}

cudaError_t launch_combine(const Ctx &c)
{
    const Shape &s = c.s;
    {
        CombineTmaParams p;
        p.y = c.y;
        p.y_sh = s.E_sh > 0 ? c.y_sh : nullptr;
        p.slot_of = c.slot_of;
        p.T = s.T; p.H = s.H; p.k = s.k; p.R = s.T * s.k;
        p.nrows = s.k + (s.E_sh > 0 ? 1 : 0);
        p.row_bytes = (uint32_t)s.H * 2u;
        p.stage_bytes = (uint32_t)p.nrows * p.row_bytes;
        p.out = c.out;
        p.status = c.audit.status;
        const int grid = std::max(1, std::min(kCombCtasPerSm * c.num_sms, s.T));
        const long long ntok = (s.T + grid - 1) / grid;
        const long long slots_bytes = (ntok * s.k * 4 + 15) / 16 * 16;
        const long long room = (long long)kCombSmemBytes - 128 - slots_bytes;
        const long long stages = room > 0 ? std::min<long long>(kCombMaxStages, room / p.stage_bytes) : 0;
        if (stages >= 2) {
            p.stages = (int)stages;
            const int smem = (int)(128 + stages * p.stage_bytes + slots_bytes);
            static std::atomic<int> smem_limit[64];
            const cudaError_t err = ensure_dynamic_smem(combine_tma_kernel, smem, smem_limit);
            if (err != cudaSuccess) return err;
            return launch_pdl(combine_tma_kernel, dim3(grid), dim3(kCombTmaThreads), (size_t)smem, c.stream, p);
        }
    }
    return launch_pdl(combine_kernel, dim3(grid_for((long long)s.T * (s.H / 8), c.num_sms)), dim3(256), 0, c.stream,
                      (const bf16 *)c.y, (const bf16 *)(s.E_sh > 0 ? c.y_sh : nullptr), (const int32_t *)c.slot_of, s.T,
                      s.H, s.k, c.out);
}

cudaError_t launch_gather_dispatch_rows(const Ctx &c, int g0, int g1)
{
    const Shape &s = c.s;
    gather_dispatch_rows_kernel<<<c.num_sms * 8, 256, 0, c.stream>>>(c.hidden, c.tok_of_slot, c.offsets, g0, g1,
                                                                     s.T * s.k, s.T, s.H, c.a_perm);
    return cudaGetLastError();
}

}  // namespace pmpe
