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
