// Stages 2 and 5 of the layer: the dispatch order of the routed rows with
// the row gather, and the weighted unpermute-combine.
//
// Dispatch order (the grouping any grouped expert execution needs): rows are
// grouped by expert id and, inside an expert, ordered by token then rank, so
// the order is a pure function of the route log.  One CTA per expert scans
// the [T, k] id list twice: first to count the routed rows of lower ids (its
// offset) and its own, then to write its rows with block-wide scans.  An id
// outside [0, E) is recorded in the status word.  The gather then copies each
// token row into its dispatch row with 16-byte vector loads.
//
// Combine: out_t = bf16( sum_{j < k} y[slot(t, j)] + y_shared[t] ), summed in
// FP32 in a fixed order (j ascending, then shared), so the result of a token
// never depends on the other tokens of the batch.
#include "pmpe_internal.cuh"

namespace pmpe {
namespace {

constexpr int kScanThreads = 1024;
constexpr int kPerThread = 4;

// Exclusive block scan of one value per thread (blockDim.x == kScanThreads).
__device__ __forceinline__ int block_exclusive_scan(int v, int *warp_tot, int &total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(~0u, x, off);
        if (lane >= off) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = warp_tot[lane];
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(~0u, w, off);
            if (lane >= off) w += y;
        }
        warp_tot[lane] = w;  // inclusive
    }
    __syncthreads();
    total = warp_tot[31];
    const int before = warp == 0 ? 0 : warp_tot[warp - 1];
    __syncthreads();  // warp_tot is reused by the next call
    return before + x - v;
}

struct DispatchParams {
    const int32_t *idx;
    const float *w;
    int R, k, E;
    uint32_t *counts, *offsets;
    int32_t *slot_of, *tok_of_slot;
    float *w_of_slot;
    uint32_t *status;
};

__global__ void __launch_bounds__(kScanThreads) dispatch_order_kernel(const DispatchParams p)
{
    __shared__ int warp_tot[32];
    const int e = blockIdx.x, tid = threadIdx.x;
    pdl_trigger();
    pdl_wait();

    // pass 1: this expert's offset = routed rows of lower expert ids; its count
    int less = 0, mine = 0;
    bool bad = false;
    for (int r = tid; r < p.R; r += kScanThreads) {
        const int id = p.idx[r];
        less += id < e;
        mine += id == e;
        bad |= id < 0 || id >= p.E;
    }
    int off, n_e;
    block_exclusive_scan(less, warp_tot, off);
    block_exclusive_scan(mine, warp_tot, n_e);
    if (tid == 0) {
        p.offsets[e] = (uint32_t)off;
        p.counts[e] = (uint32_t)n_e;
        if (e == p.E - 1) p.offsets[p.E] = (uint32_t)(off + n_e);
    }
    if (e == 0 && p.status && __syncthreads_or(bad) && tid == 0) atomicOr(p.status, PMPE_STATUS_BAD_EXPERT_ID);

    // pass 2: this expert's rows in (token, rank) order
    int running = 0;
    for (int base = 0; base < p.R; base += kScanThreads * kPerThread) {
        const int r0 = base + tid * kPerThread;
        int ids[kPerThread];
#pragma unroll
        for (int q = 0; q < kPerThread; ++q) ids[q] = (r0 + q < p.R) ? p.idx[r0 + q] : -1;
        int cnt = 0;
#pragma unroll
        for (int q = 0; q < kPerThread; ++q) cnt += ids[q] == e;
        int total;
        int rank = block_exclusive_scan(cnt, warp_tot, total);
#pragma unroll
        for (int q = 0; q < kPerThread; ++q) {
            if (ids[q] == e) {
                const int r = r0 + q;
                const int slot = off + running + rank;
                if (slot < p.R) {  // always true: off + n_e <= R
                    p.slot_of[r] = slot;
                    p.tok_of_slot[slot] = r / p.k;
                    p.w_of_slot[slot] = p.w[r];
                }
                ++rank;
            }
        }
        running += total;
    }
}

// Row gather: one thread per 16-byte chunk of a dispatch row, so a row is
// copied by H/8 consecutive threads with fully coalesced loads and stores.
__global__ void __launch_bounds__(256) gather_rows_kernel(const bf16 *__restrict__ hidden,
                                                          const int32_t *__restrict__ tok_of_slot, int R, int T,
                                                          int H, bf16 *__restrict__ a_perm)
{
    pdl_trigger();
    pdl_wait();
    const int nv = H / 8;
    const long long total = (long long)R * nv;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int row = (int)(i / nv), c = (int)(i - (long long)row * nv);
        int t = tok_of_slot[row];
        if ((unsigned)t >= (unsigned)T) t = 0;  // only reachable after a dispatch mismatch (status word set)
        reinterpret_cast<uint4 *>(a_perm + (size_t)row * H)[c] =
            __ldg(reinterpret_cast<const uint4 *>(hidden + (size_t)t * H) + c);
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
// chain of dependent memory round trips.
__global__ void __launch_bounds__(256) combine_kernel(const bf16 *__restrict__ y, const bf16 *__restrict__ y_sh,
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

cudaError_t launch_permute(const Ctx &c)
{
    const Shape &s = c.s;
    const int R = s.T * s.k;
    DispatchParams p;
    p.idx = c.idx; p.w = c.w; p.counts = c.counts;
    p.R = R; p.k = s.k; p.E = s.E();
    p.offsets = c.offsets; p.slot_of = c.slot_of; p.tok_of_slot = c.tok_of_slot; p.w_of_slot = c.w_of_slot;
    p.status = c.audit.status;
    cudaError_t err = launch_pdl(dispatch_order_kernel, dim3(s.E()), dim3(kScanThreads), 0, c.stream, p);
    if (err != cudaSuccess) return err;
    return launch_pdl(gather_rows_kernel, dim3(grid_for((long long)R * (s.H / 8), c.num_sms)), dim3(256), 0, c.stream,
                      (const bf16 *)c.hidden, (const int32_t *)c.tok_of_slot, R, s.T, s.H, c.a_perm);
}

cudaError_t launch_combine(const Ctx &c)
{
    const Shape &s = c.s;
    return launch_pdl(combine_kernel, dim3(grid_for((long long)s.T * (s.H / 8), c.num_sms)), dim3(256), 0, c.stream,
                      (const bf16 *)c.y, (const bf16 *)(s.E_sh > 0 ? c.y_sh : nullptr), (const int32_t *)c.slot_of, s.T,
                      s.H, s.k, c.out);
}

}  // namespace pmpe
