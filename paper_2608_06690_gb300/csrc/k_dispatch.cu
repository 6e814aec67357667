// Stages 2 and 5 of the layer: the dispatch order of the routed rows with
// the row gather, and the weighted unpermute-combine.
//
// Dispatch order (the grouping any grouped expert execution needs): rows are
// grouped by expert id and, inside an expert, ordered by token then rank, so
// the order is a pure function of the route log.  One CTA per expert scans
// the [T, k] id list with block-wide ballots and writes that expert's rows;
// its row count is cross-checked against the router's atomic count and a
// mismatch is recorded in the status word.  The gather then copies each
// token row into its dispatch row with 16-byte vector loads, one warp per row.
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
    const uint32_t *counts;
    int R, k, E;
    uint32_t *offsets;
    int32_t *slot_of, *tok_of_slot;
    float *w_of_slot;
    uint32_t *status;
};

__global__ void __launch_bounds__(kScanThreads) dispatch_order_kernel(const DispatchParams p)
{
    __shared__ int warp_tot[32];
    __shared__ unsigned s_off;
    const int e = blockIdx.x, tid = threadIdx.x;

    // offset of expert e = sum of the router's counts of the experts before it
    unsigned part = 0;
    for (int i = tid; i < e; i += kScanThreads) part += p.counts[i];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(~0u, part, off);
    if (tid == 0) s_off = 0;
    __syncthreads();
    if ((tid & 31) == 0 && part) atomicAdd(&s_off, part);
    __syncthreads();
    const unsigned off = s_off;
    const unsigned n_e = p.counts[e];
    if (tid == 0) {
        p.offsets[e] = off;
        if (e == p.E - 1) p.offsets[p.E] = off + n_e;
    }

    int running = 0;
    bool bad = false;
    for (int base = 0; base < p.R; base += kScanThreads * kPerThread) {
        const int r0 = base + tid * kPerThread;
        int ids[kPerThread];
#pragma unroll
        for (int q = 0; q < kPerThread; ++q) ids[q] = (r0 + q < p.R) ? p.idx[r0 + q] : -1;
        int mine = 0;
#pragma unroll
        for (int q = 0; q < kPerThread; ++q) {
            mine += ids[q] == e;
            bad |= (r0 + q < p.R) && (ids[q] < 0 || ids[q] >= p.E);
        }
        int total;
        int rank = block_exclusive_scan(mine, warp_tot, total);
#pragma unroll
        for (int q = 0; q < kPerThread; ++q) {
            if (ids[q] == e) {
                const int r = r0 + q;
                const int slot = (int)off + running + rank;
                if (slot < p.R) {  // always true when the router's counts match its ids
                    p.slot_of[r] = slot;
                    p.tok_of_slot[slot] = r / p.k;
                    p.w_of_slot[slot] = p.w[r];
                }
                ++rank;
            }
        }
        running += total;
    }
    if (p.status) {
        if (tid == 0 && (unsigned)running != n_e) atomicOr(p.status, PMPE_STATUS_DISPATCH_MISMATCH);
        if (e == 0 && __syncthreads_or(bad) && tid == 0) atomicOr(p.status, PMPE_STATUS_BAD_EXPERT_ID);
    }
}

// One warp copies one H-wide BF16 row with 16-byte vectors.
__global__ void __launch_bounds__(256) gather_rows_kernel(const bf16 *__restrict__ hidden,
                                                          const int32_t *__restrict__ tok_of_slot, int R, int T,
                                                          int H, bf16 *__restrict__ a_perm)
{
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (row >= R) return;
    int t = tok_of_slot[row];
    if ((unsigned)t >= (unsigned)T) t = 0;  // only reachable after a dispatch mismatch (status word set)
    const uint4 *src = reinterpret_cast<const uint4 *>(hidden + (size_t)t * H);
    uint4 *dst = reinterpret_cast<uint4 *>(a_perm + (size_t)row * H);
    const int nv = H / 8;
    for (int c = lane; c < nv; c += 32) dst[c] = __ldg(src + c);
}

__global__ void __launch_bounds__(256) combine_kernel(const bf16 *__restrict__ y, const bf16 *__restrict__ y_sh,
                                                      const int32_t *__restrict__ slot_of, int T, int H, int k,
                                                      bf16 *__restrict__ out)
{
    const int t = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (t >= T) return;
    int my_slot = lane < k ? slot_of[(size_t)t * k + lane] : 0;
    if ((unsigned)my_slot >= (unsigned)(T * k)) my_slot = 0;  // only after a dispatch mismatch (status word set)
    const int nv = H / 8;
    for (int c = lane; c < nv; c += 32) {
        float acc[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = 0.f;
        for (int j = 0; j < k; ++j) {
            const int slot = __shfl_sync(~0u, my_slot, j);
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(y + (size_t)slot * H) + c);
            const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = __bfloat1622float2(b[i]);
                acc[2 * i] += f.x;
                acc[2 * i + 1] += f.y;
            }
        }
        if (y_sh) {
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(y_sh + (size_t)t * H) + c);
            const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = __bfloat1622float2(b[i]);
                acc[2 * i] += f.x;
                acc[2 * i + 1] += f.y;
            }
        }
        uint4 o;
        o.x = pack_bf16x2(acc[0], acc[1]);
        o.y = pack_bf16x2(acc[2], acc[3]);
        o.z = pack_bf16x2(acc[4], acc[5]);
        o.w = pack_bf16x2(acc[6], acc[7]);
        reinterpret_cast<uint4 *>(out + (size_t)t * H)[c] = o;
    }
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
    dispatch_order_kernel<<<s.E(), kScanThreads, 0, c.stream>>>(p);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    gather_rows_kernel<<<(R + 7) / 8, 256, 0, c.stream>>>(c.hidden, c.tok_of_slot, R, s.T, s.H, c.a_perm);
    return cudaGetLastError();
}

cudaError_t launch_combine(const Ctx &c)
{
    const Shape &s = c.s;
    combine_kernel<<<(s.T + 7) / 8, 256, 0, c.stream>>>(c.y, s.E_sh > 0 ? c.y_sh : nullptr, c.slot_of, s.T, s.H,
                                                         s.k, c.out);
    return cudaGetLastError();
}

}  // namespace pmpe
