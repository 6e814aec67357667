// Stage 1 of the layer: fail-closed policy resolve, masked router, top-k and
// the route log (Sec. 3.1 Eq. 4; App. B.1 steps 2, 4, 5).
//
// One CTA owns 32 consecutive tokens.  It resolves their policy bytes, then
// packs the rows pool by pool: DENY rows first, padded to a multiple of 16,
// then ALLOW rows.  Every 16-row MMA group therefore belongs to one pool and
// multiplies only that pool's router rows -- the other pool's router weights
// are never read for it, so an ineligible expert never becomes a candidate.
// Logits are BF16 x BF16 -> FP32 on mma.sync tensor-core tiles (this GEMM is
// about 0.4 % of the layer's FLOPs), staged through shared memory, and each
// warp then selects the top-k of one token with warp shuffles.
#include "pmpe_internal.cuh"

namespace pmpe {
namespace {

constexpr int kTok = 32;               // tokens per CTA
constexpr int kRows = 48;              // DENY rows padded to 16 + ALLOW rows <= 32 + 15
constexpr int kWarps = 6;              // 3 row groups x 2 expert halves
constexpr int kThreads = kWarps * 32;
constexpr int kBK = 64;                // K elements per pipeline stage (128 bytes per row)
constexpr int kStages = 3;
constexpr int kMaxTiles = kMaxPool / 8 / 2;  // n8 tiles per warp
constexpr int kLdl = kMaxPool + 1;           // logits row stride (floats)

struct RouteParams {
    const bf16 *hidden;
    const uint8_t *policy;
    const bf16 *wr[2];  // [0] public router [E_pub, H], [1] private router [E_priv, H]
    int T, H, E_pub, E_priv, k, renorm;
    int pad[2];         // pool sizes rounded up to 16
    uint8_t *tau;
    int32_t *idx;
    float *w;
    uint32_t *counts;
    uint32_t *route_count, *route_priv_rows;  // audit words, may be NULL
};

__device__ __forceinline__ void ldmatrix_x2(uint32_t &r0, uint32_t &r1, uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];\n" : "=r"(r0), "=r"(r1) : "r"(addr));
}

__global__ void __launch_bounds__(kThreads) router_topk_kernel(const RouteParams p)
{
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int row_tok[kRows];  // token of each packed row, -1 = padding
    __shared__ int s_pd, s_na, s_nd;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int t0 = blockIdx.x * kTok;
    const int ntok = min(kTok, p.T - t0);

    // ---- resolve (only the trusted byte 0x01 is ALLOW) and pack rows by pool
    if (warp == 0) {
        const int t = t0 + lane;
        const bool valid = lane < ntok;
        const bool allow = valid && p.policy != nullptr && p.policy[t] == 0x01;
        const unsigned am = __ballot_sync(~0u, allow);
        const unsigned dm = __ballot_sync(~0u, valid && !allow);
        const int nd = __popc(dm), na = __popc(am);
        const int pd = (nd + 15) & ~15;
        const unsigned below = (1u << lane) - 1u;
        for (int r = lane; r < kRows; r += 32) row_tok[r] = -1;
        __syncwarp();
        if (valid) {
            row_tok[allow ? pd + __popc(am & below) : __popc(dm & below)] = t;
            p.tau[t] = allow ? 1 : 0;
        }
        if (lane == 0) { s_pd = pd; s_na = na; s_nd = nd; }
    }
    __syncthreads();
    const int pd = s_pd, na = s_na;
    const bool need[2] = {s_nd > 0, na > 0};
    const int stage_bytes = (kRows + p.pad[0] + p.pad[1]) * 128;

    // ---- warp role: row group g (16 rows, one pool), expert half
    const int g = warp >> 1, half = warp & 1;
    const int pool = (16 * g < pd) ? 0 : 1;
    const bool active = 16 * g < pd + na;
    const int P = pool ? p.E_priv : p.E_pub;
    const int ntp = (P + 7) >> 3;
    const int h0 = (ntp + 1) >> 1;
    const int tile0 = half ? h0 : 0;
    const int mt = half ? ntp - h0 : h0;

    auto load_stage = [&](int st, int kb) {
        const uint32_t sA = smem_u32(smem + st * stage_bytes);
        const int kofs = kb * kBK;
        for (int i = tid; i < kRows * 8; i += kThreads) {
            const int r = i >> 3, c = i & 7, t = row_tok[r];
            const bf16 *src = p.hidden + (size_t)(t < 0 ? 0 : t) * p.H + kofs + c * 8;
            cp_async16(sA + swz128(r, c), src, t < 0 ? 0 : 16);
        }
        uint32_t sB = sA + kRows * 128;
        for (int q = 0; q < 2; ++q) {
            const int E = q ? p.E_priv : p.E_pub;
            if (need[q]) {
                for (int i = tid; i < p.pad[q] * 8; i += kThreads) {
                    const int r = i >> 3, c = i & 7;
                    const bf16 *src = p.wr[q] + (size_t)min(r, E - 1) * p.H + kofs + c * 8;
                    cp_async16(sB + swz128(r, c), src, r < E ? 16 : 0);
                }
            }
            sB += p.pad[q] * 128;
        }
    };

    float acc[kMaxTiles][4];
#pragma unroll
    for (int i = 0; i < kMaxTiles; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;

    const int nkb = p.H / kBK;
#pragma unroll
    for (int s = 0; s < kStages - 1; ++s) {
        if (s < nkb) load_stage(s, s);
        cp_async_commit();
    }
    for (int kb = 0; kb < nkb; ++kb) {
        cp_async_wait<kStages - 2>();
        __syncthreads();
        const int nk = kb + kStages - 1;
        if (nk < nkb) load_stage(nk % kStages, nk);
        cp_async_commit();
        if (active && mt > 0) {
            const uint32_t sA = smem_u32(smem + (kb % kStages) * stage_bytes);
            const uint32_t sB = sA + kRows * 128 + (pool ? p.pad[0] * 128 : 0);
#pragma unroll
            for (int ks = 0; ks < kBK / 16; ++ks) {
                uint32_t a[4];
                ldmatrix_x4(a[0], a[1], a[2], a[3], sA + swz128(16 * g + (lane & 15), ks * 2 + (lane >> 4)));
#pragma unroll
                for (int nt = 0; nt < kMaxTiles; ++nt) {
                    if (nt < mt) {
                        uint32_t b0, b1;
                        ldmatrix_x2(b0, b1, sB + swz128((tile0 + nt) * 8 + (lane & 7), ks * 2 + ((lane >> 3) & 1)));
                        mma_bf16_16816(acc[nt], a, b0, b1);
                    }
                }
            }
        }
    }
    cp_async_wait<0>();
    __syncthreads();

    // ---- logits to shared memory (reusing the pipeline buffers)
    float *lg = reinterpret_cast<float *>(smem);
    if (active) {
#pragma unroll
        for (int nt = 0; nt < kMaxTiles; ++nt) {
            if (nt < mt) {
                const int e = (tile0 + nt) * 8 + 2 * (lane & 3);
                const int r = 16 * g + (lane >> 2);
                if (e < P) { lg[r * kLdl + e] = acc[nt][0]; lg[(r + 8) * kLdl + e] = acc[nt][2]; }
                if (e + 1 < P) { lg[r * kLdl + e + 1] = acc[nt][1]; lg[(r + 8) * kLdl + e + 1] = acc[nt][3]; }
            }
        }
    }
    __syncthreads();

    // ---- top-k per token: one warp per packed row
    for (int r = warp; r < kRows; r += kWarps) {
        const int t = row_tok[r];
        if (t < 0) continue;
        const int q = r < pd ? 0 : 1;
        const int Pq = q ? p.E_priv : p.E_pub;
        const int base = q ? p.E_pub : 0;
        float v[kMaxPool / 32];
        unsigned avail = 0;
#pragma unroll
        for (int i = 0; i < kMaxPool / 32; ++i) {
            const int e = lane + 32 * i;
            float x = -INFINITY;
            if (e < Pq) {
                x = lg[r * kLdl + e];
                if (x != x) x = -INFINITY;  // NaN never outranks a number
                avail |= 1u << i;
            }
            v[i] = x;
        }
        float my_v = -INFINITY, top = -INFINITY;
        int my_e = 0;
        for (int j = 0; j < p.k; ++j) {
            float bv = -INFINITY;
            int be = 0x7fffffff;
#pragma unroll
            for (int i = 0; i < kMaxPool / 32; ++i)
                if ((avail >> i) & 1u) {
                    if (be == 0x7fffffff || v[i] > bv) { bv = v[i]; be = lane + 32 * i; }
                }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                const float ov = __shfl_xor_sync(~0u, bv, off);
                const int oe = __shfl_xor_sync(~0u, be, off);
                if (ov > bv || (ov == bv && oe < be)) { bv = ov; be = oe; }
            }
            if ((be & 31) == lane) avail &= ~(1u << (be >> 5));
            if (lane == j) { my_v = bv; my_e = be; }
            if (j == 0) top = bv;
        }
        // softmax weights
        float denom = 0.f;
        if (p.renorm) {
            denom = lane < p.k ? expf(my_v - top) : 0.f;
        } else {
#pragma unroll
            for (int i = 0; i < kMaxPool / 32; ++i)
                if (lane + 32 * i < Pq) denom += expf(v[i] - top);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) denom += __shfl_xor_sync(~0u, denom, off);
        const int gid = base + my_e;
        const unsigned privm = __ballot_sync(~0u, lane < p.k && gid >= p.E_pub);
        if (lane < p.k) {
            p.idx[(size_t)t * p.k + lane] = gid;
            p.w[(size_t)t * p.k + lane] = expf(my_v - top) / denom;
            atomicAdd(&p.counts[gid], 1u);
            if (p.route_count) atomicAdd(&p.route_count[gid], 1u);
        }
        if (lane == 0 && p.route_priv_rows) atomicAdd(&p.route_priv_rows[t], (unsigned)__popc(privm));
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
    cudaError_t err = cudaMemsetAsync(c.counts, 0, sizeof(uint32_t) * s.E(), c.stream);
    if (err != cudaSuccess) return err;
    RouteParams p;
    p.hidden = c.hidden;
    p.policy = c.policy;
    p.wr[0] = c.router_pub;
    p.wr[1] = c.router_priv;
    p.T = s.T; p.H = s.H; p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.k = s.k; p.renorm = s.renorm;
    p.pad[0] = (s.E_pub + 15) & ~15;
    p.pad[1] = (s.E_priv + 15) & ~15;
    p.tau = c.tau; p.idx = c.idx; p.w = c.w; p.counts = c.counts;
    p.route_count = c.audit.route_count;
    p.route_priv_rows = c.audit.route_priv_rows;
    const int pipe = kStages * (kRows + p.pad[0] + p.pad[1]) * 128;
    const int logits = kRows * kLdl * (int)sizeof(float);
    const int smem = pipe > logits ? pipe : logits;
    err = cudaFuncSetAttribute(router_topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (err != cudaSuccess) return err;
    const int grid = (s.T + kTok - 1) / kTok;
    router_topk_kernel<<<grid, kThreads, smem, c.stream>>>(p);
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
