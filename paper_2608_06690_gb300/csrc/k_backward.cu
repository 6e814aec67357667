// Backward of the private branch (G2, Sec. 2.2 and Sec. 3.2: only the private
// experts and the private router are trained; the public parameters are frozen
// and get no gradient).  For L = sum_t dout_t . out_t and the routing the
// forward took (read from the forward's workspace):
//
//   private expert q, its dispatch rows r (tokens t, weights w):
//     Z_r   = W_down,q^T dout_t           (so dL/dw_r = Z_r . a_r, da_r = w_r Z_r)
//     g, u  = W_gate,q h_t, W_up,q h_t    (recomputed)
//     dG_r  = w_r Z_r u silu'(g),  dU_r = w_r Z_r silu(g)
//     dW_gate,q = sum_r dG_r h_t^T,  dW_up,q = sum_r dU_r h_t^T,  dW_down,q = sum_r dout_t (w_r a_r)^T
//   router, per ALLOW token (softmax over the private pool, renormalised over
//   the top-k or not):  dz = softmax gradient of dL/dw,  dW_router,e = sum_t dz_{t,e} h_t^T
//
// The expert contractions run on the tensor cores (k_backward_tc.cu); this
// file holds the row gather, the router's gradient and the launch sequence.
#include <algorithm>
#include <cstring>

#include "pmpe_internal.cuh"

namespace pmpe {
namespace {

// Upstream gradients of the dispatch rows of experts g0 .. g1 - 1, in
// dispatch order, and 64 zero rows after the last one (the weight-gradient
// GEMM reads up to 63 rows past an expert's rows, multiplied by zeros there,
// which must be finite).  One warp per row, eight 16-byte loads in flight per
// lane.
__global__ void __launch_bounds__(256) bwd_gather_kernel(const bf16 *dout, const int32_t *tok_of_slot,
                                                         const uint32_t *offsets, int g0, int g1, int R, int H,
                                                         bf16 *dout_rows)
{
    const uint32_t p0 = min(offsets[g0], (uint32_t)R), p1 = min(max(offsets[g1], p0), (uint32_t)R);
    const int nv = H / 8;
    const int rows = (int)(p1 - p0);
    const int lane = threadIdx.x & 31;
    const int warps = gridDim.x * (blockDim.x >> 5);
    constexpr int kU = 8;
    for (int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows + 64; r += warps) {
        const uint4 *src = r < rows ? reinterpret_cast<const uint4 *>(dout + (size_t)tok_of_slot[p0 + r] * H) : nullptr;
        uint4 *dst = reinterpret_cast<uint4 *>(dout_rows + (size_t)r * H);
        for (int c0 = 0; c0 < nv; c0 += 32 * kU) {
            uint4 v[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + u * 32 + lane;
                v[u] = (src != nullptr && c < nv) ? src[c] : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + u * 32 + lane;
                if (c < nv) dst[c] = v[u];
            }
        }
    }
}

// Each pool's tokens in ascending order, the DENY pool's first: pool_tok[0,
// nd) and pool_tok[nd, T), pool_n = {nd, na}.  One CTA: every thread ranks a
// contiguous run of tokens.
__global__ void __launch_bounds__(1024) bwd_pool_tokens_kernel(const uint8_t *tau, int T, int32_t *pool_tok,
                                                               int *pool_n)
{
    __shared__ int s_warp[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    pdl_wait();
    const int per = (T + blockDim.x - 1) / blockDim.x;
    const int t0 = min(T, tid * per), t1 = min(T, t0 + per);
    int a = 0;
    for (int t = t0; t < t1; ++t) a += tau[t] ? 1 : 0;
    int x = a;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(~0u, x, off);
        if (lane >= off) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    int before = 0, na = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
        before += w < warp ? s_warp[w] : 0;
        na += s_warp[w];
    }
    int ra = before + x - a, rd = t0 - (before + x - a);  // ranks of this run's first token in its pool
    const int nd = T - na;
    for (int t = t0; t < t1; ++t) {
        if (tau[t]) pool_tok[nd + ra++] = t;
        else pool_tok[rd++] = t;
    }
    if (tid == 0) {
        pool_n[0] = nd;
        pool_n[1] = na;
    }
}

// Shared-memory tiled FP32 GEMMs over one pool's tokens (blockIdx.z = pool q
// - pool0; blockIdx.x = the 64-token block of the pool's list): 64 x 64
// outputs a CTA, K in steps of 32, a 4 x 4 micro-tile a thread.  A DENY
// token's row only ever meets the public router, an ALLOW token's only the
// private one.
constexpr int kPT = 64, kPK = 32, kSkew = 4;  // tile, K step, row skew of the shared tiles

// The pool-softmax logits z[t][e] = sum_h h[t][h] W_q[e][h] of each token
// of the pool and every expert of it, as ksplit partial sums over equal
// ranges of h: blockIdx.y = 64-expert chunk * ksplit + range, partial s into
// part[s][t][e] (rows ld apart); the dz kernel adds them in range order.
__global__ void __launch_bounds__(256) bwd_pool_logits_kernel(const bf16 *hidden, const bf16 *router_pub,
                                                              const bf16 *router_priv, const int32_t *pool_tok,
                                                              const int *pool_n, int T, int H, int E_pub, int E_priv,
                                                              int pool0, int ksplit, int ld, float *part)
{
    __shared__ __align__(16) float As[kPK][kPT + kSkew], Bs[kPK][kPT + kSkew];
    __shared__ int s_tok[kPT];
    pdl_wait();
    const int q = pool0 + blockIdx.z;
    const int ks = blockIdx.y % ksplit;
    const int n = pool_n[q], i0 = blockIdx.x * kPT, e0 = (blockIdx.y / ksplit) * kPT;
    const int E_q = q ? E_priv : E_pub;
    if (i0 >= n || e0 >= E_q) return;  // uniform
    const int32_t *toks = pool_tok + (q ? pool_n[0] : 0);
    const bf16 *W = q ? router_priv : router_pub;
    const int hs = H / ksplit, h0 = ks * hs;
    float *dz = part + (size_t)ks * T * ld;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    if (tid < kPT) s_tok[tid] = i0 + tid < n ? toks[i0 + tid] : -1;
    __syncthreads();
    const int lr = tid >> 2, lk = (tid & 3) * 8;  // this thread's loads: row lr, 8 K values from lk
    const int tok = s_tok[lr], er = e0 + lr;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = h0; k0 < h0 + hs; k0 += kPK) {
        const uint4 av = tok >= 0 ? *reinterpret_cast<const uint4 *>(hidden + (size_t)tok * H + k0 + lk)
                                  : make_uint4(0u, 0u, 0u, 0u);
        const uint4 bv = er < E_q ? *reinterpret_cast<const uint4 *>(W + (size_t)er * H + k0 + lk)
                                  : make_uint4(0u, 0u, 0u, 0u);
        __syncthreads();  // the previous step's tiles are consumed
        const __nv_bfloat162 *ab = reinterpret_cast<const __nv_bfloat162 *>(&av);
        const __nv_bfloat162 *bb = reinterpret_cast<const __nv_bfloat162 *>(&bv);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 fa = __bfloat1622float2(ab[j]), fb = __bfloat1622float2(bb[j]);
            As[lk + 2 * j][lr] = fa.x; As[lk + 2 * j + 1][lr] = fa.y;
            Bs[lk + 2 * j][lr] = fb.x; Bs[lk + 2 * j + 1][lr] = fb.y;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < kPK; ++kk) {
            const float4 a4 = *reinterpret_cast<const float4 *>(&As[kk][ty * 4]);
            const float4 b4 = *reinterpret_cast<const float4 *>(&Bs[kk][tx * 4]);
            const float a[4] = {a4.x, a4.y, a4.z, a4.w}, b[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] += a[i] * b[j];
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int t = s_tok[ty * 4 + i];
        if (t < 0) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int e = e0 + tx * 4 + j;
            if (e < E_q) dz[(size_t)t * ld + e] = acc[i][j];
        }
    }
}

// The pool-softmax router term of the input gradient, added in place:
// d_hidden[t][c] += sum_e dz[t][e] W_q[e][c] over the pool's experts in
// order (blockIdx.y = 64-column block).
__global__ void __launch_bounds__(256) bwd_pool_router_term_kernel(const float *dz, int ld, const bf16 *router_pub,
                                                                   const bf16 *router_priv, const int32_t *pool_tok,
                                                                   const int *pool_n, int H, int E_pub, int E_priv,
                                                                   float *d_hidden)
{
    __shared__ __align__(16) float As[kPK][kPT + kSkew], Bs[kPK][kPT + kSkew];
    __shared__ int s_tok[kPT];
    pdl_wait();
    const int q = blockIdx.z;
    const int n = pool_n[q], i0 = blockIdx.x * kPT, c0 = blockIdx.y * kPT;
    if (i0 >= n) return;  // uniform
    const int E_q = q ? E_priv : E_pub;
    const int32_t *toks = pool_tok + (q ? pool_n[0] : 0);
    const bf16 *W = q ? router_priv : router_pub;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    if (tid < kPT) s_tok[tid] = i0 + tid < n ? toks[i0 + tid] : -1;
    __syncthreads();
    const int ar = tid >> 2, ak = (tid & 3) * 8;  // A loads: token row ar, 8 experts from ak
    const int br = tid >> 3, bc = (tid & 7) * 8;  // B loads: expert row br, 8 columns from bc
    const int tok = s_tok[ar];
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < E_q; k0 += kPK) {
        float av[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int e = k0 + ak + j;
            av[j] = (tok >= 0 && e < E_q) ? dz[(size_t)tok * ld + e] : 0.f;
        }
        uint4 bv = make_uint4(0u, 0u, 0u, 0u);
        if (k0 + br < E_q) bv = *reinterpret_cast<const uint4 *>(W + (size_t)(k0 + br) * H + c0 + bc);
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 8; ++j) As[ak + j][ar] = av[j];
        const __nv_bfloat162 *bb = reinterpret_cast<const __nv_bfloat162 *>(&bv);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 fb = __bfloat1622float2(bb[j]);
            Bs[br][bc + 2 * j] = fb.x;
            Bs[br][bc + 2 * j + 1] = fb.y;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < kPK; ++kk) {
            const float4 a4 = *reinterpret_cast<const float4 *>(&As[kk][ty * 4]);
            const float4 b4 = *reinterpret_cast<const float4 *>(&Bs[kk][tx * 4]);
            const float a[4] = {a4.x, a4.y, a4.z, a4.w}, b[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] += a[i] * b[j];
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int t = s_tok[ty * 4 + i];
        if (t < 0) continue;
        float4 *o = reinterpret_cast<float4 *>(d_hidden + (size_t)t * H + c0 + tx * 4);
        float4 v = *o;
        v.x += acc[i][0]; v.y += acc[i][1]; v.z += acc[i][2]; v.w += acc[i][3];
        *o = v;
    }
}

// Router gradient per token (one warp): the softmax gradient dz over the
// token's pool from dL/dw of its k rows (summed from the expert GEMM's per-tile
// partials, indexed by dispatch slot) -- renormalised over the top-k, or the
// pool softmax, whose probabilities need every logit of the pool: those come
// as partial sums from bwd_pool_logits_kernel.  both_pools = 0:
// the private pool only,
// dz [T][ld = E_priv], zero for DENY tokens; both_pools = 1: each token's own
// pool (tau selects it), dz [T][ld] holding that pool's E_pub or E_priv entries.
__global__ void bwd_router_kernel(const uint8_t *tau, const int32_t *idx, const float *wts, const int32_t *slot_of,
                                  const float *gw_part, int n_part, int T, int E_pub, int E_priv, int k, int renorm,
                                  int both_pools, int ld, const float *logit_part, int ksplit, float *dz)
{
    const int lane = threadIdx.x & 31;
    const int warps = gridDim.x * (blockDim.x >> 5);
    for (int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); t < T; t += warps) {
        float *dzt = dz + (size_t)t * ld;
        const int priv = tau[t] ? 1 : 0;
        if (!priv && !both_pools) {
            for (int e = lane; e < E_priv; e += 32) dzt[e] = 0.f;
            continue;
        }
        const int E_pool = priv ? E_priv : E_pub;
        const int e_base = priv ? E_pub : 0;
        // lane j < k holds pick j: its pool id and dL/dw
        int pe = -1;
        float g = 0.f, wj = 0.f;
        if (lane < k) {
            pe = idx[(size_t)t * k + lane] - e_base;
            const int slot = slot_of[(size_t)t * k + lane];
            const float *gp = gw_part + (size_t)slot * n_part;
            for (int j = 0; j < n_part; ++j) g += gp[j];  // the per-tile partials of dL/dw, in order
            wj = wts[(size_t)t * k + lane];
        }
        float sum = wj * g;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(~0u, sum, off);
        if (renorm) {
            for (int e = lane; e < E_pool; e += 32) dzt[e] = 0.f;
            __syncwarp();
            if (lane < k && pe >= 0 && pe < E_pool) dzt[pe] = wj * (g - sum);
        } else {  // the pool's logits: the partial sums in range order, then the softmax gradient
            for (int e = lane; e < E_pool; e += 32) {
                float z = 0.f;
                for (int s2 = 0; s2 < ksplit; ++s2) z += logit_part[((size_t)s2 * T + t) * ld + e];
                dzt[e] = z;
            }
            __syncwarp();
            float mx = -INFINITY;
            for (int e = lane; e < E_pool; e += 32) mx = fmaxf(mx, dzt[e]);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(~0u, mx, off));
            float den = 0.f;
            for (int e = lane; e < E_pool; e += 32) den += expf(dzt[e] - mx);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(~0u, den, off);
            __syncwarp();
            // dz_e = p_e (dL/dp_e - sum): -p_e sum everywhere, plus p_e dL/dw_j at the k picks
            float pj = 0.f;
            if (lane < k && pe >= 0 && pe < E_pool) pj = expf(dzt[pe] - mx) / den;
            __syncwarp();
            for (int e = lane; e < E_pool; e += 32) dzt[e] = -(expf(dzt[e] - mx) / den) * sum;
            __syncwarp();
            if (lane < k && pe >= 0 && pe < E_pool) dzt[pe] += pj * g;
        }
        __syncwarp();
    }
}

// dW_router[e][c] = sum_t dz[t][e] h[t][c] in FP32, split over the tokens:
// CTA (x, y, z) owns a 32 x 128 output tile and the z-th token range, staged
// through shared memory 32 tokens at a time, and writes its partial sum to
// part[z]; bwd_router_reduce_kernel adds the partials in split order, so the
// result does not depend on scheduling.  A block of 32 DENY tokens (dz
// exactly zero) is skipped: its products would add exact zeros.  A range of
// DENY tokens only writes no partial and clears active[z], so the reduction
// skips it; otherwise active[z] = 1.  dz rows are ld apart; a DENY token's
// row is read as zeros (it may hold its public pool's gradient).
__global__ void __launch_bounds__(256) bwd_router_wgrad_kernel(const float *dz, int ld, const bf16 *hidden,
                                                               const uint8_t *tau, int T, int H, int E_priv,
                                                               int tok_per_split, float *part, int *active)
{
    __shared__ float s_dz[32][33];
    __shared__ __align__(16) float s_h[32][128];
    const int e0 = blockIdx.y * 32, c0 = blockIdx.x * 128;
    const int t_begin = blockIdx.z * tok_per_split, t_end = min(T, t_begin + tok_per_split);
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 8 row groups x 32 columns
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
    bool any = false;
    for (int t0 = t_begin; t0 < t_end; t0 += 32) {
        if (!__syncthreads_or(threadIdx.x < 32 && t0 + (int)threadIdx.x < t_end && tau[t0 + threadIdx.x])) continue;
        any = true;
        for (int i = threadIdx.x; i < 32 * 32; i += 256) {
            const int tt = i >> 5, ee = i & 31;
            s_dz[tt][ee] = (t0 + tt < t_end && e0 + ee < E_priv && tau[t0 + tt]) ? dz[(size_t)(t0 + tt) * ld + e0 + ee]
                                                                                  : 0.f;
        }
        for (int i = threadIdx.x; i < 32 * 16; i += 256) {
            const int tt = i >> 4, cc = (i & 15) * 8;
            float4 lo = make_float4(0.f, 0.f, 0.f, 0.f), hi = lo;
            if (t0 + tt < t_end && c0 + cc < H) {
                const uint4 v = *reinterpret_cast<const uint4 *>(hidden + (size_t)(t0 + tt) * H + c0 + cc);
                const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&v);
                const float2 f0 = __bfloat1622float2(b2[0]), f1 = __bfloat1622float2(b2[1]);
                const float2 f2 = __bfloat1622float2(b2[2]), f3 = __bfloat1622float2(b2[3]);
                lo = make_float4(f0.x, f0.y, f1.x, f1.y);
                hi = make_float4(f2.x, f2.y, f3.x, f3.y);
            }
            *reinterpret_cast<float4 *>(&s_h[tt][cc]) = lo;
            *reinterpret_cast<float4 *>(&s_h[tt][cc + 4]) = hi;
        }
        __syncthreads();
#pragma unroll 4
        for (int tt = 0; tt < 32; ++tt) {
            float hv[4], dv[4];
#pragma unroll
            for (int b = 0; b < 4; ++b) hv[b] = s_h[tt][tx + 32 * b];
#pragma unroll
            for (int a = 0; a < 4; ++a) dv[a] = s_dz[tt][ty + 8 * a];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] += dv[a] * hv[b];
        }
        __syncthreads();
    }
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) active[blockIdx.z] = any ? 1 : 0;
    if (!any) return;  // uniform over the CTA
    float *out = part + (size_t)blockIdx.z * E_priv * H;
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int e = e0 + ty + 8 * a, c = c0 + tx + 32 * b;
            if (e < E_priv && c < H) out[(size_t)e * H + c] = acc[a][b];
        }
}

// d_router = the active partials summed in split order (a skipped range
// contributes exact zeros).
__global__ void bwd_router_reduce_kernel(const float *part, const int *active, int nsplit, int n, float *d_router)
{
    __shared__ int s_list[kMaxRouterSplits];
    __shared__ int s_n;
    if (threadIdx.x == 0) {
        int m = 0;
        for (int z = 0; z < nsplit; ++z)
            if (active[z]) s_list[m++] = z;
        s_n = m;
    }
    __syncthreads();
    const int m = s_n;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        float a = 0.f;
        int j = 0;
        for (; j + 4 <= m; j += 4) {  // four loads in flight, summed in order
            const float v0 = part[(size_t)s_list[j] * n + i], v1 = part[(size_t)s_list[j + 1] * n + i];
            const float v2 = part[(size_t)s_list[j + 2] * n + i], v3 = part[(size_t)s_list[j + 3] * n + i];
            a += v0; a += v1; a += v2; a += v3;
        }
        for (; j < m; ++j) a += part[(size_t)s_list[j] * n + i];
        d_router[i] = a;
    }
}

// Token splits of the router weight gradient: enough CTAs for eight per SM
// (ranges of DENY tokens end at once, so short ranges keep the SMs busy),
// each range a multiple of 32 tokens, at most kMaxRouterSplits ranges.
int router_splits(const Shape &s, int num_sms, int *tok_per_split)
{
    const int tiles = ((s.H + 127) / 128) * ((s.E_priv + 31) / 32);
    const int chunks = std::max(1, (s.T + 31) / 32);
    int n = std::min(std::min(kMaxRouterSplits, chunks), std::max(1, (8 * num_sms + tiles - 1) / tiles));
    const int per = ((chunks + n - 1) / n) * 32;
    n = std::max(1, (s.T + per - 1) / per);
    *tok_per_split = per;
    return n;
}

}  // namespace

// Scratch of the backward, in order: dout rows [R + 64][H], Z, [dG | dU] and
// w act in the padded row layout ([RP][I], [RP][2I], [RP][I], BF16), the dL/dw
// partials [R][I / 128], dz [T][E_priv] and the router weight-gradient
// partials [splits][E_priv][H] (FP32).
void launch_gather_rows(const bf16 *dout, const int32_t *tok_of_slot, const uint32_t *offsets, int g0, int g1, int R,
                        int H, bf16 *rows, int num_sms, cudaStream_t st)
{
    bwd_gather_kernel<<<num_sms * 8, 256, 0, st>>>(dout, tok_of_slot, offsets, g0, g1, R, H, rows);
}

int router_logit_splits(const Shape &s)
{
    const int m = s.H / 128;  // ranges of h: a divisor of H / 128, at most 8
    for (int d = 8; d > 1; --d)
        if (m % d == 0) return d;
    return 1;
}

cudaError_t launch_router_dz(const Ctx &c, const float *gw_part, int both_pools, int ld, float *dz, int32_t *pool_tok,
                             int *pool_n, float *logit_part)
{
    const Shape &s = c.s;
    cudaError_t err;
    const int ksplit = router_logit_splits(s);
    if (!s.renorm) {  // the pool softmax needs every logit of the token's pool: tiled GEMMs per pool
        bwd_pool_tokens_kernel<<<1, 1024, 0, c.stream>>>(c.tau, s.T, pool_tok, pool_n);
        if ((err = cudaGetLastError()) != cudaSuccess) return err;
        const int chunks = (std::max(both_pools ? s.E_pub : 0, s.E_priv) + kPT - 1) / kPT;
        const dim3 grid((s.T + kPT - 1) / kPT, chunks * ksplit, both_pools ? 2 : 1);
        bwd_pool_logits_kernel<<<grid, 256, 0, c.stream>>>(c.hidden, c.router_pub, c.router_priv, pool_tok, pool_n,
                                                             s.T, s.H, s.E_pub, s.E_priv, both_pools ? 0 : 1, ksplit, ld,
                                                             logit_part);
        if ((err = cudaGetLastError()) != cudaSuccess) return err;
    }
    bwd_router_kernel<<<c.num_sms * 4, 256, 0, c.stream>>>(c.tau, c.idx, c.w, c.slot_of, gw_part, s.I / 128, s.T,
                                                           s.E_pub, s.E_priv, s.k, s.renorm, both_pools, ld, logit_part,
                                                           ksplit, dz);
    return cudaGetLastError();
}

cudaError_t launch_router_term(const Ctx &c, const float *dz, int ld, const int32_t *pool_tok, const int *pool_n,
                               float *d_hidden)
{
    const Shape &s = c.s;
    const dim3 grid((s.T + kPT - 1) / kPT, s.H / kPT, 2);
    bwd_pool_router_term_kernel<<<grid, 256, 0, c.stream>>>(dz, ld, c.router_pub, c.router_priv, pool_tok, pool_n,
                                                              s.H, s.E_pub, s.E_priv, d_hidden);
    return cudaGetLastError();
}

struct BwdScratch {
    bf16 *dout_rows, *zpad, *dgu, *wact;
    float *gw_part, *dz, *part;
    int *active;  // per token range of the router weight gradient: 1 if it holds an ALLOW token
    int32_t *pool_tok;  // [T] each pool's tokens (pool softmax), then pool_n [2]
    int *pool_n;
    float *logit_part;  // [router_logit_splits][T][E_priv] partial pool logits (pool softmax)
    size_t bytes;
};

static BwdScratch backward_scratch(const Shape &s, uint8_t *base)
{
    const size_t R = (size_t)s.T * s.k, H = s.H, I = s.I, RP = backward_padded_rows(s);
    auto al = [](size_t x) { return (x + 255) / 256 * 256; };
    BwdScratch b;
    size_t o = 0;
    b.dout_rows = (bf16 *)(base + o); o += al((R + 64) * H * 2);
    b.zpad = (bf16 *)(base + o);      o += al(RP * I * 2);
    b.dgu = (bf16 *)(base + o);       o += al(RP * 2 * I * 2);
    b.wact = (bf16 *)(base + o);      o += al(RP * I * 2);
    b.gw_part = (float *)(base + o);  o += al(R * (I / 128) * 4);
    b.dz = (float *)(base + o);       o += al((size_t)s.T * s.E_priv * 4);
    b.part = (float *)(base + o);     o += al(router_wgrad_part_bytes(s));
    b.active = (int *)(base + o);     o += al(kMaxRouterSplits * 4);
    b.pool_tok = (int32_t *)(base + o); o += al((size_t)s.T * 4);
    b.pool_n = (int *)(base + o);     o += al(2 * 4);
    // (sized whatever the routing: the size query does not know it)
    b.logit_part = (float *)(base + o); o += al((size_t)router_logit_splits(s) * s.T * s.E_priv * 4);
    b.bytes = o;
    return b;
}

size_t backward_workspace_bytes(const Shape &s)
{
    if (s.T == 0) return 256;
    return backward_scratch(s, nullptr).bytes;
}

cudaError_t launch_backward_private(const Ctx &c, const bf16 *dout, float *d_router, float *d_gate, float *d_up,
                                    float *d_down, uint8_t *bws)
{
    const Shape &s = c.s;
    const int R = s.T * s.k, H = s.H;
    const BwdScratch b = backward_scratch(s, bws);
    const int E = s.E();
    cudaStream_t st = c.stream;

    launch_gather_rows(dout, c.tok_of_slot, c.offsets, s.E_pub, E, R, H, b.dout_rows, c.num_sms, st);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    if ((err = launch_backward_rows(c, b.dout_rows, b.zpad, b.dgu, b.wact, b.gw_part)) != cudaSuccess) return err;
    if ((err = launch_router_dz(c, b.gw_part, 0, s.E_priv, b.dz, b.pool_tok, b.pool_n, b.logit_part)) != cudaSuccess) return err;
    if ((err = launch_router_wgrad(c, b.dz, s.E_priv, b.part, b.active, d_router)) != cudaSuccess) return err;
    return launch_backward_wgrad(c, b.dout_rows, b.dgu, b.wact, d_gate, d_up, d_down);
}

size_t router_wgrad_part_bytes(const Shape &s)
{
    const size_t splits = (size_t)std::min(kMaxRouterSplits, (s.T + 31) / 32);
    return splits * s.E_priv * s.H * 4;
}

cudaError_t launch_router_wgrad(const Ctx &c, const float *dz, int ld, float *part, int *active, float *d_router)
{
    const Shape &s = c.s;
    int per = 32;
    const int nsplit = router_splits(s, c.num_sms, &per);
    dim3 grid((s.H + 127) / 128, (s.E_priv + 31) / 32, nsplit);
    bwd_router_wgrad_kernel<<<grid, 256, 0, c.stream>>>(dz, ld, c.hidden, c.tau, s.T, s.H, s.E_priv, per, part,
                                                        active);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    const int n = s.E_priv * s.H;
    bwd_router_reduce_kernel<<<std::min((n + 255) / 256, c.num_sms * 4), 256, 0, c.stream>>>(part, active, nsplit,
                                                                                              n, d_router);
    return cudaGetLastError();
}

}  // namespace pmpe
