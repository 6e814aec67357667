// Backward of the private branch (G2, Sec. 2.2 and Sec. 3.2: only the private
// experts and the private router are trained; the public parameters are frozen
// and get no gradient).  For L = sum_t dout_t . out_t and the routing the
// forward took (read from the forward's workspace):
//
//   private expert q, its dispatch rows r (tokens t, weights w):
//     Z_r   = W_down,q^T dout_t           (so dL/dw_r = Z_r . a_r, da_r = w_r Z_r)
//     g, u  = W_gate,q h_t, W_up,q h_t    (recomputed)
//     dG_r  = w_r Z_r u silu'(g),  dU_r = w_r Z_r silu(g)
//     dW_gate,q = sum_r dG_r h_t^T,  dW_up,q = sum_r dU_r h_t^T,  dW_down,q = sum_r (w_r dout_t) a_r^T
//   router, per ALLOW token (softmax over the private pool, renormalised over
//   the top-k or not):  dz = softmax gradient of dL/dw,  dW_router,e = sum_t dz_{t,e} h_t^T
//
// The contractions run on one grouped GEMM kernel on the BF16 tensor cores
// (mma.sync m16n8k16, FP32 accumulate): a group is a private expert whose row
// range comes from the dispatch offsets on the device, either as the M
// dimension (Z, G, U) or as the contracted K dimension (the weight gradients).
// Operands stored with M or N contiguous are loaded with ldmatrix.trans, so no
// operand is transposed in memory; rows past a group's range read as zeros.
#include <algorithm>
#include <cstring>

#include "pmpe_internal.cuh"

namespace pmpe {
namespace {

constexpr int kBM = 128, kBN = 128, kBK = 32;
constexpr int kGThreads = 256;  // 8 warps: 2 (M) x 4 (N), each 64 x 32
constexpr int kPad = 8;         // BF16 elements of row padding: conflict-free ldmatrix rows

// One operand of a grouped GEMM: element (i, j) of group q (i = M or N index,
// j = K index) is  p[base + i * ld + j]  (K contiguous)  or  p[base + j * ld + i]
// (trans: M / N contiguous), with  base = q * q_stride + row0 * ld  and row0
// the group's first dispatch row (plus the first private slot when add_p0)
// when the operand is indexed by dispatch rows (rows = 1), else 0.
struct Operand {
    const bf16 *p;
    int ld;
    long long q_stride;
    int rows;    // 1: the grouped row range indexes this operand's stored rows
    int add_p0;  // 1: stored rows are dispatch slots (offset by the first private slot)
};

enum { kGroupM = 0, kGroupK = 1 };

struct GemmBwdParams {
    int group_dim;   // kGroupM: M = the group's rows; kGroupK: K = the group's rows
    int M, N, K;     // the fixed dimensions (the grouped one is ignored)
    int E_pub, E_priv, R;
    const uint32_t *offsets;  // forward dispatch offsets [E + 1]
    Operand A, B;
    float *C;                 // FP32 output
    int ldc;
    long long c_q_stride;
    int c_rows, c_add_p0;     // as for operands: the output's rows follow the group's row range
};

struct GroupInfo {
    int rows, row0;  // rows of private expert q and its first dispatch row, relative to the first private slot
};

__device__ __forceinline__ GroupInfo group_of(const GemmBwdParams &p, int q)
{
    const uint32_t p0 = p.offsets[p.E_pub];
    const int b = min((int)p.offsets[p.E_pub + q], p.R), e = min(max((int)p.offsets[p.E_pub + q + 1], b), p.R);
    GroupInfo gi;
    gi.rows = e - b;
    gi.row0 = b - (int)min(p0, (uint32_t)p.R);
    return gi;
}

__device__ __forceinline__ long long op_base(const Operand &o, int q, int row0, int p0)
{
    return (long long)q * o.q_stride + (o.rows ? (long long)(row0 + (o.add_p0 ? p0 : 0)) * o.ld : 0);
}

// Load a 128 x 32 (i, j) operand tile into shared memory.  K-contiguous
// operands land as [128][kBK + kPad] (row = i), trans operands as
// [kBK][128 + kPad] (row = j).  Elements outside [0, ni) x [0, nj) read zero.
template <bool kTrans>
__device__ __forceinline__ void load_tile(uint32_t sdst, const bf16 *src, int ld, int i0, int j0, int ni, int nj)
{
    const int tid = threadIdx.x;
    if (!kTrans) {
        // 128 rows x 4 chunks of 8
#pragma unroll
        for (int c = tid; c < 128 * 4; c += kGThreads) {
            const int i = c >> 2, jc = (c & 3) * 8;
            const bool ok = (i0 + i) < ni && (j0 + jc) < nj;
            const bf16 *g = ok ? src + (long long)(i0 + i) * ld + j0 + jc : src;
            cp_async16(sdst + (uint32_t)(i * (kBK + kPad) + jc) * 2u, g, ok ? 16 : 0);
        }
    } else {
        // 32 rows (j) x 16 chunks of 8 (i)
#pragma unroll
        for (int c = tid; c < kBK * 16; c += kGThreads) {
            const int j = c >> 4, ic = (c & 15) * 8;
            const bool ok = (j0 + j) < nj && (i0 + ic) < ni;
            const bf16 *g = ok ? src + (long long)(j0 + j) * ld + i0 + ic : src;
            cp_async16(sdst + (uint32_t)(j * (128 + kPad) + ic) * 2u, g, ok ? 16 : 0);
        }
    }
}

__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3, uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// A fragment (16 rows of M x 16 of K) at (m, k) of the A tile.
template <bool kTrans>
__device__ __forceinline__ void frag_a(uint32_t *a, uint32_t s, int m, int k)
{
    const int lane = threadIdx.x & 31;
    if (!kTrans) {
        const int row = m + (lane & 15), col = k + (lane >> 4) * 8;
        ldmatrix_x4(a[0], a[1], a[2], a[3], s + (uint32_t)(row * (kBK + kPad) + col) * 2u);
    } else {
        // matrices: (m 0-7, k 0-7), (m 8-15, k 0-7), (m 0-7, k 8-15), (m 8-15, k 8-15)
        const int mi = lane >> 3, rr = lane & 7;
        const int kk = k + (mi >> 1) * 8 + rr, mm = m + (mi & 1) * 8;
        ldmatrix_x4_trans(a[0], a[1], a[2], a[3], s + (uint32_t)(kk * (128 + kPad) + mm) * 2u);
    }
}

// B fragments for two n8 blocks (n, n + 8) x 16 of K at (n, k) of the B tile:
// b[0], b[1] for block n, b[2], b[3] for block n + 8.
template <bool kTrans>
__device__ __forceinline__ void frag_b(uint32_t *b, uint32_t s, int n, int k)
{
    const int lane = threadIdx.x & 31;
    const int mi = lane >> 3, rr = lane & 7;
    // matrices: (n 0-7, k 0-7), (n 0-7, k 8-15), (n 8-15, k 0-7), (n 8-15, k 8-15)
    const int nn = n + (mi >> 1) * 8, kk = k + (mi & 1) * 8;
    if (!kTrans) {
        ldmatrix_x4(b[0], b[1], b[2], b[3], s + (uint32_t)((nn + rr) * (kBK + kPad) + kk) * 2u);
    } else {
        ldmatrix_x4_trans(b[0], b[1], b[2], b[3], s + (uint32_t)((kk + rr) * (128 + kPad) + nn) * 2u);
    }
}

template <bool kTA, bool kTB>
__global__ void __launch_bounds__(kGThreads) grouped_gemm_bwd_kernel(const GemmBwdParams p)
{
    constexpr int kATileBytes = (kTA ? kBK * (128 + kPad) : 128 * (kBK + kPad)) * 2;
    constexpr int kBTileBytes = (kTB ? kBK * (128 + kPad) : 128 * (kBK + kPad)) * 2;
    __shared__ __align__(128) uint8_t smem[2 * (kATileBytes + kBTileBytes)];
    __shared__ int s_prefix[kMaxPool + 1];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wm = warp >> 2, wn = warp & 3;  // warp tile: rows wm*64, cols wn*32
    const uint32_t p0 = min(p.offsets[p.E_pub], (uint32_t)p.R);

    // tile list over the private experts
    if (threadIdx.x == 0) {
        int acc = 0;
        s_prefix[0] = 0;
        for (int q = 0; q < p.E_priv; ++q) {
            const GroupInfo gi = group_of(p, q);
            const int M = p.group_dim == kGroupM ? gi.rows : p.M;
            const int K = p.group_dim == kGroupK ? gi.rows : p.K;
            // a K-grouped GEMM writes every expert's output (zeros for an expert
            // without rows); an M-grouped one has no tile for an empty expert
            const bool any = p.group_dim == kGroupK || gi.rows > 0;
            const int tiles = (any && M > 0 && K >= 0) ? ((M + kBM - 1) / kBM) * ((p.N + kBN - 1) / kBN) : 0;
            acc += tiles;
            s_prefix[q + 1] = acc;
        }
    }
    __syncthreads();
    const int total = s_prefix[p.E_priv];
    const uint32_t sbase = smem_u32(smem);

    for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
        int q = 0;
        while (s_prefix[q + 1] <= tile) ++q;
        const GroupInfo gi = group_of(p, q);
        const int M = p.group_dim == kGroupM ? gi.rows : p.M;
        const int K = p.group_dim == kGroupK ? gi.rows : p.K;
        const int nt = (p.N + kBN - 1) / kBN;
        const int local = tile - s_prefix[q];
        const int m0 = (local / nt) * kBM, n0 = (local % nt) * kBN;
        const bf16 *A = p.A.p + op_base(p.A, q, gi.row0, (int)p0);
        const bf16 *B = p.B.p + op_base(p.B, q, gi.row0, (int)p0);

        float acc[4][4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b)
#pragma unroll
                for (int c = 0; c < 4; ++c) acc[a][b][c] = 0.f;

        const int nk = (K + kBK - 1) / kBK;
        auto stage_a = [&](int s) { return sbase + (uint32_t)(s * (kATileBytes + kBTileBytes)); };
        auto stage_b = [&](int s) { return stage_a(s) + (uint32_t)kATileBytes; };
        __syncthreads();  // the previous tile's reads of the buffers are done
        if (nk > 0) {
            load_tile<kTA>(stage_a(0), A, p.A.ld, m0, 0, M, K);
            load_tile<kTB>(stage_b(0), B, p.B.ld, n0, 0, p.N, K);
        }
        cp_async_commit();
        for (int kt = 0; kt < nk; ++kt) {
            const int s = kt & 1;
            if (kt + 1 < nk) {
                load_tile<kTA>(stage_a(s ^ 1), A, p.A.ld, m0, (kt + 1) * kBK, M, K);
                load_tile<kTB>(stage_b(s ^ 1), B, p.B.ld, n0, (kt + 1) * kBK, p.N, K);
            }
            cp_async_commit();
            cp_async_wait<1>();
            __syncthreads();
#pragma unroll
            for (int kk = 0; kk < kBK; kk += 16) {
                uint32_t af[4][4], bfr[2][4];
#pragma unroll
                for (int im = 0; im < 4; ++im) frag_a<kTA>(af[im], stage_a(s), wm * 64 + im * 16, kk);
#pragma unroll
                for (int jn = 0; jn < 2; ++jn) frag_b<kTB>(bfr[jn], stage_b(s), wn * 32 + jn * 16, kk);
#pragma unroll
                for (int im = 0; im < 4; ++im)
#pragma unroll
                    for (int jn = 0; jn < 2; ++jn) {
                        mma_bf16_16816(acc[im][jn * 2], af[im], bfr[jn][0], bfr[jn][1]);
                        mma_bf16_16816(acc[im][jn * 2 + 1], af[im], bfr[jn][2], bfr[jn][3]);
                    }
            }
            __syncthreads();
        }
        cp_async_wait<0>();
        // FP32 store of the tile (fragment layout: rows lane/4 and +8, cols (lane%4)*2 and +1)
        float *C = p.C + (long long)q * p.c_q_stride +
                   (p.c_rows ? (long long)(gi.row0 + (p.c_add_p0 ? (int)p0 : 0)) * p.ldc : 0);
#pragma unroll
        for (int im = 0; im < 4; ++im)
#pragma unroll
            for (int jn = 0; jn < 4; ++jn) {
                const int r = m0 + wm * 64 + im * 16 + (lane >> 2);
                const int c = n0 + wn * 32 + jn * 8 + (lane & 3) * 2;
                if (c < p.N) {
                    if (r < M) *reinterpret_cast<float2 *>(C + (long long)r * p.ldc + c) =
                                   make_float2(acc[im][jn][0], acc[im][jn][1]);
                    if (r + 8 < M) *reinterpret_cast<float2 *>(C + (long long)(r + 8) * p.ldc + c) =
                                       make_float2(acc[im][jn][2], acc[im][jn][3]);
                }
            }
    }
}

// Private dispatch rows: the upstream gradient of each row's token, and the
// same scaled by the row's routing weight (the down projection's gradient).
__global__ void bwd_gather_kernel(const bf16 *dout, const int32_t *tok_of_slot, const float *w_of_slot,
                                  const uint32_t *offsets, int E_pub, int E, int R, int H, bf16 *dout_rows,
                                  bf16 *dy_rows)
{
    const uint32_t p0 = min(offsets[E_pub], (uint32_t)R), p1 = min(max(offsets[E], p0), (uint32_t)R);
    const int nv = H / 8;
    const long long total = (long long)(p1 - p0) * nv;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int r = (int)(i / nv), c = (int)(i - (long long)r * nv);
        const int slot = (int)p0 + r;
        const int t = tok_of_slot[slot];
        const float w = w_of_slot[slot];
        const uint4 v = reinterpret_cast<const uint4 *>(dout + (size_t)t * H)[c];
        reinterpret_cast<uint4 *>(dout_rows + (size_t)r * H)[c] = v;
        const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&v);
        uint4 o;
        uint32_t *po = reinterpret_cast<uint32_t *>(&o);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 f = __bfloat1622float2(b[k]);
            po[k] = pack_bf16x2(w * f.x, w * f.y);
        }
        reinterpret_cast<uint4 *>(dy_rows + (size_t)r * H)[c] = o;
    }
}

// Per private row (one warp): dL/dw = Z . a, and through SwiGLU
// dG = w Z u silu'(g), dU = w Z silu(g) (BF16 operands of the weight gradients).
__global__ void bwd_swiglu_kernel(const float *Z, const float *G, const float *U, const bf16 *act,
                                  const float *w_of_slot, const uint32_t *offsets, int E_pub, int E, int R, int I,
                                  float *gw, bf16 *dG, bf16 *dU)
{
    const uint32_t p0 = min(offsets[E_pub], (uint32_t)R), p1 = min(max(offsets[E], p0), (uint32_t)R);
    const int lane = threadIdx.x & 31;
    const int warps = gridDim.x * (blockDim.x >> 5);
    for (int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < (int)(p1 - p0); r += warps) {
        const int slot = (int)p0 + r;
        const float w = w_of_slot[slot];
        float dot = 0.f;
        for (int i = lane; i < I; i += 32) {
            const size_t o = (size_t)r * I + i;
            const float z = Z[o], g = G[o], u = U[o];
            dot += z * __bfloat162float(act[(size_t)slot * I + i]);
            const float sg = 1.f / (1.f + expf(-g));
            const float da = w * z;
            dG[o] = __float2bfloat16_rn(da * u * sg * (1.f + g * (1.f - sg)));
            dU[o] = __float2bfloat16_rn(da * g * sg);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(~0u, dot, off);
        if (lane == 0) gw[r] = dot;
    }
}

// Router gradient per ALLOW token (one warp): the softmax gradient dz over the
// private pool from dL/dw of its k rows -- renormalised over the top-k, or the
// pool softmax, whose probabilities need every private logit, recomputed here
// in FP32 from the BF16 operands.  dz [T][E_priv] (zero for DENY tokens).
__global__ void bwd_router_kernel(const bf16 *hidden, const bf16 *router_priv, const uint8_t *tau,
                                  const int32_t *idx, const float *wts, const int32_t *slot_of, const float *gw,
                                  const uint32_t *offsets, int T, int H, int E_pub, int E_priv, int k, int renorm,
                                  int R, float *dz)
{
    const uint32_t p0 = min(offsets[E_pub], (uint32_t)R);
    const int lane = threadIdx.x & 31;
    const int warps = gridDim.x * (blockDim.x >> 5);
    for (int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); t < T; t += warps) {
        float *dzt = dz + (size_t)t * E_priv;
        if (!tau[t]) {
            for (int e = lane; e < E_priv; e += 32) dzt[e] = 0.f;
            continue;
        }
        // lane j < k holds pick j: its pool id and dL/dw
        int pe = -1;
        float g = 0.f, wj = 0.f;
        if (lane < k) {
            pe = idx[(size_t)t * k + lane] - E_pub;
            const int slot = slot_of[(size_t)t * k + lane];
            g = gw[slot - (int)p0];
            wj = wts[(size_t)t * k + lane];
        }
        float sum = wj * g;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(~0u, sum, off);
        if (renorm) {
            for (int e = lane; e < E_priv; e += 32) dzt[e] = 0.f;
            __syncwarp();
            if (lane < k && pe >= 0 && pe < E_priv) dzt[pe] = wj * (g - sum);
        } else {
            // pool softmax over the private experts: logits of this token
            const bf16 *h = hidden + (size_t)t * H;
            for (int e0 = 0; e0 < E_priv; e0 += 32) {
                const int e = e0 + lane;
                float z = -INFINITY;
                if (e < E_priv) {
                    const bf16 *wr = router_priv + (size_t)e * H;
                    float a = 0.f;
                    for (int c = 0; c < H; c += 8) {
                        const uint4 hv = *reinterpret_cast<const uint4 *>(h + c);
                        const uint4 rv = *reinterpret_cast<const uint4 *>(wr + c);
                        const __nv_bfloat162 *hb = reinterpret_cast<const __nv_bfloat162 *>(&hv);
                        const __nv_bfloat162 *rb = reinterpret_cast<const __nv_bfloat162 *>(&rv);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float2 x = __bfloat1622float2(hb[q]), y = __bfloat1622float2(rb[q]);
                            a += x.x * y.x + x.y * y.y;
                        }
                    }
                    z = a;
                }
                if (e < E_priv) dzt[e] = z;  // logits parked in dz, finished below
            }
            __syncwarp();
            float mx = -INFINITY;
            for (int e = lane; e < E_priv; e += 32) mx = fmaxf(mx, dzt[e]);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(~0u, mx, off));
            float den = 0.f;
            for (int e = lane; e < E_priv; e += 32) den += expf(dzt[e] - mx);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(~0u, den, off);
            __syncwarp();
            // dz_e = p_e (dL/dp_e - sum): -p_e sum everywhere, plus p_e dL/dw_j at the k picks
            float pj = 0.f;
            if (lane < k && pe >= 0 && pe < E_priv) pj = expf(dzt[pe] - mx) / den;
            __syncwarp();
            for (int e = lane; e < E_priv; e += 32) dzt[e] = -(expf(dzt[e] - mx) / den) * sum;
            __syncwarp();
            if (lane < k && pe >= 0 && pe < E_priv) dzt[pe] += pj * g;
        }
        __syncwarp();
    }
}

// dW_router[e][c] = sum_t dz[t][e] h[t][c] in FP32, split over the tokens:
// CTA (x, y, z) owns a 32 x 128 output tile and the z-th token range, staged
// through shared memory 32 tokens at a time, and writes its partial sum to
// part[z]; bwd_router_reduce_kernel adds the partials in split order, so the
// result does not depend on scheduling.
__global__ void __launch_bounds__(256) bwd_router_wgrad_kernel(const float *dz, const bf16 *hidden, int T, int H,
                                                               int E_priv, int tok_per_split, float *part)
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
    for (int t0 = t_begin; t0 < t_end; t0 += 32) {
        for (int i = threadIdx.x; i < 32 * 32; i += 256) {
            const int tt = i >> 5, ee = i & 31;
            s_dz[tt][ee] = (t0 + tt < t_end && e0 + ee < E_priv) ? dz[(size_t)(t0 + tt) * E_priv + e0 + ee] : 0.f;
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
    float *out = part + (size_t)blockIdx.z * E_priv * H;
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int e = e0 + ty + 8 * a, c = c0 + tx + 32 * b;
            if (e < E_priv && c < H) out[(size_t)e * H + c] = acc[a][b];
        }
}

__global__ void bwd_router_reduce_kernel(const float *part, int nsplit, int n, float *d_router)
{
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        float a = 0.f;
        for (int z = 0; z < nsplit; ++z) a += part[(size_t)z * n + i];
        d_router[i] = a;
    }
}

// Token splits of the router weight gradient: enough CTAs for two per SM,
// each range a multiple of 32 tokens, at most kMaxRouterSplits ranges.
constexpr int kMaxRouterSplits = 64;
int router_splits(const Shape &s, int num_sms, int *tok_per_split)
{
    const int tiles = ((s.H + 127) / 128) * ((s.E_priv + 31) / 32);
    const int chunks = std::max(1, (s.T + 31) / 32);
    int n = std::min(std::min(kMaxRouterSplits, chunks), std::max(1, (2 * num_sms + tiles - 1) / tiles));
    const int per = ((chunks + n - 1) / n) * 32;
    n = std::max(1, (s.T + per - 1) / per);
    *tok_per_split = per;
    return n;
}

template <bool kTA, bool kTB>
cudaError_t launch_gemm_bwd(const GemmBwdParams &p, int num_sms, cudaStream_t st)
{
    grouped_gemm_bwd_kernel<kTA, kTB><<<num_sms * 2, kGThreads, 0, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

size_t backward_workspace_bytes(const Shape &s)
{
    const size_t R = (size_t)s.T * s.k, H = s.H, I = s.I;
    auto al = [](size_t x) { return (x + 255) / 256 * 256; };
    if (s.T == 0) return 256;
    const size_t splits = (size_t)std::min(kMaxRouterSplits, (s.T + 31) / 32);
    const size_t n = al(R * H * 2) * 2 + al(R * I * 4) * 3 + al(R * I * 2) * 2 + al(R * 4) +
                     al((size_t)s.T * s.E_priv * 4) + al(splits * s.E_priv * H * 4);
    return n < 256 ? 256 : n;
}

cudaError_t launch_backward_private(const Ctx &c, const bf16 *dout, float *d_router, float *d_gate, float *d_up,
                                    float *d_down, uint8_t *bws)
{
    const Shape &s = c.s;
    const int R = s.T * s.k, H = s.H, I = s.I;
    auto al = [](size_t x) { return (x + 255) / 256 * 256; };
    uint8_t *q = bws;
    bf16 *dout_rows = (bf16 *)q; q += al((size_t)R * H * 2);
    bf16 *dy_rows = (bf16 *)q;   q += al((size_t)R * H * 2);
    float *Z = (float *)q;       q += al((size_t)R * I * 4);
    float *G = (float *)q;       q += al((size_t)R * I * 4);
    float *U = (float *)q;       q += al((size_t)R * I * 4);
    bf16 *dG = (bf16 *)q;        q += al((size_t)R * I * 2);
    bf16 *dU = (bf16 *)q;        q += al((size_t)R * I * 2);
    float *gw = (float *)q;      q += al((size_t)R * 4);
    float *dz = (float *)q;      q += al((size_t)s.T * s.E_priv * 4);
    float *part = (float *)q;
    const int E = s.E();
    cudaStream_t st = c.stream;

    bwd_gather_kernel<<<c.num_sms * 8, 256, 0, st>>>(dout, c.tok_of_slot, c.w_of_slot, c.offsets, s.E_pub, E, R, H,
                                                     dout_rows, dy_rows);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;

    GemmBwdParams p;
    memset(&p, 0, sizeof(p));
    p.E_pub = s.E_pub; p.E_priv = s.E_priv; p.R = R; p.offsets = c.offsets;
    // Z[r][i] = sum_h dout_rows[r][h] W_down[q][h][i]
    p.group_dim = kGroupM; p.N = I; p.K = H;
    p.A = {dout_rows, H, 0, 1, 0};
    p.B = {c.down[1], I, (long long)H * I, 0, 0};
    p.C = Z; p.ldc = I; p.c_q_stride = 0; p.c_rows = 1; p.c_add_p0 = 0;
    if ((err = launch_gemm_bwd<false, true>(p, c.num_sms, st)) != cudaSuccess) return err;
    // G, U [r][i] = sum_h a_perm[slot][h] W_gate / W_up[q][i][h]
    p.N = I; p.K = H;
    p.A = {c.a_perm, H, 0, 1, 1};
    p.B = {c.gate[1], H, (long long)I * H, 0, 0};
    p.C = G;
    if ((err = launch_gemm_bwd<false, false>(p, c.num_sms, st)) != cudaSuccess) return err;
    p.B = {c.up[1], H, (long long)I * H, 0, 0};
    p.C = U;
    if ((err = launch_gemm_bwd<false, false>(p, c.num_sms, st)) != cudaSuccess) return err;

    bwd_swiglu_kernel<<<c.num_sms * 8, 256, 0, st>>>(Z, G, U, c.act, c.w_of_slot, c.offsets, s.E_pub, E, R, I, gw, dG,
                                                     dU);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;

    // weight gradients: contraction over the expert's rows (K = the group's rows)
    p.group_dim = kGroupK; p.c_rows = 0; p.c_add_p0 = 0;
    // dW_gate[q][i][h] = sum_r dG[r][i] a_perm[slot][h]
    p.M = I; p.N = H;
    p.A = {dG, I, 0, 1, 0};
    p.B = {c.a_perm, H, 0, 1, 1};
    p.C = d_gate; p.ldc = H; p.c_q_stride = (long long)I * H;
    if ((err = launch_gemm_bwd<true, true>(p, c.num_sms, st)) != cudaSuccess) return err;
    p.A = {dU, I, 0, 1, 0};
    p.C = d_up;
    if ((err = launch_gemm_bwd<true, true>(p, c.num_sms, st)) != cudaSuccess) return err;
    // dW_down[q][h][i] = sum_r dy_rows[r][h] act[slot][i]
    p.M = H; p.N = I;
    p.A = {dy_rows, H, 0, 1, 0};
    p.B = {c.act, I, 0, 1, 1};
    p.C = d_down; p.ldc = I; p.c_q_stride = (long long)H * I;
    if ((err = launch_gemm_bwd<true, true>(p, c.num_sms, st)) != cudaSuccess) return err;

    // router
    bwd_router_kernel<<<c.num_sms * 4, 256, 0, st>>>(c.hidden, c.router_priv, c.tau, c.idx, c.w, c.slot_of, gw,
                                                     c.offsets, s.T, H, s.E_pub, s.E_priv, s.k, s.renorm, R, dz);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    int per = 32;
    const int nsplit = router_splits(s, c.num_sms, &per);
    dim3 grid((H + 127) / 128, (s.E_priv + 31) / 32, nsplit);
    bwd_router_wgrad_kernel<<<grid, 256, 0, st>>>(dz, c.hidden, s.T, H, s.E_priv, per, part);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    const int n = s.E_priv * H;
    bwd_router_reduce_kernel<<<std::min((n + 255) / 256, c.num_sms * 4), 256, 0, st>>>(part, nsplit, n, d_router);
    return cudaGetLastError();
}

}  // namespace pmpe
