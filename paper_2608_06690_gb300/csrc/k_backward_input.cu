// Gradient of the layer's input through the frozen layer (what the layer
// below needs when its own private branch is trained, Sec. 3.2).  For
// L = sum_t dout_t . out_t and the routing the forward took:
//
//   every pick (t, j) of expert e with weight w, its dispatch row r:
//     Z_r = W_down,e^T dout_t,  g, u = W_gate,e h_t, W_up,e h_t (recomputed)
//     dG_r = w Z_r u silu'(g),  dU_r = w Z_r silu(g)
//     dA_r = W_gate,e^T dG_r + W_up,e^T dU_r
//   every shared expert s (weight 1): the same with the token's own row
//   the router of the token's pool (the pool the mask of Sec. 3.1 Eq. 4
//   selects: public for DENY, private for ALLOW): dz = softmax gradient of
//   dL/dw, dh += W_router^T dz
//
//   d_hidden_t = sum_j dA_{r(t, j)} + sum_s dA_{s, t} + sum_e dz_{t, e} W_router,e
//
// Z, [dG | dU] and dA run on the tensor cores (the row launches of
// k_backward_tc.cu over all routed experts, then over the shared experts);
// this file holds the final per-token sum and the launch sequence.
#include <algorithm>
#include <cstring>

#include "pmpe_internal.cuh"

namespace pmpe {
namespace {

constexpr int kPadRows = 128;  // the padded row layout of the row launches

// d_hidden_t in FP32, one CTA per token at a time, each thread 8 columns.
// The sum runs in a fixed order (picks in top-k order, shared experts, the
// pool's router rows), so the result does not depend on scheduling.  The
// padded start of every routed expert's rows is rebuilt per CTA from the
// dispatch offsets.
__global__ void __launch_bounds__(256) bwd_input_reduce_kernel(
    const bf16 *da, const bf16 *da_sh, const float *dz, int ld, const bf16 *router_pub, const bf16 *router_priv,
    const uint8_t *tau, const int32_t *idx, const int32_t *slot_of, const uint32_t *offsets, int T, int H, int E_pub,
    int E_priv, int E_sh, int k, int R, int renorm, int Tp, float *d_hidden)
{
    __shared__ int pad_start[2 * kMaxPool];
    __shared__ int s_carry;
    const int E = E_pub + E_priv;
    const int tid = threadIdx.x, lane = tid & 31;
    pdl_wait();
    // exclusive scan of the padded row counts, 256 experts per pass
    if (tid == 0) s_carry = 0;
    __syncthreads();
    __shared__ int s_warp[8];
    for (int b = 0; b < E; b += blockDim.x) {
        const int e = b + tid;
        int v = 0;
        if (e < E) {
            const int lo = (int)min(offsets[e], (uint32_t)R), hi = (int)min(max(offsets[e + 1], (uint32_t)lo), (uint32_t)R);
            v = (hi - lo + kPadRows - 1) / kPadRows * kPadRows;
        }
        int x = v;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(~0u, x, off);
            if (lane >= off) x += y;
        }
        if (lane == 31) s_warp[tid >> 5] = x;
        __syncthreads();
        int before = s_carry;
        for (int w = 0; w < (tid >> 5); ++w) before += s_warp[w];
        if (e < E) pad_start[e] = before + x - v;
        __syncthreads();
        if (tid == blockDim.x - 1) s_carry = before + x;
        __syncthreads();
    }

    const int nv = H / 8;
    __shared__ int s_row[kMaxTopK];      // padded dA row of each pick (-1: none)
    __shared__ int s_pe[kMaxTopK];       // router row of each pick in the token's pool (-1: none)
    __shared__ float s_dz[kMaxTopK];
    for (int t = blockIdx.x; t < T; t += gridDim.x) {
        const int priv = tau[t] ? 1 : 0;
        const int e_base = priv ? E_pub : 0, E_pool = priv ? E_priv : E_pub;
        const bf16 *router = priv ? router_priv : router_pub;
        const float *dzt = dz + (size_t)t * ld;
        __syncthreads();  // the previous token's picks are consumed
        if (tid < k) {
            const int e = idx[(size_t)t * k + tid];
            const int slot = slot_of[(size_t)t * k + tid];
            const bool ok = e >= 0 && e < E && slot >= 0 && slot < R;
            s_row[tid] = ok ? pad_start[e] + slot - (int)offsets[e] : -1;
            const int pe = e - e_base;
            const bool in_pool = pe >= 0 && pe < E_pool;
            s_pe[tid] = in_pool ? pe : -1;
            s_dz[tid] = in_pool ? dzt[pe] : 0.f;
        }
        __syncthreads();
        for (int c = tid; c < nv; c += blockDim.x) {
            float acc[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = 0.f;
            auto add = [&](const uint4 &v, float scale) {
                const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float2 f = __bfloat1622float2(b[i]);
                    acc[2 * i] += scale * f.x;
                    acc[2 * i + 1] += scale * f.y;
                }
            };
            // the picks' rows are requested 8 at a time before they are summed
            constexpr int kBatch = 8;
            uint4 v[kBatch];
            for (int j0 = 0; j0 < k; j0 += kBatch) {
#pragma unroll
                for (int j = 0; j < kBatch; ++j) {
                    const int r = j0 + j < k ? s_row[j0 + j] : -1;
                    v[j] = r >= 0 ? __ldcs(reinterpret_cast<const uint4 *>(da + (size_t)r * H) + c)
                                  : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int j = 0; j < kBatch; ++j)
                    if (j0 + j < k && s_row[j0 + j] >= 0) add(v[j], 1.f);
            }
            for (int s = 0; s < E_sh; ++s)
                add(__ldcs(reinterpret_cast<const uint4 *>(da_sh + ((size_t)s * Tp + t) * H) + c), 1.f);
            if (renorm) {  // dz is zero outside the token's k picks
                for (int j0 = 0; j0 < k; j0 += kBatch) {
#pragma unroll
                    for (int j = 0; j < kBatch; ++j) {
                        const int pe = j0 + j < k ? s_pe[j0 + j] : -1;
                        v[j] = pe >= 0 ? reinterpret_cast<const uint4 *>(router + (size_t)pe * H)[c]
                                       : make_uint4(0u, 0u, 0u, 0u);
                    }
#pragma unroll
                    for (int j = 0; j < kBatch; ++j)
                        if (j0 + j < k && s_pe[j0 + j] >= 0) add(v[j], s_dz[j0 + j]);
                }
            }  // the pool softmax's dense router term is added afterwards (launch_router_term)
            float4 *o = reinterpret_cast<float4 *>(d_hidden + (size_t)t * H) + 2 * c;
            __stcs(o, make_float4(acc[0], acc[1], acc[2], acc[3]));
            __stcs(o + 1, make_float4(acc[4], acc[5], acc[6], acc[7]));
        }
    }
}

}  // namespace

struct InScratch {
    bf16 *dout_rows, *zpad, *dgu, *da, *zpad_sh, *dgu_sh, *da_sh;
    float *gw_part, *dz;
    int32_t *pool_tok;  // [T] each pool's tokens (pool softmax), then pool_n [2]
    int *pool_n;
    float *logit_part;  // partial pool logits (pool softmax)
    uint64_t rp, rp_sh;  // padded rows: routed, shared
    int tp;              // tokens rounded up to the padded layout (rows of one shared expert)
    size_t bytes;
};

static InScratch input_scratch(const Shape &s, uint8_t *base)
{
    const size_t R = (size_t)s.T * s.k, H = s.H, I = s.I;
    auto al = [](size_t x) { return (x + 255) / 256 * 256; };
    InScratch b;
    b.rp = R + (uint64_t)kPadRows * s.E();
    b.tp = (s.T + kPadRows - 1) / kPadRows * kPadRows;
    b.rp_sh = (uint64_t)s.E_sh * b.tp;
    size_t o = 0;
    b.dout_rows = (bf16 *)(base + o); o += al((R + 64) * H * 2);
    b.zpad = (bf16 *)(base + o);      o += al(b.rp * I * 2);
    b.dgu = (bf16 *)(base + o);       o += al(b.rp * 2 * I * 2);
    b.da = (bf16 *)(base + o);        o += al(b.rp * H * 2);
    b.zpad_sh = (bf16 *)(base + o);   o += al(b.rp_sh * I * 2);
    b.dgu_sh = (bf16 *)(base + o);    o += al(b.rp_sh * 2 * I * 2);
    b.da_sh = (bf16 *)(base + o);     o += al(b.rp_sh * H * 2);
    b.gw_part = (float *)(base + o);  o += al(R * (I / 128) * 4);
    b.dz = (float *)(base + o);       o += al((size_t)s.T * std::max(s.E_pub, s.E_priv) * 4);
    b.pool_tok = (int32_t *)(base + o); o += al((size_t)s.T * 4);
    b.pool_n = (int *)(base + o);     o += al(2 * 4);
    b.logit_part = (float *)(base + o);
    o += al((size_t)router_logit_splits(s) * s.T * std::max(s.E_pub, s.E_priv) * 4);  // whatever the routing
    b.bytes = o;
    return b;
}

// The per-token sum of the picks' dA, the shared experts' dA and the router
// term (dz rows max(E_pub, E_priv) apart): renormalised routing adds the k
// picks' router rows in the same kernel, the pool softmax its dense term in
// a tiled GEMM afterwards.
static cudaError_t launch_input_reduce(const Ctx &c, const InScratch &b, float *d_hidden)
{
    const Shape &s = c.s;
    const int ld = std::max(s.E_pub, s.E_priv);
    const cudaError_t err = launch_pdl(bwd_input_reduce_kernel, dim3(std::min(s.T, c.num_sms * 8)), dim3(256), 0, c.stream,
                      (const bf16 *)b.da, (const bf16 *)b.da_sh, (const float *)b.dz, ld, c.router_pub,
                      c.router_priv, (const uint8_t *)c.tau, (const int32_t *)c.idx, (const int32_t *)c.slot_of,
                      (const uint32_t *)c.offsets, s.T, s.H, s.E_pub, s.E_priv, s.E_sh, s.k, s.T * s.k, s.renorm,
                      b.tp, d_hidden);
    if (err != cudaSuccess || s.renorm) return err;
    return launch_router_term(c, b.dz, ld, b.pool_tok, b.pool_n, d_hidden);
}

size_t backward_input_workspace_bytes(const Shape &s)
{
    if (s.T == 0) return 256;
    return input_scratch(s, nullptr).bytes;
}

cudaError_t launch_backward_input(const Ctx &c, const bf16 *dout, float *d_hidden, uint8_t *bws)
{
    const Shape &s = c.s;
    const int R = s.T * s.k, H = s.H, E = s.E();
    const InScratch b = input_scratch(s, bws);
    cudaStream_t st = c.stream;

    // routed experts: the upstream gradient of every dispatch row, then Z,
    // [dG | dU] (and dL/dw partials) and dA over all E experts
    launch_gather_rows(dout, c.tok_of_slot, c.offsets, 0, E, R, H, b.dout_rows, c.num_sms, st);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    const RowsGroups g{0, E, 0, b.rp};
    if ((err = launch_rows_z(c, g, b.dout_rows, (uint64_t)R + 64, 1, b.zpad)) != cudaSuccess) return err;
    if ((err = launch_rows_gu(c, g, c.a_perm, (uint64_t)R, b.zpad, b.dgu, nullptr, b.gw_part)) != cudaSuccess)
        return err;
    if ((err = launch_rows_da(c, g, b.dgu, b.da)) != cudaSuccess) return err;
    // shared experts: every token's own row, weight 1
    if (s.E_sh > 0) {
        const RowsGroups gs{0, s.E_sh, s.T, b.rp_sh};
        if ((err = launch_rows_z(c, gs, dout, (uint64_t)s.T, 0, b.zpad_sh)) != cudaSuccess) return err;
        if ((err = launch_rows_gu(c, gs, c.hidden, (uint64_t)s.T, b.zpad_sh, b.dgu_sh, nullptr, nullptr)) !=
            cudaSuccess)
            return err;
        if ((err = launch_rows_da(c, gs, b.dgu_sh, b.da_sh)) != cudaSuccess) return err;
    }
    // the router of each token's pool
    const int ld = std::max(s.E_pub, s.E_priv);
    if ((err = launch_router_dz(c, b.gw_part, 1, ld, b.dz, b.pool_tok, b.pool_n, b.logit_part)) != cudaSuccess) return err;
    return launch_input_reduce(c, b, d_hidden);
}

// ------------------------------------------------------------- both

// The private-parameter gradients and the input gradient of one backward from
// a single set of row launches over all routed experts: Z and [dG | dU] of
// the private experts are the same rows either way, so they are computed
// once.  The weight gradients read the private experts' rows in the padded
// layout of all experts; w act is written for the private experts only; the
// router's dz of both pools serves the input gradient and, read as zeros on
// DENY rows, the private router's weight gradient.  Every result is bitwise
// the one the two separate passes give.
struct StepScratch {
    InScratch in;
    bf16 *wact;
    float *part;
    int *active;
    size_t bytes;
};

static StepScratch step_scratch(const Shape &s, uint8_t *base)
{
    auto al = [](size_t x) { return (x + 255) / 256 * 256; };
    StepScratch b;
    b.in = input_scratch(s, base);
    size_t o = b.in.bytes;
    b.wact = (bf16 *)(base + o);   o += al(b.in.rp * s.I * 2);
    b.part = (float *)(base + o);  o += al(router_wgrad_part_bytes(s));
    b.active = (int *)(base + o);  o += al(kMaxRouterSplits * 4);
    b.bytes = o;
    return b;
}

size_t backward_step_workspace_bytes(const Shape &s)
{
    if (s.T == 0) return 256;
    return step_scratch(s, nullptr).bytes;
}

cudaError_t launch_backward_step(const Ctx &c, const bf16 *dout, float *d_router, float *d_gate, float *d_up,
                                 float *d_down, float *d_hidden, uint8_t *bws)
{
    const Shape &s = c.s;
    const int R = s.T * s.k, H = s.H, E = s.E();
    const StepScratch st = step_scratch(s, bws);
    const InScratch &b = st.in;
    cudaStream_t stream = c.stream;

    launch_gather_rows(dout, c.tok_of_slot, c.offsets, 0, E, R, H, b.dout_rows, c.num_sms, stream);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    const RowsGroups g{0, E, 0, b.rp};
    if ((err = launch_rows_z(c, g, b.dout_rows, (uint64_t)R + 64, 1, b.zpad)) != cudaSuccess) return err;
    if ((err = launch_rows_gu(c, g, c.a_perm, (uint64_t)R, b.zpad, b.dgu, st.wact, b.gw_part)) != cudaSuccess)
        return err;
    if ((err = launch_rows_da(c, g, b.dgu, b.da)) != cudaSuccess) return err;
    if (s.E_sh > 0) {
        const RowsGroups gs{0, s.E_sh, s.T, b.rp_sh};
        if ((err = launch_rows_z(c, gs, dout, (uint64_t)s.T, 0, b.zpad_sh)) != cudaSuccess) return err;
        if ((err = launch_rows_gu(c, gs, c.hidden, (uint64_t)s.T, b.zpad_sh, b.dgu_sh, nullptr, nullptr)) !=
            cudaSuccess)
            return err;
        if ((err = launch_rows_da(c, gs, b.dgu_sh, b.da_sh)) != cudaSuccess) return err;
    }
    const int ld = std::max(s.E_pub, s.E_priv);
    if ((err = launch_router_dz(c, b.gw_part, 1, ld, b.dz, b.pool_tok, b.pool_n, b.logit_part)) != cudaSuccess) return err;
    if ((err = launch_router_wgrad(c, b.dz, ld, st.part, st.active, d_router)) != cudaSuccess) return err;
    if ((err = launch_backward_wgrad(c, b.dout_rows, b.dgu, st.wact, d_gate, d_up, d_down, &g)) != cudaSuccess)
        return err;
    return launch_input_reduce(c, b, d_hidden);
}

}  // namespace pmpe
