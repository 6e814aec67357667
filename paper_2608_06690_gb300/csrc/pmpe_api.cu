// Host side of the C ABI declared in include/pmpe.h: argument validation,
// the workspace carve-up, stage dispatch and the bounded audit read.
#include <algorithm>
#include <chrono>
#include <thread>

#include "pmpe_internal.cuh"

namespace pmpe {

static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Each routed group adds at most one partial 128-row block beyond R/128; the
// shared-expert group covers the T tokens.  The last two words are the expert
// kernel's tile counter (the next tile of its list to hand out) and its grid
// barrier counter.
size_t gemm_ready_words(const Shape &s)
{
    const size_t R = (size_t)s.T * (size_t)s.k;
    return (R + 127) / 128 + (size_t)s.E() + ((size_t)s.T + 127) / 128 + 6;
}

static bool shape_ok(const Shape &s)
{
    return s.T >= 0 && s.H > 0 && s.I > 0 && s.k >= 1 && s.k <= kMaxTopK && s.E_pub >= s.k && s.E_priv >= s.k &&
           s.E_pub <= kMaxPool && s.E_priv <= kMaxPool && s.E_sh >= 0 && s.E_sh <= kMaxPool &&
           s.H % kDimAlign == 0 && s.I % kDimAlign == 0;
}

int compute_layout(const Shape &s, pmpe_workspace_layout *L)
{
    if (!shape_ok(s)) return PMPE_ERR_INVALID_ARG;
    const size_t T = (size_t)s.T, E = (size_t)s.E(), R = T * (size_t)s.k;
    size_t o = 0;
    auto take = [&](size_t bytes, size_t align) {
        o = align_up(o, align);
        const size_t at = o;
        o += bytes;
        return at;
    };
    L->tau = take(T, 256);
    L->counts = take(4 * E, 256);
    const size_t slots = (size_t)router_slots(s.T);
    const size_t rctas = slots * (size_t)std::max(router_chunks(s.E_pub), router_chunks(s.E_priv));
    const size_t rctas_all = slots * (size_t)(router_chunks(s.E_pub) + router_chunks(s.E_priv));
    L->tile_done = take(4 * slots, 4);
    L->gemm_ready = take(4 * gemm_ready_words(s), 4);
    L->tile_counts = take(4 * E * (size_t)router_slots4(s.T), 16);  // read as 16-byte vectors
    L->offsets = take(4 * (E + 1), 256);
    L->topk_idx = take(4 * R, 256);
    L->topk_w = take(4 * R, 256);
    L->slot_of = take(4 * R, 256);
    L->ticket = take(4 * R, 256);
    L->tok_of_slot = take(4 * R, 256);
    L->w_of_slot = take(4 * R, 256);
    L->router_lists = take(8 * rctas_all * 128 * (size_t)s.k, 256);
    L->router_meta = take(16 * rctas_all * 128, 256);
    L->router_rows = take(2 * rctas * 128 * (size_t)s.H, 1024);
    L->a_perm = take(2 * R * s.H, 1024);
    L->act = take(2 * R * s.I, 1024);
    L->y = take(2 * R * s.H, 1024);
    L->act_sh = s.E_sh > 0 ? take(2 * T * s.E_sh * s.I, 1024) : 0;
    L->y_sh = s.E_sh > 0 ? take(2 * T * s.H, 1024) : 0;
    L->total = align_up(o, 1024);
    return PMPE_OK;
}

Audit audit_ptrs(uint32_t *a, int T, int E)
{
    Audit r;
    if (!a) {
        r.status = r.shared_rows = r.route_count = r.exec_rows = r.exec_tiles = r.route_priv_rows = r.exec_priv_rows =
            nullptr;
        return r;
    }
    r.status = a;
    r.shared_rows = a + 1;
    r.route_count = a + 2;
    r.exec_rows = a + 2 + E;
    r.exec_tiles = a + 2 + 2 * E;
    r.route_priv_rows = a + 2 + 3 * E;
    r.exec_priv_rows = a + 2 + 3 * E + T;
    return r;
}

static bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

static Shape shape_of(const pmpe_moe_desc *d)
{
    Shape s;
    s.T = d->T; s.H = d->H; s.I = d->I; s.E_pub = d->E_pub; s.E_priv = d->E_priv; s.E_sh = d->E_shared;
    s.k = d->k; s.renorm = d->renormalize ? 1 : 0;
    return s;
}

// Validate the descriptor and resolve it into a launch context.
static int make_ctx(const pmpe_moe_desc *d, void *stream, Ctx *c)
{
    if (!d) return PMPE_ERR_INVALID_ARG;
    const Shape s = shape_of(d);
    if (s.T < 0 || s.k < 1 || s.k > s.E_pub || s.k > s.E_priv || s.E_sh < 0) return PMPE_ERR_INVALID_ARG;
    if (!shape_ok(s)) return PMPE_ERR_UNSUPPORTED_SHAPE;
    const void *required[] = {d->hidden, d->w_router_pub, d->w_router_priv, d->w_gate_pub, d->w_up_pub,
                              d->w_down_pub, d->w_gate_priv, d->w_up_priv, d->w_down_priv, d->out};
    for (const void *q : required)
        if (!q && s.T > 0) return PMPE_ERR_INVALID_ARG;
    if (s.E_sh > 0 && (!d->w_gate_sh || !d->w_up_sh || !d->w_down_sh)) return PMPE_ERR_INVALID_ARG;
    if (d->unmasked_control != 0 && d->unmasked_control != 1) return PMPE_ERR_INVALID_ARG;
    if (d->unmasked_control) {
        const int nall = router_chunks(s.E_pub) + router_chunks(s.E_priv);
        if (nall > 16 || nall * s.k > 96) return PMPE_ERR_UNSUPPORTED_SHAPE;
    }
    const void *all[] = {d->hidden, d->w_router_pub, d->w_router_priv, d->w_gate_pub, d->w_up_pub, d->w_down_pub,
                         d->w_gate_priv, d->w_up_priv, d->w_down_priv, d->w_gate_sh, d->w_up_sh, d->w_down_sh,
                         d->out, d->topk_idx, d->topk_w, d->audit, d->workspace, d->saved_gu};
    for (const void *q : all)
        if (!aligned16(q)) return PMPE_ERR_UNSUPPORTED_SHAPE;
    pmpe_workspace_layout L;
    compute_layout(s, &L);
    if (s.T > 0 && (!d->workspace || d->workspace_bytes < L.total || ((uintptr_t)d->workspace & 255u)))
        return PMPE_ERR_WORKSPACE;

    c->s = s;
    c->hidden = (const bf16 *)d->hidden;
    c->policy = d->policy;
    c->router_pub = (const bf16 *)d->w_router_pub;
    c->router_priv = (const bf16 *)d->w_router_priv;
    c->gate[0] = (const bf16 *)d->w_gate_pub; c->up[0] = (const bf16 *)d->w_up_pub; c->down[0] = (const bf16 *)d->w_down_pub;
    c->gate[1] = (const bf16 *)d->w_gate_priv; c->up[1] = (const bf16 *)d->w_up_priv; c->down[1] = (const bf16 *)d->w_down_priv;
    c->gate[2] = (const bf16 *)d->w_gate_sh; c->up[2] = (const bf16 *)d->w_up_sh; c->down[2] = (const bf16 *)d->w_down_sh;
    c->out = (bf16 *)d->out;
    uint8_t *ws = (uint8_t *)d->workspace;
    c->idx = d->topk_idx ? d->topk_idx : (int32_t *)(ws + L.topk_idx);
    c->w = d->topk_w ? d->topk_w : (float *)(ws + L.topk_w);
    c->audit = audit_ptrs(d->audit, s.T, s.E());
    c->tau = ws + L.tau;
    c->counts = (uint32_t *)(ws + L.counts);
    c->offsets = (uint32_t *)(ws + L.offsets);
    c->slot_of = (int32_t *)(ws + L.slot_of);
    c->ticket = (int32_t *)(ws + L.ticket);
    c->tok_of_slot = (int32_t *)(ws + L.tok_of_slot);
    c->w_of_slot = (float *)(ws + L.w_of_slot);
    c->tile_done = (uint32_t *)(ws + L.tile_done);
    c->tile_counts = (uint32_t *)(ws + L.tile_counts);
    c->gemm_ready = (uint32_t *)(ws + L.gemm_ready);
    c->router_lists = (float2 *)(ws + L.router_lists);
    c->router_meta = (float4 *)(ws + L.router_meta);
    c->router_rows = (bf16 *)(ws + L.router_rows);
    c->a_perm = (bf16 *)(ws + L.a_perm);
    c->act = (bf16 *)(ws + L.act);
    c->y = (bf16 *)(ws + L.y);
    c->act_sh = s.E_sh > 0 ? (bf16 *)(ws + L.act_sh) : nullptr;
    c->y_sh = s.E_sh > 0 ? (bf16 *)(ws + L.y_sh) : nullptr;
    c->stream = (cudaStream_t)stream;
    c->unmasked = d->unmasked_control;
    c->saved_gu = d->saved_gu;
    if (s.T == 0) return PMPE_OK;  // a no-op: no device query, no launch
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PMPE_ERR_CUDA;
    if (cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return PMPE_ERR_CUDA;
    return PMPE_OK;
}

}  // namespace pmpe

using namespace pmpe;

extern "C" {

size_t pmpe_moe_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k)
{
    Shape s{T, H, I, E_pub, E_priv, E_shared, k, 1};
    pmpe_workspace_layout L;
    return compute_layout(s, &L) == PMPE_OK ? L.total : 0;
}

int pmpe_moe_workspace_layout(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k,
                              pmpe_workspace_layout *out)
{
    if (!out) return PMPE_ERR_INVALID_ARG;
    Shape s{T, H, I, E_pub, E_priv, E_shared, k, 1};
    return compute_layout(s, out);
}

size_t pmpe_audit_words(int T, int E)
{
    if (T < 0 || E < 0) return 0;
    return 2 + 3 * (size_t)E + 2 * (size_t)T;
}

int pmpe_policy_resolve(const uint8_t *policy, int T, uint8_t *tau, void *stream)
{
    if (T < 0 || (T > 0 && !tau)) return PMPE_ERR_INVALID_ARG;
    if (T == 0) return PMPE_OK;
    return launch_resolve(policy, T, tau, (cudaStream_t)stream) == cudaSuccess ? PMPE_OK : PMPE_ERR_CUDA;
}

int pmpe_policy_from_requests(const uint8_t *req_policy, const int32_t *cu_seqlens, int n_req, int T,
                              uint8_t *policy_out, void *stream)
{
    if (n_req < 0 || T < 0 || !cu_seqlens || (T > 0 && !policy_out) || (n_req > 0 && !req_policy))
        return PMPE_ERR_INVALID_ARG;
    if (T == 0) return PMPE_OK;
    return launch_policy_from_requests(req_policy, cu_seqlens, n_req, T, policy_out, (cudaStream_t)stream) ==
                   cudaSuccess
               ? PMPE_OK
               : PMPE_ERR_CUDA;
}

int pmpe_moe_forward_stages(const pmpe_moe_desc *d, unsigned stages, void *stream)
{
    Ctx c;
    const int rc = make_ctx(d, stream, &c);
    if (rc != PMPE_OK) return rc;
    if (c.s.T == 0 || stages == 0) return PMPE_OK;
    if (stages & ~PMPE_STAGE_ALL) return PMPE_ERR_INVALID_ARG;
    cudaError_t err = cudaSuccess;
    // The whole forward at T <= 128: the persistent expert launch routes the
    // tokens and derives the dispatch order itself.  Otherwise, with both the
    // router and the dispatch in this call, the router writes the dispatch
    // order at T <= 128; else the dispatch runs inside the persistent expert
    // launch when that launch follows the router in this call (the router
    // zeroes its grid barrier), else as a kernel.
    const bool all = (stages & PMPE_STAGE_ROUTE) && (stages & PMPE_STAGE_PERMUTE) && (stages & PMPE_STAGE_GATEUP) &&
                     (stages & PMPE_STAGE_DOWN);
    if (all && experts_fuse_route(c)) {  // the combine too, when asked for
        err = launch_experts_routed(c, (stages & PMPE_STAGE_COMBINE) != 0);
        return err == cudaSuccess ? PMPE_OK : PMPE_ERR_CUDA;
    }
    const bool route_disp = (stages & PMPE_STAGE_ROUTE) && (stages & PMPE_STAGE_PERMUTE) && route_writes_dispatch(c);
    const bool fuse = !route_disp && (stages & PMPE_STAGE_ROUTE) && (stages & PMPE_STAGE_PERMUTE) &&
                      (stages & PMPE_STAGE_GATEUP) && (stages & PMPE_STAGE_DOWN) && experts_fuse_dispatch(c);
    if (err == cudaSuccess && (stages & PMPE_STAGE_ROUTE)) err = launch_route(c, route_disp);
    if (err == cudaSuccess && (stages & PMPE_STAGE_PERMUTE) && !fuse && !route_disp) err = launch_permute(c);
    if ((stages & PMPE_STAGE_GATEUP) && (stages & PMPE_STAGE_DOWN)) {
        // one persistent launch; its readiness counters are cleared by the
        // dispatch when the dispatch runs in this call (inside it, when fused)
        if (err == cudaSuccess) err = launch_experts(c, !(stages & PMPE_STAGE_PERMUTE), fuse);
    } else {
        if (err == cudaSuccess && (stages & PMPE_STAGE_GATEUP)) err = launch_gateup(c);
        if (err == cudaSuccess && (stages & PMPE_STAGE_DOWN)) err = launch_down(c);
    }
    if (err == cudaSuccess && (stages & PMPE_STAGE_COMBINE)) err = launch_combine(c);
    return err == cudaSuccess ? PMPE_OK : PMPE_ERR_CUDA;
}

size_t pmpe_moe_backward_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k)
{
    Shape s;
    s.T = T; s.H = H; s.I = I; s.E_pub = E_pub; s.E_priv = E_priv; s.E_sh = E_shared; s.k = k; s.renorm = 1;
    if (!shape_ok(s)) return 0;
    return backward_workspace_bytes(s);
}

int pmpe_moe_backward_private(const pmpe_moe_desc *d, const void *dout, float *d_router_priv, float *d_gate_priv,
                              float *d_up_priv, float *d_down_priv, void *bwd_workspace, size_t bwd_workspace_bytes,
                              void *stream)
{
    // every argument is checked before the first CUDA call
    if (!d) return PMPE_ERR_INVALID_ARG;
    const Shape s = shape_of(d);
    const void *need[] = {d_router_priv, d_gate_priv, d_up_priv, d_down_priv};
    for (const void *q : need)
        if (!q || !aligned16(q)) return PMPE_ERR_INVALID_ARG;
    if (s.T > 0 && (!dout || !aligned16(dout))) return PMPE_ERR_INVALID_ARG;
    if (d->unmasked_control == 1) return PMPE_ERR_UNSUPPORTED_SHAPE;  // the control is not trained
    if (shape_ok(s) && s.T > 0 &&
        (!bwd_workspace || bwd_workspace_bytes < backward_workspace_bytes(s) || ((uintptr_t)bwd_workspace & 255u)))
        return PMPE_ERR_WORKSPACE;
    Ctx c;
    const int rc = make_ctx(d, stream, &c);
    if (rc != PMPE_OK) return rc;
    if (s.T == 0) {  // nothing routed: every gradient is zero
        cudaStream_t st = (cudaStream_t)stream;
        const size_t ih = (size_t)s.E_priv * s.I * s.H * sizeof(float);
        cudaError_t err = cudaMemsetAsync(d_router_priv, 0, (size_t)s.E_priv * s.H * sizeof(float), st);
        if (err == cudaSuccess) err = cudaMemsetAsync(d_gate_priv, 0, ih, st);
        if (err == cudaSuccess) err = cudaMemsetAsync(d_up_priv, 0, ih, st);
        if (err == cudaSuccess) err = cudaMemsetAsync(d_down_priv, 0, ih, st);
        return err == cudaSuccess ? PMPE_OK : PMPE_ERR_CUDA;
    }
    // the forward gathers its rows on the fly; the backward's GEMMs read the
    // private experts' dispatched rows as one matrix
    if (launch_gather_dispatch_rows(c, s.E_pub, s.E()) != cudaSuccess) return PMPE_ERR_CUDA;
    return launch_backward_private(c, (const bf16 *)dout, d_router_priv, d_gate_priv, d_up_priv, d_down_priv,
                                   (uint8_t *)bwd_workspace) == cudaSuccess
               ? PMPE_OK
               : PMPE_ERR_CUDA;
}

size_t pmpe_moe_backward_input_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k)
{
    Shape s;
    s.T = T; s.H = H; s.I = I; s.E_pub = E_pub; s.E_priv = E_priv; s.E_sh = E_shared; s.k = k; s.renorm = 1;
    if (!shape_ok(s)) return 0;
    return backward_input_workspace_bytes(s);
}

int pmpe_moe_backward_input(const pmpe_moe_desc *d, const void *dout, float *d_hidden, void *bwd_workspace,
                            size_t bwd_workspace_bytes, void *stream)
{
    // every argument is checked before the first CUDA call
    if (!d) return PMPE_ERR_INVALID_ARG;
    const Shape s = shape_of(d);
    if (s.T > 0 && (!dout || !aligned16(dout) || !d_hidden || !aligned16(d_hidden))) return PMPE_ERR_INVALID_ARG;
    if (d->unmasked_control == 1) return PMPE_ERR_UNSUPPORTED_SHAPE;
    if (shape_ok(s) && s.T > 0 &&
        (!bwd_workspace || bwd_workspace_bytes < backward_input_workspace_bytes(s) ||
         ((uintptr_t)bwd_workspace & 255u)))
        return PMPE_ERR_WORKSPACE;
    Ctx c;
    const int rc = make_ctx(d, stream, &c);
    if (rc != PMPE_OK) return rc;
    if (s.T == 0) return PMPE_OK;  // no tokens: nothing to write
    if (launch_gather_dispatch_rows(c, 0, s.E()) != cudaSuccess) return PMPE_ERR_CUDA;
    return launch_backward_input(c, (const bf16 *)dout, d_hidden, (uint8_t *)bwd_workspace) == cudaSuccess
               ? PMPE_OK
               : PMPE_ERR_CUDA;
}

size_t pmpe_saved_gu_floats(int T, int I, int E_shared, int k)
{
    if (T < 0 || I < 0 || E_shared < 0 || k < 0) return 0;
    return (size_t)T * k * 2 * I + (size_t)T * 2 * E_shared * I;
}

size_t pmpe_moe_backward_step_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k)
{
    Shape s;
    s.T = T; s.H = H; s.I = I; s.E_pub = E_pub; s.E_priv = E_priv; s.E_sh = E_shared; s.k = k; s.renorm = 1;
    if (!shape_ok(s)) return 0;
    return backward_step_workspace_bytes(s);
}

int pmpe_moe_backward_step(const pmpe_moe_desc *d, const void *dout, float *d_router_priv, float *d_gate_priv,
                           float *d_up_priv, float *d_down_priv, float *d_hidden, void *bwd_workspace,
                           size_t bwd_workspace_bytes, void *stream)
{
    // every argument is checked before the first CUDA call
    if (!d) return PMPE_ERR_INVALID_ARG;
    const Shape s = shape_of(d);
    const void *need[] = {d_router_priv, d_gate_priv, d_up_priv, d_down_priv};
    for (const void *q : need)
        if (!q || !aligned16(q)) return PMPE_ERR_INVALID_ARG;
    if (s.T > 0 && (!dout || !aligned16(dout) || !d_hidden || !aligned16(d_hidden))) return PMPE_ERR_INVALID_ARG;
    if (d->unmasked_control == 1) return PMPE_ERR_UNSUPPORTED_SHAPE;
    if (shape_ok(s) && s.T > 0 &&
        (!bwd_workspace || bwd_workspace_bytes < backward_step_workspace_bytes(s) ||
         ((uintptr_t)bwd_workspace & 255u)))
        return PMPE_ERR_WORKSPACE;
    Ctx c;
    const int rc = make_ctx(d, stream, &c);
    if (rc != PMPE_OK) return rc;
    if (s.T == 0) {  // nothing routed: every parameter gradient is zero, d_hidden is empty
        cudaStream_t st = (cudaStream_t)stream;
        const size_t ih = (size_t)s.E_priv * s.I * s.H * sizeof(float);
        cudaError_t err = cudaMemsetAsync(d_router_priv, 0, (size_t)s.E_priv * s.H * sizeof(float), st);
        if (err == cudaSuccess) err = cudaMemsetAsync(d_gate_priv, 0, ih, st);
        if (err == cudaSuccess) err = cudaMemsetAsync(d_up_priv, 0, ih, st);
        if (err == cudaSuccess) err = cudaMemsetAsync(d_down_priv, 0, ih, st);
        return err == cudaSuccess ? PMPE_OK : PMPE_ERR_CUDA;
    }
    if (launch_gather_dispatch_rows(c, 0, s.E()) != cudaSuccess) return PMPE_ERR_CUDA;
    return launch_backward_step(c, (const bf16 *)dout, d_router_priv, d_gate_priv, d_up_priv, d_down_priv, d_hidden,
                                (uint8_t *)bwd_workspace) == cudaSuccess
               ? PMPE_OK
               : PMPE_ERR_CUDA;
}

int pmpe_moe_forward(const pmpe_moe_desc *d, void *stream)
{
    return pmpe_moe_forward_stages(d, PMPE_STAGE_ALL, stream);
}

int pmpe_audit_reset(uint32_t *audit, int T, int E, void *stream)
{
    if (!audit || T < 0 || E < 0) return PMPE_ERR_INVALID_ARG;
    return cudaMemsetAsync(audit, 0, sizeof(uint32_t) * pmpe_audit_words(T, E), (cudaStream_t)stream) == cudaSuccess
               ? PMPE_OK
               : PMPE_ERR_CUDA;
}

int pmpe_audit_read(const uint32_t *audit, int T, int E, uint32_t *host_out, void *stream, int timeout_ms)
{
    if (!audit || !host_out || T < 0 || E < 0 || timeout_ms < 0) return PMPE_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    if (cudaMemcpyAsync(host_out, audit, sizeof(uint32_t) * pmpe_audit_words(T, E), cudaMemcpyDeviceToHost, st) !=
        cudaSuccess)
        return PMPE_ERR_CUDA;
    cudaEvent_t ev;
    if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess) return PMPE_ERR_CUDA;
    if (cudaEventRecord(ev, st) != cudaSuccess) {
        cudaEventDestroy(ev);
        return PMPE_ERR_CUDA;
    }
    const auto deadline = std::chrono::steady_clock::now() + std::chrono::milliseconds(timeout_ms);
    int rc = PMPE_OK;
    for (;;) {
        const cudaError_t q = cudaEventQuery(ev);
        if (q == cudaSuccess) break;
        if (q != cudaErrorNotReady) { rc = PMPE_ERR_CUDA; break; }
        if (std::chrono::steady_clock::now() >= deadline) { rc = PMPE_ERR_TIMEOUT; break; }
        std::this_thread::sleep_for(std::chrono::microseconds(50));
    }
    cudaEventDestroy(ev);
    if (rc == PMPE_OK && host_out[0] != 0) rc = PMPE_ERR_DEVICE_STATUS;
    return rc;
}

const char *pmpe_status_string(int status)
{
    switch (status) {
    case PMPE_OK: return "ok";
    case PMPE_ERR_INVALID_ARG: return "invalid argument";
    case PMPE_ERR_UNSUPPORTED_SHAPE: return "unsupported shape or alignment";
    case PMPE_ERR_WORKSPACE: return "workspace missing or too small";
    case PMPE_ERR_CUDA: return "CUDA runtime error";
    case PMPE_ERR_TIMEOUT: return "timed out waiting for the device";
    case PMPE_ERR_DEVICE_STATUS: return "a kernel recorded an error in the audit status word";
    default: return "unknown status";
    }
}

}  // extern "C"
