/*
 * pmpe.h -- C ABI of libpmpe: the GB300 (sm_103a) forward pass of one
 * policy-masked sparse-MoE layer, the method of "Policy-Masked Private
 * Experts" (arXiv 2608.06690).
 *
 * The layer (Sec. 3.1 and App. B.1 of the paper):
 *   1. a trusted per-token policy byte is resolved fail-closed: only 0x01 is
 *      ALLOW (tau = 1), every other byte and a missing (NULL) policy is DENY
 *      (Sec. 2.1, App. B.1 "Policy resolution and masked routing");
 *   2. tau selects one of two mutually exclusive expert pools -- the private
 *      pool for ALLOW, the original public pool for DENY -- and the router
 *      logits are computed over that pool only, so an ineligible expert never
 *      enters the candidate set (Sec. 3.1, Eq. 4 and the sentence after it);
 *   3. top-k inside the pool with softmax weights (renormalised over the top-k,
 *      or the pool softmax without renormalisation);
 *   4. token rows are grouped by expert, each expert runs its SwiGLU MLP
 *      (gate/up projection, silu(gate) * up, down projection; private experts
 *      copy the public expert architecture, Sec. 3.1), and the outputs are
 *      combined with the routing weights, plus always-on shared experts;
 *   5. the expert kernels themselves count the rows they execute, an audit
 *      trail independent of the route log (Sec. 5.2 and App. F.1: the
 *      independent hooks that counted physical private rows).
 *
 * Global expert ids: public 0 .. E_pub-1, private E_pub .. E_pub+E_priv-1
 * (the concatenated public/private pool of Sec. 4.2).
 *
 * Conventions for every entry point:
 *   - All tensor pointers are DEVICE pointers unless stated otherwise; the
 *     caller allocates and owns every buffer.  The library keeps no mutable
 *     global state between calls and never allocates device memory.
 *   - BF16 tensors are passed as raw 16-bit words (void *), row-major, with
 *     the [out, in] layout of a linear layer.  Every pointer must be 16-byte
 *     aligned.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Calls
 *     are asynchronous on it unless stated otherwise.
 *   - Return value: PMPE_OK or a negative PMPE_ERR_* code.  When a call
 *     returns an error before launching, nothing has been enqueued and no
 *     output has been touched.
 *   - A malformed policy byte is never an error: it resolves to DENY.
 */
#ifndef PMPE_H
#define PMPE_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define PMPE_API __attribute__((visibility("default")))
#else
#define PMPE_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ----------------------------------------------------------- status codes */
#define PMPE_OK 0
#define PMPE_ERR_INVALID_ARG (-1)       /* NULL required pointer, k < 1, k > a pool size, T < 0, ... */
#define PMPE_ERR_UNSUPPORTED_SHAPE (-2) /* H or I not a multiple of 128, a pool above 256, k above 32,
                                           or a pointer not 16-byte aligned */
#define PMPE_ERR_WORKSPACE (-3)         /* workspace NULL or smaller than pmpe_moe_workspace_size() */
#define PMPE_ERR_CUDA (-4)              /* a CUDA runtime call failed */
#define PMPE_ERR_TIMEOUT (-5)           /* a bounded host wait ran out */
#define PMPE_ERR_DEVICE_STATUS (-6)     /* a kernel recorded an error in the audit status word */

/* Bits a kernel may OR into the device status word (audit word 0). */
#define PMPE_STATUS_DISPATCH_MISMATCH 0x1u /* an expert kernel ran a row whose token's route does not name that expert */
#define PMPE_STATUS_PIPELINE_TIMEOUT 0x2u  /* a bounded wait inside an expert kernel gave up */
#define PMPE_STATUS_BAD_EXPERT_ID 0x4u     /* a routed id outside [0, E) reached the dispatcher */

/* Stage bits for pmpe_moe_forward_stages(). */
#define PMPE_STAGE_ROUTE 0x01u   /* resolve + masked router + top-k + route log */
#define PMPE_STAGE_PERMUTE 0x02u /* per-expert dispatch order (slot maps) */
#define PMPE_STAGE_GATEUP 0x04u  /* grouped gate/up GEMM on rows gathered from hidden, fused silu(g)*u,
                                    execution audit */
#define PMPE_STAGE_DOWN 0x08u    /* grouped down GEMM, scaled by the routing weight */
#define PMPE_STAGE_COMBINE 0x10u /* weighted unpermute-combine (+ shared experts) */
#define PMPE_STAGE_ALL 0x1Fu

/* ------------------------------------------------------------ layer desc */
typedef struct pmpe_moe_desc {
    int T;            /* tokens, >= 0 (0 is a no-op) */
    int H;            /* hidden size, multiple of 128 */
    int I;            /* expert intermediate size, multiple of 128 */
    int E_pub;        /* public routed experts, k <= E_pub <= 256 */
    int E_priv;       /* private routed experts, k <= E_priv <= 256 */
    int E_shared;     /* always-on shared experts (0 = none), weight 1, run for every token */
    int k;            /* experts per token inside the selected pool, 1 <= k <= 32 */
    int renormalize;  /* 1: w = softmax over the k selected logits; 0: w = pool-softmax probabilities */

    const void *hidden;          /* [T, H] BF16 */
    const uint8_t *policy;       /* [T] trusted policy bytes; NULL = metadata missing = all DENY */

    const void *w_router_pub;    /* [E_pub, H] BF16 */
    const void *w_router_priv;   /* [E_priv, H] BF16 */
    const void *w_gate_pub;      /* [E_pub, I, H] BF16 */
    const void *w_up_pub;        /* [E_pub, I, H] BF16 */
    const void *w_down_pub;      /* [E_pub, H, I] BF16 */
    const void *w_gate_priv;     /* [E_priv, I, H] BF16 */
    const void *w_up_priv;       /* [E_priv, I, H] BF16 */
    const void *w_down_priv;     /* [E_priv, H, I] BF16 */
    const void *w_gate_sh;       /* [E_shared, I, H] BF16, or NULL when E_shared == 0 */
    const void *w_up_sh;         /* [E_shared, I, H] BF16 */
    const void *w_down_sh;       /* [E_shared, H, I] BF16 */

    void *out;                   /* [T, H] BF16 output */
    int32_t *topk_idx;           /* optional [T, k] route log: global expert ids, descending score */
    float *topk_w;               /* optional [T, k] routing weights */
    uint32_t *audit;             /* optional pmpe_audit_words(T, E_pub+E_priv) counters; accumulate
                                    across calls until pmpe_audit_reset() */
    void *workspace;             /* device scratch, >= pmpe_moe_workspace_size() bytes, 256-byte aligned */
    size_t workspace_bytes;

    /* 0: the method.  1: the paper's soft-router control (Sec. 4.2 "Matched
     * adaptation and controls" and App. E, the control matrix's
     * soft-router-only arm): every token routes over the concatenated public/private
     * pool without the hard mask, whatever its policy byte.  A negative
     * control for audits: private rows then execute for DENY tokens, which
     * the audit counters record.  Requires the merge of the router's chunk
     * lists to fit in shared memory: ceil(E_pub/32) + ceil(E_priv/32) <= 16
     * and that count * k <= 96; PMPE_ERR_UNSUPPORTED_SHAPE otherwise. */
    int unmasked_control;

    /* Optional, for training: pmpe_saved_gu_floats() FP32 values, 16-byte
     * aligned, or NULL.  When set, the forward also writes the gate and up
     * pre-activations (the FP32 accumulators its SwiGLU reads): first
     * [T*k, 2I], G | U of each dispatch row, then, with shared experts,
     * [T, 2*E_shared*I], the shared experts' G side by side, then their U.
     * The backward calls given the same descriptor read them instead of
     * recomputing the gate/up GEMMs; their results are then bitwise those of
     * the recomputation. */
    float *saved_gu;
} pmpe_moe_desc;

/* FP32 values of the optional saved_gu buffer: T*k*2*I + T*2*E_shared*I. */
PMPE_API size_t pmpe_saved_gu_floats(int T, int I, int E_shared, int k);

/* Bytes of device workspace pmpe_moe_forward() needs for this shape.
 * Returns 0 for an invalid shape. */
PMPE_API size_t pmpe_moe_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k);

/* Byte offsets of the named regions inside the workspace (for tests that
 * inspect intermediate results, and for the stage-by-stage entry point).
 * Router geometry used below: S = ceil(T/128) + 1 token-tile slots,
 * C = S * max(ceil(E_pub/32), ceil(E_priv/32)) router CTAs (one per tile and
 * 32-expert chunk of its pool) and C2 = S * (ceil(E_pub/32) + ceil(E_priv/32))
 * (the unmasked control's chunks of the concatenated pool).  Returns PMPE_ERR_INVALID_ARG for an invalid
 * shape. */
typedef struct pmpe_workspace_layout {
    size_t total;
    size_t tau;          /* uint8  [T]      resolved policy bits */
    size_t counts;       /* uint32 [E]      rows routed to each expert (router's integer atomics) */
    size_t offsets;      /* uint32 [E+1]    exclusive prefix sum of counts */
    size_t topk_idx;     /* int32  [T, k]   used when desc.topk_idx is NULL */
    size_t topk_w;       /* float  [T, k]   used when desc.topk_w is NULL */
    size_t slot_of;      /* int32  [T, k]   dispatch row of (t, j) */
    size_t ticket;       /* int32  [T, k]   128 * (router tile of t) + position of (t, j) among the
                          * tile's rows of its expert (the tile's tokens in ascending order) */
    size_t tok_of_slot;  /* int32  [T*k]    token of each dispatch row */
    size_t w_of_slot;    /* float  [T*k]    routing weight of each dispatch row */
    size_t router_rows;  /* BF16   [C*128, H]  token rows of each router CTA whose tile is not consecutive */
    size_t a_perm;       /* BF16   [T*k, H] token rows in dispatch order, written by the backward calls
                          * (the forward's expert kernel gathers them from `hidden` as it goes) */
    size_t act;          /* BF16   [T*k, I] silu(g)*u of each dispatch row */
    size_t y;            /* BF16   [T*k, H] w * expert output of each dispatch row */
    size_t act_sh;       /* BF16   [T, E_shared*I] shared-expert activations (0 if none) */
    size_t y_sh;         /* BF16   [T, H] summed shared-expert outputs (0 if none) */
    size_t tile_done;    /* uint32 [S]      router CTAs finished per 128-token tile */
    size_t router_lists; /* float2 [C2*128, k] per 32-expert chunk: each token's best k (score, id) */
    size_t router_meta;  /* float4 [C2*128] per chunk: max score, sum exp(score - max), entries */
    size_t gemm_ready;   /* uint32 [(T*k+127)/128 + E + (T+127)/128 + 1]  gate/up epilogue warps done per
                          * (expert group, 128-row block), read by the down tiles of the same launch */
    size_t tile_counts;  /* uint32 [E, S4]  rows of expert e in router tile s (S4 = S rounded up to 4).
                          * With the tiles of a pool in ascending token order, slot
                          * offsets[e] + sum_{s' < s} tile_counts[e, s'] + position gives every expert
                          * its rows in ascending (t, j) order: the dispatch order is deterministic */
} pmpe_workspace_layout;
PMPE_API int pmpe_moe_workspace_layout(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k,
                              pmpe_workspace_layout *out);

/* Number of uint32 words of the audit buffer for T tokens and E routed
 * experts.  Layout (word offsets):
 *   [0]                  status   OR of PMPE_STATUS_* bits
 *   [1]                  shared_rows      (token, shared expert) pairs executed
 *   [2, 2+E)             route_count[e]   rows the router sent to expert e
 *   [2+E, 2+2E)          exec_rows[e]     rows the expert kernels executed for e
 *   [2+2E, 2+3E)         exec_tiles[e]    row tiles the expert kernels ran for e
 *   [2+3E, 2+3E+T)       route_priv_rows[t]  private experts in token t's route
 *   [2+3E+T, 2+3E+2T)    exec_priv_rows[t]   private expert rows executed for token t
 * The route words come from the router; the exec words are written from inside
 * the grouped expert GEMM tiles, from the rows each tile processed: a row
 * counts in exec_rows[e] only if its token's route names e (each row is
 * checked against the route log), exec_priv_rows counts the private rows
 * physically run per token, and a row that fails the check sets
 * PMPE_STATUS_DISPATCH_MISMATCH in the status word. */
PMPE_API size_t pmpe_audit_words(int T, int E);

/* Resolve T trusted policy bytes to tau (0/1 bytes): tau[t] = (policy[t] == 0x01).
 * policy == NULL means missing metadata: every tau is 0.  tau: [T] device.
 * App. B.1, step 2 of the fail-closed procedure. */
PMPE_API int pmpe_policy_resolve(const uint8_t *policy, int T, uint8_t *tau, void *stream);

/* ------------------------------------------------- private-branch backward */

/* Bytes of device scratch pmpe_moe_backward_private() needs; 0 for an invalid
 * shape. */
PMPE_API size_t pmpe_moe_backward_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared, int k);

/* Gradients of L = sum_t dout_t . out_t with respect to the PRIVATE
 * parameters only, for the routing of the forward just run with the same
 * descriptor (G2, Sec. 2.2; Sec. 3.2: only the private branch is trained, the
 * public parameters are frozen and get no gradient, and DENY tokens reach no
 * private parameter).  The descriptor's workspace must still hold that
 * forward's state (route log, dispatch order, dispatched rows, activations):
 * run the forward, then this, on the same stream, with nothing in between
 * that reuses the workspace, passing that forward's descriptor (its route
 * outputs topk_idx / topk_w included; its `out` is not written).
 * dout: [T, H] BF16 upstream gradient.  Outputs
 * (FP32, overwritten, 16-byte aligned): d_router_priv [E_priv, H],
 * d_gate_priv and d_up_priv [E_priv, I, H], d_down_priv [E_priv, H, I].  The
 * rounding points of the forward (FP32 logits, BF16 activations) are taken as
 * the identity.  Not defined for the unmasked control
 * (PMPE_ERR_UNSUPPORTED_SHAPE).  bwd_workspace: >= the size above, 256-byte
 * aligned (PMPE_ERR_WORKSPACE otherwise).  Asynchronous on `stream`. */
PMPE_API int pmpe_moe_backward_private(const pmpe_moe_desc *d, const void *dout, float *d_router_priv,
                                       float *d_gate_priv, float *d_up_priv, float *d_down_priv,
                                       void *bwd_workspace, size_t bwd_workspace_bytes, void *stream);

/* ------------------------------------------------- input gradient */

/* Bytes of device scratch pmpe_moe_backward_input() needs; 0 for an invalid
 * shape. */
PMPE_API size_t pmpe_moe_backward_input_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared,
                                                       int k);

/* Gradient of L = sum_t dout_t . out_t with respect to the layer's input
 * hidden [T, H], through the frozen layer, for the routing of the forward just
 * run with the same descriptor: what the layer below needs when its own private
 * branch is trained (Sec. 3.2).  Every term of the forward contributes: each
 * token's k routed experts of its own pool (the pool the mask of Sec. 3.1
 * Eq. 4 selects: public for DENY, private for ALLOW) through their routing
 * weights, the shared experts with weight 1, and the router of that pool
 * through the routing softmax (renormalised over the top-k, or over the
 * pool).  The routing itself (which experts, the hard
 * mask) is piecewise constant and contributes no gradient.  The descriptor's
 * workspace must still hold that forward's state, as for
 * pmpe_moe_backward_private().  dout: [T, H] BF16.  d_hidden: [T, H] FP32,
 * overwritten, 16-byte aligned.  The per-pick input gradients are rounded to
 * BF16 before the FP32 sum.  Not defined for the unmasked control
 * (PMPE_ERR_UNSUPPORTED_SHAPE).  bwd_workspace: >= the size above, 256-byte
 * aligned (PMPE_ERR_WORKSPACE otherwise).  Asynchronous on `stream`. */
PMPE_API int pmpe_moe_backward_input(const pmpe_moe_desc *d, const void *dout, float *d_hidden, void *bwd_workspace,
                                     size_t bwd_workspace_bytes, void *stream);

/* ------------------------------------------------- both, in one pass */

/* Bytes of device scratch pmpe_moe_backward_step() needs; 0 for an invalid
 * shape. */
PMPE_API size_t pmpe_moe_backward_step_workspace_size(int T, int H, int I, int E_pub, int E_priv, int E_shared,
                                                      int k);

/* The private-parameter gradients of pmpe_moe_backward_private() and the
 * input gradient of pmpe_moe_backward_input() in one pass, for a training
 * step that needs both (Sec. 3.2: the private branch of every wrapped layer
 * is trained, so each layer also passes dL/dh to the layer below).  The
 * private experts' rows are recomputed once for both.  Every output is
 * bitwise the one the two separate calls give.  Arguments, preconditions and
 * errors are those of the two calls: the forward's descriptor and workspace,
 * dout [T, H] BF16, d_router_priv [E_priv, H], d_gate_priv and d_up_priv
 * [E_priv, I, H], d_down_priv [E_priv, H, I] and d_hidden [T, H], all FP32,
 * overwritten and 16-byte aligned; bwd_workspace of at least the size above,
 * 256-byte aligned.  Asynchronous on `stream`. */
PMPE_API int pmpe_moe_backward_step(const pmpe_moe_desc *d, const void *dout, float *d_router_priv,
                                    float *d_gate_priv, float *d_up_priv, float *d_down_priv, float *d_hidden,
                                    void *bwd_workspace, size_t bwd_workspace_bytes, void *stream);

/* Per-token policy bytes from per-request ones, for callers that carry one
 * trusted authorisation byte per request and the requests' cumulative token
 * offsets (cu_seqlens[0..n_req], device int32) instead of a byte per token.
 * policy_out[t] = req_policy[r] for cu_seqlens[r] <= t < cu_seqlens[r+1];
 * tokens after cu_seqlens[n_req] get 0x00 (DENY).  Malformed offsets
 * (cu_seqlens[0] != 0, a decreasing step, or cu_seqlens[n_req] > T) are
 * malformed metadata: every token gets 0x00 (Sec. 2.1, App. B.1 fail
 * closed).  The result feeds pmpe_moe_desc.policy.  All pointers device;
 * asynchronous on `stream`; PMPE_ERR_INVALID_ARG for negative sizes or a
 * NULL pointer that is needed.  (The request-offset ABI of the serving path;
 * the paper specifies the authorisation per request, Sec. 2.1.) */
PMPE_API int pmpe_policy_from_requests(const uint8_t *req_policy, const int32_t *cu_seqlens, int n_req, int T,
                                       uint8_t *policy_out, void *stream);

/* The whole layer forward (all stages) on `stream`.  No host synchronisation;
 * expert row counts stay on the device.  The expert launch is persistent, one
 * CTA per SM, and its CTAs wait for one another (grid barriers, readiness
 * counters): it assumes the whole grid is resident at once, which the library
 * checks for this device before it takes that form.  If other work on the GPU
 * holds SMs for longer than the bounded waits (4 s), the waits expire, the
 * kernel sets PMPE_STATUS_PIPELINE_TIMEOUT in the status word and returns;
 * the outputs of that call are then not valid. */
PMPE_API int pmpe_moe_forward(const pmpe_moe_desc *d, void *stream);

/* Run a subset of the stages (PMPE_STAGE_* bits), in pipeline order.  Each
 * stage reads what the previous stages left in the same workspace, so a
 * stage may only be run after its predecessors have run on that workspace
 * with the same inputs.  pmpe_moe_forward() == stages PMPE_STAGE_ALL. */
PMPE_API int pmpe_moe_forward_stages(const pmpe_moe_desc *d, unsigned stages, void *stream);

/* Self-test of the failure path of the layer's pipelined kernels: launches one
 * kernel whose shared-memory barrier wait can never complete (nothing
 * arrives), through the same bounded wait the layer's tensor-core kernels use
 * at every pipeline stage, with a limit of limit_us microseconds (1 ..
 * 1,000,000).  The wait expires, ORs PMPE_STATUS_PIPELINE_TIMEOUT into
 * *status (a device word, e.g. audit word 0) and the kernel returns; the CUDA
 * context stays usable.  Asynchronous on `stream`.  Not part of the paper's
 * method: it tests the library's failure detection (device waits are bounded,
 * expiry is reported, never a hang or a trap). */
PMPE_API int pmpe_selftest_wait_timeout(uint32_t *status, int limit_us, void *stream);

/* Size of the device scratch array that pmpe_moe_forward_noalloc() uses in
 * place of a caller workspace: 32 MiB, reserved on every GPU that loads the
 * library until the process exits.  (A 64-token decode step of a layer with
 * H = 2048, I = 768, top-8 needs about 5 MB of it.) */
#define PMPE_STATIC_SCRATCH_BYTES (32u << 20)

/* The layer forward for callers that cannot allocate device memory where
 * they run it -- a plugin whose host owns all device memory and offers it no
 * allocator, or a serving loop that must not pay cudaMalloc's device-wide
 * synchronisation or risk running out of memory mid-request.  The paper has
 * no counterpart to this entry point; it is a deployment convenience.
 *   - Same arguments and results as pmpe_moe_forward(), except that
 *     d->workspace and d->workspace_bytes are ignored: the scratch is the
 *     library's own static device array of PMPE_STATIC_SCRATCH_BYTES.
 *   - Returns PMPE_ERR_WORKSPACE, launching nothing, when the shape's
 *     pmpe_moe_workspace_size() exceeds PMPE_STATIC_SCRATCH_BYTES.
 *   - Allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current) and caches it per
 *     device and CUDA context; a call in a new context on the device (after
 *     cudaDeviceReset, for instance) looks it up again.  Make the first call
 *     on a device, and in each new context, before any stream capture.
 *   - All calls on a device share the one array, which keeps the last call's
 *     contents (the forward clears what must start at zero).  Calls whose
 *     kernels overlap on the GPU race on it: order them on one stream or with
 *     events. */
PMPE_API int pmpe_moe_forward_noalloc(const pmpe_moe_desc *d, void *stream);

/* Zero the audit buffer (pmpe_audit_words(T, E) words). */
PMPE_API int pmpe_audit_reset(uint32_t *audit, int T, int E, void *stream);

/* Copy the audit buffer to caller host memory `host_out` (same word count)
 * and wait for the copy with a bounded poll.  Returns PMPE_ERR_TIMEOUT if it
 * has not completed after timeout_ms milliseconds (the copy stays enqueued),
 * PMPE_ERR_DEVICE_STATUS if the status word is nonzero, PMPE_OK otherwise. */
PMPE_API int pmpe_audit_read(const uint32_t *audit, int T, int E, uint32_t *host_out, void *stream, int timeout_ms);

/* Human-readable text of a status code (static storage). */
PMPE_API const char *pmpe_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* PMPE_H */
