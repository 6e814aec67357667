// Internal declarations shared by the libpmpe translation units: the launch
// context, the workspace carve-up and small device helpers.  Nothing here is
// part of the C ABI (include/pmpe.h is).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <utility>

#include "../../include/pmpe.h"

namespace pmpe {

typedef __nv_bfloat16 bf16;

// Limits checked on the host before any launch.
constexpr int kMaxPool = 256;   // experts per pool (router smem tiles)
constexpr int kMaxTopK = 32;    // one warp lane per selected expert
constexpr int kDimAlign = 128;  // H and I granularity

struct Shape {
    int T, H, I, E_pub, E_priv, E_sh, k, renorm;
    int E() const { return E_pub + E_priv; }
};

// Pointers into the audit buffer (all NULL when the caller passed none).
struct Audit {
    uint32_t *status, *shared_rows, *route_count, *exec_rows, *exec_tiles, *route_priv_rows, *exec_priv_rows;
};

Audit audit_ptrs(uint32_t *base, int T, int E);

// Everything one forward call needs, resolved from the descriptor.
struct Ctx {
    Shape s;
    const bf16 *hidden;
    const uint8_t *policy;
    const bf16 *router_pub, *router_priv;
    // [0] public, [1] private, [2] shared
    const bf16 *gate[3], *up[3], *down[3];
    bf16 *out;
    int32_t *idx;
    float *w;
    Audit audit;
    // workspace regions
    uint8_t *tau;
    uint32_t *counts, *offsets;
    int32_t *slot_of, *tok_of_slot;
    int32_t *ticket;    // [T, k] 128 * router tile + position among the tile's rows of its expert
    float *w_of_slot;
    uint32_t *tile_done;  // [router slots] chunk CTAs finished per router tile
    uint32_t *tile_counts; // [E][router_slots4] rows of each expert per router tile
    uint32_t *gemm_ready; // [gemm_ready_words] gate/up warps done per (group, 128-row block)
    float2 *router_lists; // [router CTAs * 128, k] per-chunk sorted (score, id)
    float4 *router_meta;  // [router CTAs * 128] per-chunk softmax partials
    bf16 *router_rows;  // [router CTAs * 128, H] copied token rows of non-contiguous router tiles
    bf16 *a_perm;  // [T*k, H] dispatched rows: filled only by the backward (the forward gathers on the fly)
    bf16 *act, *y, *act_sh, *y_sh;
    cudaStream_t stream;
    int num_sms;
    int unmasked;  // the soft-router control: no hard mask (a negative control, not the method)
    float *saved_gu;  // optional [T*k][2I] FP32 G | U written by the forward, read by the backward
};

int compute_layout(const Shape &s, pmpe_workspace_layout *L);
// Router geometry: 32-expert chunks of a pool, 128-token tile slots for T tokens.
int router_chunks(int pool_size);
int router_slots(int T);
// router_slots rounded up to a multiple of 4 (the row pitch of tile_counts).
int router_slots4(int T);
// Readiness counters of the persistent expert GEMMs: one per (group, 128-row
// block), an upper bound over all routings.
size_t gemm_ready_words(const Shape &s);
// Output columns per down tile: 256 when H allows, else 128.
int column_block(int H);

// Launchers (one per stage); each returns the launch's cudaError_t.
// The router; with write_dispatch (only where route_writes_dispatch holds)
// it also writes the dispatch order and clears the expert launch's
// readiness counters, in place of the dispatch step.
cudaError_t launch_route(const Ctx &c, bool write_dispatch);
// Whether the router can write the dispatch order itself: T <= 128 (each
// pool fills at most one router tile) and the cluster router runs.
bool route_writes_dispatch(const Ctx &c);
// Whether launch_route takes the cluster router (no memset before it; the
// dispatch derives the per-expert counts from tile_counts) or the chunked one.
bool route_uses_cluster_kernel(const Shape &s, int unmasked, int num_sms);
cudaError_t launch_permute(const Ctx &c);
cudaError_t launch_gateup(const Ctx &c);
cudaError_t launch_down(const Ctx &c);
// Backward of the private branch (k_backward.cu): scratch bytes and launch.
size_t backward_workspace_bytes(const Shape &s);
cudaError_t launch_backward_private(const Ctx &c, const bf16 *dout, float *d_router, float *d_gate, float *d_up,
                                    float *d_down, uint8_t *bws);
// Its pieces shared with the input gradient: the upstream gradients of the
// dispatch rows of experts g0 .. g1 - 1 (and 64 zero rows after them); the
// router's softmax gradient from the dL/dw partials per slot (both_pools = 0:
// the private pool, zero for DENY tokens; 1: each token's own pool), dz [T][ld]
// (pool softmax: the pools' token lists go to pool_tok [T] and pool_n [2]).
void launch_gather_rows(const bf16 *dout, const int32_t *tok_of_slot, const uint32_t *offsets, int g0, int g1, int R,
                        int H, bf16 *rows, int num_sms, cudaStream_t st);
cudaError_t launch_router_dz(const Ctx &c, const float *gw_part, int both_pools, int ld, float *dz, int32_t *pool_tok,
                             int *pool_n, float *logit_part);
// Ranges of h the pool-softmax logits are split over: logit_part holds
// router_logit_splits(s) * T * ld floats.
int router_logit_splits(const Shape &s);
// The pool-softmax router term of the input gradient, added to d_hidden
// (pool lists from launch_router_dz).
cudaError_t launch_router_term(const Ctx &c, const float *dz, int ld, const int32_t *pool_tok, const int *pool_n,
                               float *d_hidden);
constexpr int kMaxRouterSplits = 64;  // token ranges of the router weight gradient
// The private router's weight gradient from dz (rows ld apart; DENY rows read
// as zeros): token-range partials (part, router_wgrad_part_bytes) and their
// fixed-order sum into d_router [E_priv, H]; active: kMaxRouterSplits words.
size_t router_wgrad_part_bytes(const Shape &s);
cudaError_t launch_router_wgrad(const Ctx &c, const float *dz, int ld, float *part, int *active, float *d_router);
// Gradient of the layer's input (k_backward_input.cu): scratch bytes and launch.
size_t backward_input_workspace_bytes(const Shape &s);
cudaError_t launch_backward_input(const Ctx &c, const bf16 *dout, float *d_hidden, uint8_t *bws);
// Both in one pass (k_backward_input.cu): the private gradients and the input
// gradient from one set of row launches over all routed experts.
size_t backward_step_workspace_bytes(const Shape &s);
cudaError_t launch_backward_step(const Ctx &c, const bf16 *dout, float *d_router, float *d_gate, float *d_up,
                                 float *d_down, float *d_hidden, uint8_t *bws);
// Its tensor-core GEMMs (k_backward_tc.cu): rows of the padded layout, the
// dL/da and gate/up recompute launches, and the weight-gradient launch.
size_t backward_padded_rows(const Shape &s);
cudaError_t launch_backward_rows(const Ctx &c, const bf16 *dout_rows, bf16 *zpad, bf16 *dgu, bf16 *wact,
                                 float *gw_part);
// The groups of one row launch: routed experts g0 .. g0 + G - 1 (shared_T = 0)
// or the G = E_sh shared experts over shared_T tokens; padded_rows bounds the
// padded row layout of their outputs (each group's rows rounded up to 128).
struct RowsGroups {
    int g0, G, shared_T;
    uint64_t padded_rows;
};
// Z = D W_down (D rows: tight = relative to expert g0's first slot, else the
// slot or token) -> zpad; the gate/up recompute with the SwiGLU backward ->
// [dG | dU] (and w act, dL/dw partials when non-null); dA = [dG | dU] [W_gate; W_up].
cudaError_t launch_rows_z(const Ctx &c, const RowsGroups &g, const bf16 *d, uint64_t d_rows, int tight, bf16 *zpad);
cudaError_t launch_rows_gu(const Ctx &c, const RowsGroups &g, const bf16 *a, uint64_t a_rows, const bf16 *zpad,
                           bf16 *dgu, bf16 *wact, float *gw_part);
cudaError_t launch_rows_da(const Ctx &c, const RowsGroups &g, const bf16 *dgu, bf16 *da);
// all == null: the operands use the private experts' own padded layout and
// dout_rows starts at the first private slot; otherwise the padded layout of
// all routed experts (`all`) and dout_rows indexed by dispatch slot.
cudaError_t launch_backward_wgrad(const Ctx &c, const bf16 *dout_rows, const bf16 *dgu, const bf16 *wact,
                                  float *d_gate, float *d_up, float *d_down, const RowsGroups *all = nullptr);
// Gate/up and down in one persistent launch (down tiles wait for their
// activation rows); zero_ready clears the readiness counters first.  When the
// device cannot host one CTA per SM at once, the two GEMMs run as two launches.
// The persistent gate/up + down launch.  With fuse_dispatch (the router ran
// just before in the same call, and experts_fuse_dispatch holds) the launch
// also derives the dispatch order itself, in place of launch_permute.
cudaError_t launch_experts(const Ctx &c, bool zero_ready, bool fuse_dispatch);
bool experts_fuse_dispatch(const Ctx &c);
// Whether the expert launch can route the tokens itself (T <= 128, the
// masked router, pools of at most 256 experts, H <= 2048, a resident grid),
// and that form of the forward: a kernel clearing the counters, then the
// persistent launch (routing, dispatch, both GEMMs and, with `combine`, the
// weighted combine).
bool experts_fuse_route(const Ctx &c);
cudaError_t launch_experts_routed(const Ctx &c, bool combine);
cudaError_t launch_combine(const Ctx &c);
// The token rows of the dispatch slots of groups g0 .. g1 - 1 copied from the
// hidden states into the workspace's dispatched-row matrix (a_perm), which the
// backward's GEMMs read.
cudaError_t launch_gather_dispatch_rows(const Ctx &c, int g0, int g1);
cudaError_t launch_resolve(const uint8_t *policy, int T, uint8_t *tau, cudaStream_t stream);
cudaError_t launch_policy_from_requests(const uint8_t *req_policy, const int32_t *cu_seqlens, int n_req, int T,
                                        uint8_t *policy_out, cudaStream_t stream);

// Raise `kernel`'s dynamic shared-memory limit on the current device to at
// least `bytes`, calling the runtime only when the limit must grow (the
// setting persists for the process; `limit` caches it per device, 64 devices).
template <typename Kernel>
cudaError_t ensure_dynamic_smem(Kernel kernel, int bytes, std::atomic<int> *limit)
{
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 0 || dev >= 64) return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (limit[dev].load() >= bytes) return cudaSuccess;
    err = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (err == cudaSuccess) {
        int cur = limit[dev].load();
        while (cur < bytes && !limit[dev].compare_exchange_weak(cur, bytes)) {
        }
    }
    return err;
}

// Launch with programmatic dependent launch: the kernel may start (and run
// its prologue) while the previous kernel in the stream finishes; it must
// execute pdl_wait() before touching anything that kernel wrote, or writing
// anything a previous kernel might still read.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ------------------------------------------------------------ device helpers

// Wait until the previous kernel in the stream has completed and its memory
// operations are visible (programmatic dependent launch).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
// Allow the next kernel in the stream to launch now (it still waits for this
// one to complete before touching its results).
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte async copy global -> shared; src_bytes = 0 zero-fills the 16 bytes.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldmatrix_x4(uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3, uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// D += A * B for one m16n8k16 BF16 tile, FP32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float *d, const uint32_t *a, uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Byte offset of 16-byte chunk `c` of row `r` in a tile whose rows are 128
// bytes (64 BF16): chunks are XOR-swizzled by the row's low 3 bits so that
// ldmatrix reads of 8 consecutive rows hit 8 distinct bank groups.
__device__ __forceinline__ uint32_t swz128(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

// silu(g) * u with the fast reciprocal-based division (for g -> -inf the
// denominator overflows to +inf and the quotient is 0, the correct limit).
__device__ __forceinline__ float silu_mul(float g, float u) { return __fdividef(g, 1.0f + __expf(-g)) * u; }

}  // namespace pmpe
