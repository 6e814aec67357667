// Stages 3 and 4 of the layer: the grouped SwiGLU expert GEMMs.
//
//   gate/up:  for every expert e with n_e > 0 rows,  g = A_e W_gate,e^T,
//             u = A_e W_up,e^T (FP32), act = bf16(silu(g) * u)
//   down:     y = bf16(w_row * (act_e W_down,e^T))
//
// Groups are the E routed experts (rows of the dispatch order) plus, when the
// layer has shared experts, one dense group of all T tokens whose gate/up
// weights are the E_sh experts side by side ([E_sh * I, H]) and whose down
// projection sums the E_sh experts' outputs in one FP32 accumulator.
//
// A persistent grid walks a tile list built on the device from the dispatch
// offsets, so no row count ever goes back to the host and empty experts
// contribute no tile.  Every tile of N-tile 0 adds the rows it actually
// processed to the execution audit (exec_rows / exec_tiles / exec_priv_rows
// per token / shared_rows): counts observed where the expert runs,
// independent of the router's route log.
#include "pmpe_internal.cuh"

namespace pmpe {
namespace {

constexpr int BM = 64;          // rows per tile
constexpr int BK = 64;          // K per pipeline stage (one 128-byte row segment)
constexpr int kStages = 3;
constexpr int kThreads = 128;   // 4 warps as 2 (rows) x 2 (columns)
constexpr int kBRows = 128;     // gate/up: 64 gate + 64 up rows; down: 128 output columns
constexpr int kStageBytes = (BM + kBRows) * 128;
constexpr int kSmem = kStages * kStageBytes;
constexpr int kMaxGroups = 2 * kMaxPool + 1;

enum { kGateUp = 0, kDown = 1 };

struct GemmParams {
    int mode;
    int E, E_pub, E_sh, T, H, I, R;
    const uint32_t *offsets;
    const bf16 *A_routed, *A_shared;
    const bf16 *B0[3], *B1[3];  // [pool]: gate/up (gate/up mode) or down (B1 unused)
    bf16 *C_routed, *C_shared;
    const float *w_of_slot;
    const int32_t *tok_of_slot;
    uint32_t *exec_rows, *exec_tiles, *exec_priv_rows, *shared_rows;
};

struct Group {
    int rows, row_base, K, N, lda, ldc;
};

__device__ __forceinline__ Group group_info(const GemmParams &p, int g)
{
    Group G;
    const bool shared = g >= p.E;
    if (shared) {
        G.rows = p.T;
        G.row_base = 0;
    } else {  // clamped to [0, R): the offsets are a prefix sum, this only guards against a corrupt workspace
        const int b = min((int)p.offsets[g], p.R), e = min(max((int)p.offsets[g + 1], b), p.R);
        G.rows = e - b;
        G.row_base = b;
    }
    if (p.mode == kGateUp) {
        G.K = p.H;
        G.N = shared ? p.E_sh * p.I : p.I;
        G.lda = p.H;
        G.ldc = G.N;
    } else {
        G.K = shared ? p.E_sh * p.I : p.I;
        G.N = p.H;
        G.lda = G.K;
        G.ldc = p.H;
    }
    return G;
}

// Address of B row n (output column), K offset kk, for group g.
__device__ __forceinline__ const bf16 *b_row(const GemmParams &p, int g, int which, int n, int kk)
{
    const bool shared = g >= p.E;
    const int q = shared ? 2 : (g < p.E_pub ? 0 : 1);
    const int ei = shared ? 0 : (q == 0 ? g : g - p.E_pub);
    if (p.mode == kGateUp) {
        const bf16 *W = which ? p.B1[q] : p.B0[q];
        return W + ((size_t)ei * p.I + n) * p.H + kk;  // shared: n spans E_sh * I rows
    }
    if (shared) {
        const int s = kk / p.I;
        return p.B0[2] + ((size_t)s * p.H + n) * p.I + (kk - s * p.I);
    }
    return p.B0[q] + ((size_t)ei * p.H + n) * p.I + kk;
}

__global__ void __launch_bounds__(kThreads) grouped_gemm_kernel(const GemmParams p)
{
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int prefix[kMaxGroups + 1];
    __shared__ int counts_s[kMaxGroups];

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int G = p.E + (p.E_sh > 0 ? 1 : 0);
    const int BN = p.mode == kGateUp ? 64 : 128;

    // tile list: prefix of (m tiles x n tiles) over the groups
    for (int g = tid; g < G; g += kThreads) {
        const Group gi = group_info(p, g);
        counts_s[g] = ((gi.rows + BM - 1) / BM) * (gi.N / BN);
    }
    __syncthreads();
    if (warp == 0) {
        int carry = 0;
        for (int base = 0; base < G; base += 32) {
            int v = base + lane < G ? counts_s[base + lane] : 0;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(~0u, v, off);
                if (lane >= off) v += y;
            }
            if (base + lane < G) prefix[base + lane + 1] = carry + v;
            carry += __shfl_sync(~0u, v, 31);
        }
        if (lane == 0) prefix[0] = 0;
    }
    __syncthreads();
    const int total = prefix[G];

    const int wm = warp >> 1, wn = warp & 1;
    for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
        int lo = 0, hi = G - 1;  // last g with prefix[g] <= tile
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (prefix[mid] <= tile) lo = mid; else hi = mid - 1;
        }
        const int g = lo;
        const Group gi = group_info(p, g);
        const int mtiles = (gi.rows + BM - 1) / BM;
        const int local = tile - prefix[g];
        const int n_tile = local / mtiles, m_tile = local - n_tile * mtiles;
        const int m0 = m_tile * BM, n0 = n_tile * BN;
        const int valid = min(BM, gi.rows - m0);
        const bool shared = g >= p.E;
        const bf16 *A = (shared ? p.A_shared : p.A_routed) + (size_t)(gi.row_base + m0) * gi.lda;

        auto load_stage = [&](int st, int kb) {
            const uint32_t sA = smem_u32(smem + st * kStageBytes);
            const uint32_t sB = sA + BM * 128;
            const int kk = kb * BK;
            for (int i = tid; i < BM * 8; i += kThreads) {
                const int r = i >> 3, c = i & 7;
                const bool ok = r < valid;
                cp_async16(sA + swz128(r, c), A + (size_t)(ok ? r : 0) * gi.lda + kk + c * 8, ok ? 16 : 0);
            }
            for (int i = tid; i < kBRows * 8; i += kThreads) {
                const int r = i >> 3, c = i & 7;
                const bf16 *src = p.mode == kGateUp ? b_row(p, g, r >= 64, n0 + (r & 63), kk)
                                                    : b_row(p, g, 0, n0 + r, kk);
                cp_async16(sB + swz128(r, c), src + c * 8, 16);
            }
        };

        float acc[2][8][4];
#pragma unroll
        for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int b = 0; b < 8; ++b) acc[a][b][0] = acc[a][b][1] = acc[a][b][2] = acc[a][b][3] = 0.f;

        const int nkb = gi.K / BK;
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
            const uint32_t sA = smem_u32(smem + (kb % kStages) * kStageBytes);
            const uint32_t sB = sA + BM * 128;
#pragma unroll
            for (int ks = 0; ks < BK / 16; ++ks) {
                uint32_t a[2][4];
#pragma unroll
                for (int mi = 0; mi < 2; ++mi)
                    ldmatrix_x4(a[mi][0], a[mi][1], a[mi][2], a[mi][3],
                                sA + swz128(wm * 32 + mi * 16 + (lane & 15), ks * 2 + (lane >> 4)));
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    // B rows of n8 tiles 2np and 2np+1
                    const int brow = p.mode == kGateUp ? (np < 2 ? wn * 32 + np * 16 : 64 + wn * 32 + (np - 2) * 16)
                                                       : wn * 64 + np * 16;
                    uint32_t b0, b1, b2, b3;
                    ldmatrix_x4(b0, b1, b2, b3,
                                sB + swz128(brow + (lane & 7) + ((lane >> 4) << 3), ks * 2 + ((lane >> 3) & 1)));
#pragma unroll
                    for (int mi = 0; mi < 2; ++mi) {
                        mma_bf16_16816(acc[mi][2 * np], a[mi], b0, b1);
                        mma_bf16_16816(acc[mi][2 * np + 1], a[mi], b2, b3);
                    }
                }
            }
        }
        cp_async_wait<0>();
        __syncthreads();  // all warps done with the stages before the next tile reloads them

        // ---- epilogue
        bf16 *C = (shared ? p.C_shared : p.C_routed) + (size_t)(gi.row_base + m0) * gi.ldc + n0;
        if (p.mode == kGateUp) {
#pragma unroll
            for (int mi = 0; mi < 2; ++mi)
#pragma unroll
                for (int nt = 0; nt < 4; ++nt) {
                    const int col = wn * 32 + nt * 8 + 2 * (lane & 3);
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int r = wm * 32 + mi * 16 + (lane >> 2) + 8 * h;
                        if (r < valid) {
                            const float *gg = &acc[mi][nt][2 * h];
                            const float *uu = &acc[mi][nt + 4][2 * h];
                            *reinterpret_cast<uint32_t *>(C + (size_t)r * gi.ldc + col) =
                                pack_bf16x2(silu_mul(gg[0], uu[0]), silu_mul(gg[1], uu[1]));
                        }
                    }
                }
            // execution audit, from the rows this tile processed
            if (!shared && n_tile == 0) {
                if (tid == 0) {
                    if (p.exec_rows) atomicAdd(&p.exec_rows[g], (unsigned)valid);
                    if (p.exec_tiles) atomicAdd(&p.exec_tiles[g], 1u);
                }
                if (g >= p.E_pub && p.exec_priv_rows && tid < valid)
                    atomicAdd(&p.exec_priv_rows[p.tok_of_slot[gi.row_base + m0 + tid]], 1u);
            }
            if (shared && p.shared_rows && tid == 0 && (n0 % p.I) == 0) atomicAdd(p.shared_rows, (unsigned)valid);
        } else {
#pragma unroll
            for (int mi = 0; mi < 2; ++mi)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int r = wm * 32 + mi * 16 + (lane >> 2) + 8 * h;
                    if (r < valid) {
                        const float sc = shared ? 1.f : p.w_of_slot[gi.row_base + m0 + r];
#pragma unroll
                        for (int nt = 0; nt < 8; ++nt) {
                            const int col = wn * 64 + nt * 8 + 2 * (lane & 3);
                            *reinterpret_cast<uint32_t *>(C + (size_t)r * gi.ldc + col) =
                                pack_bf16x2(acc[mi][nt][2 * h] * sc, acc[mi][nt][2 * h + 1] * sc);
                        }
                    }
                }
        }
    }
}

cudaError_t launch_gemm(const Ctx &c, int mode)
{
    const Shape &s = c.s;
    GemmParams p;
    p.mode = mode;
    p.E = s.E(); p.E_pub = s.E_pub; p.E_sh = s.E_sh; p.T = s.T; p.H = s.H; p.I = s.I; p.R = s.T * s.k;
    p.offsets = c.offsets;
    if (mode == kGateUp) {
        p.A_routed = c.a_perm; p.A_shared = c.hidden;
        for (int q = 0; q < 3; ++q) { p.B0[q] = c.gate[q]; p.B1[q] = c.up[q]; }
        p.C_routed = c.act; p.C_shared = c.act_sh;
    } else {
        p.A_routed = c.act; p.A_shared = c.act_sh;
        for (int q = 0; q < 3; ++q) { p.B0[q] = c.down[q]; p.B1[q] = nullptr; }
        p.C_routed = c.y; p.C_shared = c.y_sh;
    }
    p.w_of_slot = c.w_of_slot;
    p.tok_of_slot = c.tok_of_slot;
    p.exec_rows = c.audit.exec_rows;
    p.exec_tiles = c.audit.exec_tiles;
    p.exec_priv_rows = c.audit.exec_priv_rows;
    p.shared_rows = c.audit.shared_rows;
    cudaError_t err = cudaFuncSetAttribute(grouped_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
    if (err != cudaSuccess) return err;
    grouped_gemm_kernel<<<c.num_sms * 2, kThreads, kSmem, c.stream>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gateup(const Ctx &c) { return launch_gemm(c, kGateUp); }
cudaError_t launch_down(const Ctx &c) { return launch_gemm(c, kDown); }

}  // namespace pmpe
