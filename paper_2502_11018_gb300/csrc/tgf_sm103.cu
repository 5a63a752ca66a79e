// gv_tgf: the Token-Guided Fusion module of GRIFFIN's draft model (Section
// 4.2, Eqs. 6-8), bf16 on sm_103a, over R rows of features F and token
// embeddings x (d wide):
//
//   h = [F ; x] Wm^T + bm                   (Eq. 6)   GEMM, K = 2d, N = d
//   z = [N_h(h) ; N_x(x)] Wu^T + bu         (Eq. 7)   GEMM, K = 2d, N = e
//   o = silu(z) Wd^T + bd + h               (Eq. 8)   GEMM, K = e, N = d
//
// with N_h, N_x two layer norms of their own.  The three projections are the
// weight streams of gv_linear (tensor cores, split K, fp32 partial sums); the
// concatenation [F ; x] is never built (the GEMM reads its K range from two
// input blocks), and the bias, the two layer norms and the concatenation
// [N_h(h) ; N_x(x)] happen in one kernel after the first projection.  Each
// projection is either a cluster split-K launch (the splits reduced through
// distributed shared memory, the epilogue applied there) or a GEMM plus a
// reduce kernel, as gv_linear's planner picks; four to six launches.  The weights (4d^2 + 4de bytes) are the traffic.
#include "gv_internal.cuh"

namespace gv {

constexpr int TGF_THREADS = 512;
constexpr int TGF_MAXC = 2;              // 16-byte chunks per thread: d <= 8192

__device__ __forceinline__ void unpack8(const uint4 v, float* f) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        f[2 * e] = __uint_as_float(w[e] << 16);
        f[2 * e + 1] = __uint_as_float(w[e] & 0xffff0000u);
    }
}

__device__ __forceinline__ uint4 pack8(const float* f) {
    uint32_t pk[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        __nv_bfloat162 h2 = __floats2bfloat162_rn(f[2 * e], f[2 * e + 1]);
        pk[e] = *reinterpret_cast<uint32_t*>(&h2);
    }
    return make_uint4(pk[0], pk[1], pk[2], pk[3]);
}

// Sum of (a, b) over the CTA; red holds 2 * TGF_THREADS / 32 floats and is
// reused after a barrier.
__device__ __forceinline__ float2 block_sum2(float a, float b, float* red) {
    a = warp_sum(a);
    b = warp_sum(b);
    const int w = threadIdx.x >> 5;
    __syncthreads();                     // (red's previous use is over)
    constexpr int NW = TGF_THREADS / 32;
    if ((threadIdx.x & 31) == 0) {
        red[w] = a;
        red[NW + w] = b;
    }
    __syncthreads();
    float2 t = make_float2(0.f, 0.f);
#pragma unroll
    for (int k = 0; k < NW; ++k) {
        t.x += red[k];
        t.y += red[NW + k];
    }
    return t;
}

// One CTA per row r: h = sum of the K splits + bm, stored as bf16 (or, with
// KS == 0, h as the projection stored it, bias included); then the two
// layer norms (fp32, population variance, two passes over values held in
// registers) of the stored h and of x, written side by side as zin[r] =
// [N_h(h) ; N_x(x)] (2d wide), the next GEMM's input.
__global__ void __launch_bounds__(TGF_THREADS)
tgf_norm_kernel(const float* __restrict__ part, int KS, int rows, int d, const __nv_bfloat16* __restrict__ bm,
                const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ g_h,
                const __nv_bfloat16* __restrict__ b_h, const __nv_bfloat16* __restrict__ g_x,
                const __nv_bfloat16* __restrict__ b_x, float eps, __nv_bfloat16* h_out,
                __nv_bfloat16* __restrict__ zin) {
    __shared__ float red[2 * TGF_THREADS / 32];
    pdl_trigger();   // (early: see the split-K reduce note in gv_internal.cuh)
    pdl_wait();
    const int r = blockIdx.x, tid = threadIdx.x;
    float hv[TGF_MAXC][8], xv[TGF_MAXC][8];
#pragma unroll
    for (int q = 0; q < TGF_MAXC; ++q) {
        const int c = (tid + q * TGF_THREADS) * 8;
#pragma unroll
        for (int e = 0; e < 8; ++e) hv[q][e] = xv[q][e] = 0.f;
        if (c < d) {
            // KS == 0: h (bias included) was stored by the projection itself
            unpack8(*reinterpret_cast<const uint4*>((KS == 0 ? h_out + (size_t)r * d : bm) + c), hv[q]);
            unpack8(*reinterpret_cast<const uint4*>(x + (size_t)r * d + c), xv[q]);
        }
    }
    // all the chunks' split sums at once (loads in flight; the partials sit in L2)
#pragma unroll 4
    for (int ks = 0; ks < KS; ++ks) {
        const float* prow = part + ((size_t)ks * rows + r) * d;
#pragma unroll
        for (int q = 0; q < TGF_MAXC; ++q) {
            const int c = (tid + q * TGF_THREADS) * 8;
            if (c < d) {
                const float4 a0 = *reinterpret_cast<const float4*>(prow + c);
                const float4 a1 = *reinterpret_cast<const float4*>(prow + c + 4);
                hv[q][0] += a0.x; hv[q][1] += a0.y; hv[q][2] += a0.z; hv[q][3] += a0.w;
                hv[q][4] += a1.x; hv[q][5] += a1.y; hv[q][6] += a1.z; hv[q][7] += a1.w;
            }
        }
    }
    float sh = 0.f, sx = 0.f;
#pragma unroll
    for (int q = 0; q < TGF_MAXC; ++q) {
        const int c = (tid + q * TGF_THREADS) * 8;
        if (c >= d) break;
        if (KS > 0) {
            const uint4 hp = pack8(hv[q]);
            *reinterpret_cast<uint4*>(h_out + (size_t)r * d + c) = hp;
            unpack8(hp, hv[q]);                      // the stored (rounded) h
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            sh += hv[q][e];
            sx += xv[q][e];
        }
    }
    const float2 mean = block_sum2(sh, sx, red);
    const float mh = mean.x / (float)d, mx = mean.y / (float)d;
    float vh = 0.f, vx = 0.f;
#pragma unroll
    for (int q = 0; q < TGF_MAXC; ++q) {
        const int c = (tid + q * TGF_THREADS) * 8;
        if (c >= d) break;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float a = hv[q][e] - mh, b = xv[q][e] - mx;
            vh += a * a;
            vx += b * b;
        }
    }
    const float2 var = block_sum2(vh, vx, red);
    const float rh = rsqrtf(var.x / (float)d + eps), rx = rsqrtf(var.y / (float)d + eps);
#pragma unroll
    for (int q = 0; q < TGF_MAXC; ++q) {
        const int c = (tid + q * TGF_THREADS) * 8;
        if (c >= d) break;
        float g[8], b[8], o[8];
        unpack8(*reinterpret_cast<const uint4*>(g_h + c), g);
        unpack8(*reinterpret_cast<const uint4*>(b_h + c), b);
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = (hv[q][e] - mh) * rh * g[e] + b[e];
        *reinterpret_cast<uint4*>(zin + (size_t)r * 2 * d + c) = pack8(o);
        unpack8(*reinterpret_cast<const uint4*>(g_x + c), g);
        unpack8(*reinterpret_cast<const uint4*>(b_x + c), b);
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = (xv[q][e] - mx) * rx * g[e] + b[e];
        *reinterpret_cast<uint4*>(zin + (size_t)r * 2 * d + d + c) = pack8(o);
    }
}

static size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

// Workspace: [fp32 partial sums, the largest of the three GEMMs'] [zin bf16
// rows x 2d] [silu(z) bf16 rows x e].
size_t tgf_workspace_bytes(int rows, int d, int e) {
    size_t part = linear_workspace_bytes(rows, 2 * d, d);
    const size_t p2 = linear_workspace_bytes(rows, 2 * d, e), p3 = linear_workspace_bytes(rows, e, d);
    if (p2 > part) part = p2;
    if (p3 > part) part = p3;
    return al256(part) + al256((size_t)rows * 2 * d * 2) + al256((size_t)rows * e * 2);
}

int launch_tgf(const void* F, const void* x, int rows, int d, int e, const void* Wm, const void* bm,
               const void* g_h, const void* b_h, const void* g_x, const void* b_x, const void* Wu, const void* bu,
               const void* Wd, const void* bd, float eps, void* h_out, void* o_out, void* ws, cudaStream_t st) {
    size_t part = linear_workspace_bytes(rows, 2 * d, d);
    const size_t p2 = linear_workspace_bytes(rows, 2 * d, e), p3 = linear_workspace_bytes(rows, e, d);
    if (p2 > part) part = p2;
    if (p3 > part) part = p3;
    uint8_t* base = static_cast<uint8_t*>(ws);
    __nv_bfloat16* zin = reinterpret_cast<__nv_bfloat16*>(base + al256(part));
    __nv_bfloat16* s = reinterpret_cast<__nv_bfloat16*>(base + al256(part) + al256((size_t)rows * 2 * d * 2));

    // Eq. 6: h = [F ; x] Wm^T + bm, then both layer norms (Eq. 7's input)
    LinearOp m;
    m.x = F;
    m.x2 = x;
    m.k_split = d;
    m.W = Wm;
    m.rows = rows;
    m.K = 2 * d;
    m.n_out = d;
    m.bias = bm;
    m.out = h_out;
    m.ws = ws;
    int rc = launch_linear(m, st);
    if (rc != GV_OK) return rc;
    launch_pdl(tgf_norm_kernel, dim3(rows), dim3(TGF_THREADS), 0, st, static_cast<const float*>(nullptr), 0, rows, d,
               static_cast<const __nv_bfloat16*>(bm), static_cast<const __nv_bfloat16*>(x),
               static_cast<const __nv_bfloat16*>(g_h), static_cast<const __nv_bfloat16*>(b_h),
               static_cast<const __nv_bfloat16*>(g_x), static_cast<const __nv_bfloat16*>(b_x), eps,
               static_cast<__nv_bfloat16*>(h_out), zin);
    rc = check_launch("tgf_norm_kernel");
    if (rc != GV_OK) return rc;

    // Eq. 7 expansion with the SiLU of Eq. 8 in its epilogue
    LinearOp u;
    u.x = zin;
    u.W = Wu;
    u.rows = rows;
    u.K = 2 * d;
    u.n_out = e;
    u.epi = GV_LINEAR_SILU;
    u.bias = bu;
    u.out = s;
    u.ws = ws;
    rc = launch_linear(u, st);
    if (rc != GV_OK) return rc;

    // Eq. 8: down projection, bias and the residual h
    LinearOp dn;
    dn.x = s;
    dn.W = Wd;
    dn.rows = rows;
    dn.K = e;
    dn.n_out = d;
    dn.epi = GV_LINEAR_ADD;
    dn.bias = bd;
    dn.residual = h_out;
    dn.out = o_out;
    dn.ws = ws;
    return launch_linear(dn, st);
}

}  // namespace gv
