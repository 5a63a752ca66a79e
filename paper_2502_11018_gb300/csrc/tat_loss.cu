// gv_tat_loss: the token-alignable training objective of the draft model
// (GRIFFIN Section 4.1, Eqs. 2-5; per-step loss of the Implementation Details
// appendix), one training pass n over a batch of sequences.
//
// Per position t of sequence b (row r = b * T + t):
//   mbar_t = 1 iff the ground-truth token x_t is among the top-k draft logits
//            (ties toward the lower id: fewer than k tokens v with
//            logit_v > logit_x, or logit_v == logit_x and v < x);
//   ell_t  = lam_tok * (logsumexp(logits_t) - logit_x) + lam_feat * |Fd_t - Ft_t|_1;
// then per sequence, with the chain alignment mask of Eq. 3,
//   m_t = prod_{j=1}^{n-1} mbar^(j)_{t-n+j}  (0 for t < n-1; 1 everywhere for n = 1),
//   L_b = sum_t m_t ell_t / sum_t m_t        (0 when no position is aligned).
//
// tat_row_kernel: one CTA per row streams the row's V logits once (16-byte
// loads), keeping a running max and a rescaled sum of exponentials, and counts
// the logits ahead of the target's, all in one pass, then the feature rows;
// one CTA-wide reduction.  The target logit is read first, so the count needs
// no second pass.  HBM-bound: V * sizeof(logit) + 2 * H * sizeof(feature)
// bytes per row.
// tat_reduce_kernel: one CTA per sequence forms m_t from the earlier passes'
// predictable masks and reduces the masked sum (in double).
#include "gv_internal.cuh"

namespace gv {

constexpr int TAT_THREADS = 256;
constexpr float TAT_LOG2E = 1.4426950408889634f;
constexpr float TAT_LN2 = 0.6931471805599453f;

__device__ __forceinline__ float tat_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// 16 bytes of a row as floats: 4 fp32 or 8 bf16 values.
template <typename T> struct Vec16;
template <> struct Vec16<float> {
    static constexpr int N = 4;
    __device__ static void load(const float* p, float* o) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(p));
        o[0] = v.x; o[1] = v.y; o[2] = v.z; o[3] = v.w;
    }
};
template <> struct Vec16<__nv_bfloat16> {
    static constexpr int N = 8;
    __device__ static void load(const __nv_bfloat16* p, float* o) {
        const uint4 v = __ldcs(reinterpret_cast<const uint4*>(p));
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            o[2 * e] = __uint_as_float(w[e] << 16);
            o[2 * e + 1] = __uint_as_float(w[e] & 0xffff0000u);
        }
    }
};

// Running (max, sum of 2^(v - max)) in the log2 domain, and the count of
// logits ahead of the target.
struct RowAcc {
    float m;   // max * log2(e)
    float s;
    int ahead;
};

__device__ __forceinline__ void acc_values(RowAcc& a, const float* v, int n, int idx0, float tl, int x) {
    float mv = -INFINITY;
    for (int e = 0; e < n; ++e) mv = fmaxf(mv, v[e]);
    const float m2 = mv * TAT_LOG2E;
    if (m2 > a.m) {
        a.s *= tat_exp2(a.m - m2);   // 0 while a.m = -inf
        a.m = m2;
    }
    for (int e = 0; e < n; ++e) {
        a.s += tat_exp2(fmaf(v[e], TAT_LOG2E, -a.m));
        a.ahead += (v[e] > tl || (v[e] == tl && idx0 + e < x)) ? 1 : 0;
    }
}

__device__ __forceinline__ void acc_merge(RowAcc& a, const RowAcc& b) {
    const float m = fmaxf(a.m, b.m);
    if (m == -INFINITY) {
        a.ahead += b.ahead;
        return;
    }
    a.s = a.s * tat_exp2(a.m - m) + b.s * tat_exp2(b.m - m);
    a.m = m;
    a.ahead += b.ahead;
}

template <typename TL, typename TF, bool VL, bool VF>
__global__ void __launch_bounds__(TAT_THREADS)
tat_row_kernel(const TL* __restrict__ logits, const int32_t* __restrict__ tokens,
               const TF* __restrict__ fd, const TF* __restrict__ ft, int V, int H, int k,
               float lam_tok, float lam_feat, uint8_t* __restrict__ mbar, float* __restrict__ ell) {
    __shared__ float s_tl;
    __shared__ int s_bad;
    __shared__ RowAcc s_acc[TAT_THREADS / 32];
    __shared__ float s_l1[TAT_THREADS / 32];
    pdl_wait();
    pdl_trigger();
    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const TL* row = logits + (size_t)r * V;
    if (tid == 0) {
        const int x = tokens[r];
        const bool bad = x < 0 || x >= V;
        s_bad = bad ? 1 : 0;
        s_tl = bad ? 0.f : static_cast<float>(row[bad ? 0 : x]);
    }
    __syncthreads();
    const int x = tokens[r];
    const float tl = s_tl;
    RowAcc a{-INFINITY, 0.f, 0};
    if (VL) {
        constexpr int N = Vec16<TL>::N;
        for (int i = tid * N; i < V; i += TAT_THREADS * N) {
            float v[N];
            Vec16<TL>::load(row + i, v);
            acc_values(a, v, N, i, tl, x);
        }
    } else {
        for (int i = tid; i < V; i += TAT_THREADS) {
            const float v = static_cast<float>(row[i]);
            acc_values(a, &v, 1, i, tl, x);
        }
    }
    float l1 = 0.f;
    const TF* a_row = fd + (size_t)r * H;
    const TF* b_row = ft + (size_t)r * H;
    if (VF) {
        constexpr int N = Vec16<TF>::N;
        for (int i = tid * N; i < H; i += TAT_THREADS * N) {
            float u[N], w[N];
            Vec16<TF>::load(a_row + i, u);
            Vec16<TF>::load(b_row + i, w);
#pragma unroll
            for (int e = 0; e < N; ++e) l1 += fabsf(u[e] - w[e]);
        }
    } else {
        for (int i = tid; i < H; i += TAT_THREADS)
            l1 += fabsf(static_cast<float>(a_row[i]) - static_cast<float>(b_row[i]));
    }
    // CTA reduction: warps by shuffles, then the warp results in shared memory.
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        RowAcc b{__shfl_xor_sync(FULL, a.m, o), __shfl_xor_sync(FULL, a.s, o),
                 __shfl_xor_sync(FULL, a.ahead, o)};
        acc_merge(a, b);
        l1 += __shfl_xor_sync(FULL, l1, o);
    }
    if (lane == 0) {
        s_acc[warp] = a;
        s_l1[warp] = l1;
    }
    __syncthreads();
    if (tid == 0) {
        RowAcc t = s_acc[0];
        float f = s_l1[0];
        for (int w = 1; w < TAT_THREADS / 32; ++w) {
            acc_merge(t, s_acc[w]);
            f += s_l1[w];
        }
        const float lse = (t.m + log2f(t.s)) * TAT_LN2;
        if (s_bad) {
            mbar[r] = 0;
            ell[r] = NAN;
        } else {
            mbar[r] = t.ahead < k ? 1 : 0;
            ell[r] = lam_tok * (lse - tl) + lam_feat * f;
        }
    }
}

__global__ void __launch_bounds__(TAT_THREADS)
tat_reduce_kernel(int B, int T, int n, const uint8_t* __restrict__ mbar_prev,
                  const float* __restrict__ ell, uint8_t* __restrict__ mask,
                  float* __restrict__ seq_loss) {
    __shared__ double s_num[TAT_THREADS / 32], s_den[TAT_THREADS / 32];
    __shared__ int s_nan[TAT_THREADS / 32];
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    double num = 0.0, den = 0.0;
    int nan = 0;
    for (int t = tid; t < T; t += TAT_THREADS) {
        int m = 1;
        if (n > 1) {
            m = t - n + 1 >= 0 ? 1 : 0;
            for (int j = 1; j < n && m; ++j)
                m = mbar_prev[((size_t)(j - 1) * B + b) * T + (t - n + j)] ? 1 : 0;
        }
        const float e = ell[(size_t)b * T + t];
        mask[(size_t)b * T + t] = (uint8_t)m;
        nan |= e != e ? 1 : 0;
        if (m) {
            num += (double)e;
            den += 1.0;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        num += __shfl_xor_sync(FULL, num, o);
        den += __shfl_xor_sync(FULL, den, o);
        nan |= __shfl_xor_sync(FULL, nan, o);
    }
    if (lane == 0) {
        s_num[warp] = num;
        s_den[warp] = den;
        s_nan[warp] = nan;
    }
    __syncthreads();
    if (tid == 0) {
        double tn = 0.0, td = 0.0;
        int any_nan = 0;
        for (int w = 0; w < TAT_THREADS / 32; ++w) {
            tn += s_num[w];
            td += s_den[w];
            any_nan |= s_nan[w];
        }
        // A token outside the vocabulary anywhere in the sequence makes its
        // loss NaN, so that bad data cannot pass silently.
        seq_loss[b] = any_nan ? NAN : (td > 0.0 ? (float)(tn / td) : 0.f);
    }
}

template <typename TL, typename TF>
static int launch_rows(const void* logits, const int32_t* tokens, const void* fd, const void* ft, int R,
                       int V, int H, int k, float lam_tok, float lam_feat, uint8_t* mbar, float* ell,
                       cudaStream_t st) {
    const bool vl = ((size_t)V * sizeof(TL)) % 16 == 0 && aligned16(logits);
    const bool vf = ((size_t)H * sizeof(TF)) % 16 == 0 && aligned16(fd) && aligned16(ft);
    const TL* L = static_cast<const TL*>(logits);
    const TF* A = static_cast<const TF*>(fd);
    const TF* Bf = static_cast<const TF*>(ft);
    const dim3 grid(R), block(TAT_THREADS);
    if (vl && vf)
        launch_pdl(tat_row_kernel<TL, TF, true, true>, grid, block, 0, st, L, tokens, A, Bf, V, H, k, lam_tok,
                   lam_feat, mbar, ell);
    else if (vl)
        launch_pdl(tat_row_kernel<TL, TF, true, false>, grid, block, 0, st, L, tokens, A, Bf, V, H, k, lam_tok,
                   lam_feat, mbar, ell);
    else if (vf)
        launch_pdl(tat_row_kernel<TL, TF, false, true>, grid, block, 0, st, L, tokens, A, Bf, V, H, k, lam_tok,
                   lam_feat, mbar, ell);
    else
        launch_pdl(tat_row_kernel<TL, TF, false, false>, grid, block, 0, st, L, tokens, A, Bf, V, H, k,
                   lam_tok, lam_feat, mbar, ell);
    return check_launch("tat_row_kernel");
}

int launch_tat_loss(const void* logits, int logits_dt, const int32_t* tokens, const void* fd,
                    const void* ft, int feat_dt, int B, int T, int V, int H, int k, int n,
                    const uint8_t* mbar_prev, float lam_tok, float lam_feat, uint8_t* mbar,
                    uint8_t* mask, float* ell, float* seq_loss, cudaStream_t st) {
    const int R = B * T;
    int rc;
    if (logits_dt == GV_F32)
        rc = feat_dt == GV_F32
                 ? launch_rows<float, float>(logits, tokens, fd, ft, R, V, H, k, lam_tok, lam_feat, mbar, ell, st)
                 : launch_rows<float, __nv_bfloat16>(logits, tokens, fd, ft, R, V, H, k, lam_tok, lam_feat, mbar,
                                                     ell, st);
    else
        rc = feat_dt == GV_F32
                 ? launch_rows<__nv_bfloat16, float>(logits, tokens, fd, ft, R, V, H, k, lam_tok, lam_feat, mbar,
                                                     ell, st)
                 : launch_rows<__nv_bfloat16, __nv_bfloat16>(logits, tokens, fd, ft, R, V, H, k, lam_tok, lam_feat,
                                                             mbar, ell, st);
    if (rc != GV_OK) return rc;
    launch_pdl(tat_reduce_kernel, dim3(B), dim3(TAT_THREADS), 0, st, B, T, n, mbar_prev, ell, mask, seq_loss);
    return check_launch("tat_reduce_kernel");
}

}  // namespace gv
