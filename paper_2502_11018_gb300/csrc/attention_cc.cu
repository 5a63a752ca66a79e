// gv_rope_table, and the fp32 path of gv_verify_attention: RoPE prologue,
// CUDA-core (FFMA) split-KV tree attention and split combine.  fp32 operands
// stay on CUDA cores: tf32 tensor-core inputs would round them to 10-bit
// mantissas, outside the 1e-4 relative tolerance fp32 results are held to.
//
// GRIFFIN Section 3: all draft tokens are verified in one target forward
// pass; in each attention layer node i attends to the cached prefix and to
// the tree nodes on its own root chain (Section 4.1: a rejected token takes
// its subtree with it, so exactly the ancestor set is visible).
//
// Work split (flash-decoding style): the keys of sequence b, KV head g are cut
// into splits of KPS prefix keys plus one final split holding the N tree keys
// (masked per query row by the ancestor bitmask).  Every split produces, per
// query row, the running max m, the sum l of exp(s - m) and the unnormalised
// output; attn_combine_kernel rescales and sums the splits.  Query rows of one
// KV head are its G query heads x N nodes (row = head_in_group * N + node), so
// every K/V tile is read once for all heads that share it.
#include <cmath>

#include "gv_internal.cuh"
#include "attention.cuh"

namespace gv {

// -------------------------------------------------------------- rope table --
// One thread per (sequence, node, frequency j < d/2).  The frequencies
// base^(-2j/d) arrive from the host in double (one pow per frequency and
// call); the angle a = pos * base^(-2j/d) is formed in double and reduced
// modulo 2 pi there (2 pi as the sum of two doubles, each product taken in a
// fused multiply-add, so a - k 2pi_hi is rounded once), so r = a - 2 pi k in
// [-pi, pi] keeps double accuracy.  r = r_hi + r_lo in two
// floats; cos and sin of r_hi in fp32 and one first-order step in r_lo give
// cos(r), sin(r) to a few fp32 ulps, stored as fp32 (cos, sin).  (Double
// sin/cos would cost a hundred fp64 operations per thread.)
struct RopeFreqs {
    double theta[128];
};

__global__ void __launch_bounds__(64)
rope_table_kernel(const int32_t* __restrict__ pos, int B, int N, int half, RopeFreqs f,
                  float2* __restrict__ rope) {
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    const int j = idx % half;
    const double theta = f.theta[j];
    pdl_wait();
    pdl_trigger();
    if (idx >= B * N * half) return;
    const double a = (double)pos[idx / half] * theta;
    constexpr double kTwoPiHi = 6.283185307179586;            // 2 pi rounded to double
    constexpr double kTwoPiLo = 2.4492935982947064e-16;       // 2 pi - kTwoPiHi
    constexpr double kInvTwoPi = 0.15915494309189535;
    const double k = rint(a * kInvTwoPi);
    const double r = fma(-k, kTwoPiLo, fma(-k, kTwoPiHi, a));
    const float rh = (float)r, rl = (float)(r - (double)rh);
    float sh, ch;
    sincosf(rh, &sh, &ch);
    rope[idx] = make_float2(fmaf(-sh, rl, ch), fmaf(ch, rl, sh));
}

int launch_rope_table(const int32_t* pos, int B, int N, int d, float base, float* rope,
                      cudaStream_t st) {
    const int half = d / 2, total = B * N * half;
    RopeFreqs f{};
    for (int j = 0; j < half; ++j) f.theta[j] = std::pow((double)base, -2.0 * (double)j / (double)d);
    launch_pdl(rope_table_kernel, dim3((total + 63) / 64), dim3(64), 0, st, pos, B, N, half, f,
               reinterpret_cast<float2*>(rope));
    return check_launch("rope_table_kernel");
}

// ---------------------------------------------------------------- prologue --
// fp32 path: one thread per (sequence, node, frequency, head) rotates that
// frequency's pair of one query head (into the q_rot workspace, grouped by
// KV head) or of one key head (into the tree K scratch, copying v with it).
__global__ void __launch_bounds__(128)
rope_tree_f32_kernel(const float* __restrict__ q, const float* __restrict__ k_new,
                     const float* __restrict__ v_new, const float2* __restrict__ rope, int B, int N,
                     int Hq, int Hkv, int d, float* __restrict__ q_rot, float* __restrict__ treeK,
                     float* __restrict__ treeV, int q_rows_pad) {
    pdl_wait();
    pdl_trigger();
    const int half = d >> 1;
    const int H = Hq + Hkv;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)B * N * half * H) return;
    const int hh = (int)(idx % H);
    const long long pidx = idx / H;                 // (b, i, j)
    const int j = (int)(pidx % half);
    const int i = (int)((pidx / half) % N);
    const int b = (int)(pidx / ((long long)half * N));
    const float2 r = rope[pidx];
    const float c = r.x, s = r.y;
    const int G = Hq / Hkv;
    if (hh < Hq) {
        const int h = hh;
        const size_t src = (((size_t)b * N + i) * Hq + h) * d;
        const float x0 = q[src + j], x1 = q[src + j + half];
        const int g = h / G, hl = h % G;
        const size_t dst = (((size_t)b * Hkv + g) * q_rows_pad + (size_t)hl * N + i) * d;
        q_rot[dst + j] = x0 * c - x1 * s;
        q_rot[dst + j + half] = x1 * c + x0 * s;
    } else {
        const int g = hh - Hq;
        const size_t src = (((size_t)b * N + i) * Hkv + g) * d;
        const size_t dst = (((size_t)b * Hkv + g) * N + i) * d;
        const float x0 = k_new[src + j], x1 = k_new[src + j + half];
        const float v0 = v_new[src + j], v1 = v_new[src + j + half];
        treeK[dst + j] = x0 * c - x1 * s;
        treeK[dst + j + half] = x1 * c + x0 * s;
        treeV[dst + j] = v0;
        treeV[dst + j + half] = v1;
    }
}

int launch_rope_tree_f32(const AttnArgs& a, cudaStream_t st) {
    const long long total = (long long)a.B * a.N * (a.d / 2) * (a.Hq + a.Hkv);
    launch_pdl(rope_tree_f32_kernel, dim3((unsigned)((total + 127) / 128)), dim3(128), 0, st,
        static_cast<const float*>(a.q), static_cast<const float*>(a.k_new),
        static_cast<const float*>(a.v_new), reinterpret_cast<const float2*>(a.rope), a.B, a.N, a.Hq,
        a.Hkv, a.d, static_cast<float*>(a.q_rot), static_cast<float*>(a.treeK),
        static_cast<float*>(a.treeV), a.q_rows_pad);
    return check_launch("rope_tree_f32_kernel");
}

// ----------------------------------------------------------------- combine --
// One warp per output row (b, node, head): out = sum_s e^{m_s - M} o_s / sum_s e^{m_s - M} l_s.
// Lane s reads split s's (m, l) (32 splits per pass), so the splits' loads are
// in flight together; the partial rows follow four splits at a time.
template <typename T, int D>
__global__ void __launch_bounds__(256)
attn_combine_kernel(const float* __restrict__ part_o, const float* __restrict__ part_ml, int B,
                    int N, int Hq, int Hkv, int nsplit, int R, T* __restrict__ out) {
    pdl_wait();
    pdl_trigger();
    const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= B * N * Hq) return;
    const int h = w % Hq, i = (w / Hq) % N, b = w / (Hq * N);
    const int G = Hq / Hkv, g = h / G, hl = h % G;
    const int r = hl * N + i;
    const size_t bg = (size_t)b * Hkv + g;
    float M = -INFINITY;
    for (int s0 = 0; s0 < nsplit; s0 += 32)
        if (s0 + lane < nsplit) M = fmaxf(M, part_ml[((bg * nsplit + s0 + lane) * R + r) * 2]);
    M = warp_max(M);
    float L = 0.f;
    float acc[D / 32] = {};
    for (int s0 = 0; s0 < nsplit; s0 += 32) {
        const int sl = s0 + lane;
        float wgt = 0.f;
        if (sl < nsplit) {
            const size_t pr = (bg * nsplit + sl) * R + r;
            const float m = part_ml[pr * 2];
            if (m != -INFINITY) {
                wgt = __expf(m - M);
                L += wgt * part_ml[pr * 2 + 1];
            }
        }
        const int cnt = min(32, nsplit - s0);
#pragma unroll 4
        for (int t = 0; t < cnt; ++t) {
            const float wt = __shfl_sync(FULL, wgt, t);
            if (wt == 0.f) continue;
            const float* po = part_o + ((bg * nsplit + s0 + t) * R + r) * D;
#pragma unroll
            for (int j = 0; j < D / 32; ++j) acc[j] = fmaf(wt, po[lane + 32 * j], acc[j]);
        }
    }
    L = warp_sum(L);
    const float inv = 1.0f / L;
    T* o = out + (((size_t)b * N + i) * Hq + h) * D;
#pragma unroll
    for (int j = 0; j < D / 32; ++j) o[lane + 32 * j] = from_f32<T>(acc[j] * inv);
}

int launch_attn_combine_f32(const AttnArgs& a, cudaStream_t st) {
    const int warps = a.B * a.N * a.Hq;
    const int blocks = (warps * 32 + 255) / 256;
    float* out = static_cast<float*>(a.out);
    if (a.d == 128)
        launch_pdl(attn_combine_kernel<float, 128>, dim3(blocks), dim3(256), 0, st, a.part_o, a.part_ml, a.B, a.N,
                   a.Hq, a.Hkv, a.nsplit, a.R, out);
    else
        launch_pdl(attn_combine_kernel<float, 64>, dim3(blocks), dim3(256), 0, st, a.part_o, a.part_ml, a.B, a.N,
                   a.Hq, a.Hkv, a.nsplit, a.R, out);
    return check_launch("attn_combine_kernel");
}

// -------------------------------------------------------- CUDA-core splits --
// Block = (sequence, KV head, chunk of ROWS query rows) x split, 256 threads:
// TPR = 256 / ROWS threads per query row, each scoring KPT = 64 / TPR keys of
// a 64-key tile (a whole split: one round of loads per block) and owning
// D / TPR output columns (c = lane_in_row + TPR j, so a row's threads hit
// different banks).  ROWS = 16 when the unit has at most 16 query rows (small
// workloads: every thread has a row), else 64.
constexpr int CC_KEYS = 64;

template <typename T, int D, int ROWS>
__global__ void __launch_bounds__(256)
attn_cc_kernel(AttnArgs a) {
    static_assert(sizeof(T) == 4, "the CUDA-core attention stages fp32 rows");
    constexpr int TPR = 256 / ROWS, KPT = CC_KEYS / TPR, CPT = D / TPR;
    extern __shared__ float smem[];
    float* sQ = smem;                          // [ROWS][D+1]
    float* sK = sQ + ROWS * (D + 1);           // [CC_KEYS][D+1]
    float* sV = sK + CC_KEYS * (D + 1);        // [CC_KEYS][D+1]
    float* sS = sV + CC_KEYS * (D + 1);        // [ROWS][CC_KEYS + 1]
    pdl_wait();
    pdl_trigger();
    const int nrc = (a.R + ROWS - 1) / ROWS;
    const int bg = blockIdx.x / nrc, rc = blockIdx.x % nrc;
    const int b = bg / a.Hkv;
    const int split = blockIdx.y;
    const int P = min(max(a.prefix_len[b], 0), a.S_max);
    const bool tree = split == a.nsplit - 1;
    const int k_lo = tree ? 0 : split * a.kps;
    const int k_hi = tree ? a.N : min(P, k_lo + a.kps);
    const int tid = threadIdx.x, row = tid / TPR, kg = tid % TPR;
    const int r = rc * ROWS + row;
    float* po = a.part_o + ((size_t)bg * a.nsplit + split) * a.R * D;
    float* pml = a.part_ml + ((size_t)bg * a.nsplit + split) * a.R * 2;
    if (k_lo >= k_hi) {
        if (r < a.R) {
            for (int j = 0; j < CPT; ++j) po[(size_t)r * D + kg + TPR * j] = 0.f;
            if (kg == 0) {
                pml[r * 2] = -INFINITY;
                pml[r * 2 + 1] = 0.f;
            }
        }
        return;
    }
    const unsigned long long anc =
        (tree && r < a.R) ? a.anc[(size_t)b * a.N + (r % a.N)] : 0ull;
    const float* qsrc = static_cast<const float*>(a.q_rot) + (size_t)bg * a.q_rows_pad * D;
    {
        // (each thread's loads issued together before its stores)
        constexpr int NQ = ROWS * D / 4 / 256;
        float4 x[NQ];
#pragma unroll
        for (int i = 0; i < NQ; ++i) {
            const int e = tid + 256 * i, rr = e / (D / 4), c = 4 * (e % (D / 4));
            const int gr = rc * ROWS + rr;
            x[i] = gr < a.R ? *reinterpret_cast<const float4*>(qsrc + (size_t)gr * D + c)
                            : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int i = 0; i < NQ; ++i) {
            const int e = tid + 256 * i, rr = e / (D / 4), c = 4 * (e % (D / 4));
            float* q = sQ + rr * (D + 1) + c;
            q[0] = x[i].x;
            q[1] = x[i].y;
            q[2] = x[i].z;
            q[3] = x[i].w;
        }
    }
    const T* Kb = tree ? static_cast<const T*>(a.treeK) + (size_t)bg * a.N * D
                       : static_cast<const T*>(a.cacheK) + (size_t)bg * a.S_max * D;
    const T* Vb = tree ? static_cast<const T*>(a.treeV) + (size_t)bg * a.N * D
                       : static_cast<const T*>(a.cacheV) + (size_t)bg * a.S_max * D;
    float m = -INFINITY, l = 0.f;
    float o[CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) o[j] = 0.f;
    for (int kt = k_lo; kt < k_hi; kt += CC_KEYS) {
        __syncthreads();
        {
            // K and V rows of the tile, zeros past k_hi (each thread's loads
            // issued together before its stores)
            constexpr int NK = CC_KEYS * D / 4 / 256;
            float4 xk[NK], xv[NK];
#pragma unroll
            for (int i = 0; i < NK; ++i) {
                const int e = tid + 256 * i, kk = e / (D / 4), c = 4 * (e % (D / 4));
                const int key = kt + kk;
                xk[i] = xv[i] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (key < k_hi) {
                    xk[i] = *reinterpret_cast<const float4*>(Kb + (size_t)key * D + c);
                    xv[i] = *reinterpret_cast<const float4*>(Vb + (size_t)key * D + c);
                }
            }
#pragma unroll
            for (int i = 0; i < NK; ++i) {
                const int e = tid + 256 * i, kk = e / (D / 4), c = 4 * (e % (D / 4));
                float* k = sK + kk * (D + 1) + c;
                float* v = sV + kk * (D + 1) + c;
                k[0] = xk[i].x;
                k[1] = xk[i].y;
                k[2] = xk[i].z;
                k[3] = xk[i].w;
                v[0] = xv[i].x;
                v[1] = xv[i].y;
                v[2] = xv[i].z;
                v[3] = xv[i].w;
            }
        }
        __syncthreads();
        // Scores of this thread's KPT keys: each query value read once.
        float acc[KPT];
#pragma unroll
        for (int jj = 0; jj < KPT; ++jj) acc[jj] = 0.f;
#pragma unroll 8
        for (int c = 0; c < D; ++c) {
            const float qv = sQ[row * (D + 1) + c];
#pragma unroll
            for (int jj = 0; jj < KPT; ++jj) acc[jj] = fmaf(qv, sK[(kg * KPT + jj) * (D + 1) + c], acc[jj]);
        }
        float s[KPT];
        float tmax = -INFINITY;
#pragma unroll
        for (int jj = 0; jj < KPT; ++jj) {
            const int key = kt + kg * KPT + jj;
            const bool ok = key < k_hi && (!tree || ((anc >> key) & 1ull));
            s[jj] = ok ? acc[jj] * a.scale : -INFINITY;
            tmax = fmaxf(tmax, s[jj]);
        }
#pragma unroll
        for (int o2 = 1; o2 < TPR; o2 <<= 1) tmax = fmaxf(tmax, __shfl_xor_sync(FULL, tmax, o2));
        const float mnew = fmaxf(m, tmax);
        const float alpha = (mnew == -INFINITY) ? 1.f : __expf(m - mnew);
        float psum = 0.f;
#pragma unroll
        for (int jj = 0; jj < KPT; ++jj) {
            const float p = (s[jj] == -INFINITY) ? 0.f : __expf(s[jj] - mnew);
            sS[row * (CC_KEYS + 1) + kg * KPT + jj] = p;
            psum += p;
        }
#pragma unroll
        for (int o2 = 1; o2 < TPR; o2 <<= 1) psum += __shfl_xor_sync(FULL, psum, o2);
        l = l * alpha + psum;
        m = mnew;
        __syncwarp();
#pragma unroll
        for (int j = 0; j < CPT; ++j) o[j] *= alpha;
        for (int kk = 0; kk < CC_KEYS; ++kk) {
            const float p = sS[row * (CC_KEYS + 1) + kk];
#pragma unroll
            for (int j = 0; j < CPT; ++j) o[j] = fmaf(p, sV[kk * (D + 1) + kg + TPR * j], o[j]);
        }
    }
    if (r < a.R) {
#pragma unroll
        for (int j = 0; j < CPT; ++j) po[(size_t)r * D + kg + TPR * j] = o[j];
        if (kg == 0) {
            pml[r * 2] = m;
            pml[r * 2 + 1] = l;
        }
    }
}

template <typename T, int D, int ROWS>
static int launch_cc(const AttnArgs& a, cudaStream_t st) {
    const size_t smem = sizeof(float) * (ROWS * (D + 1) + 2 * CC_KEYS * (D + 1) + ROWS * (CC_KEYS + 1));
    static thread_local int attr_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (attr_dev != dev) {
        cudaFuncSetAttribute(attn_cc_kernel<T, D, ROWS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        attr_dev = dev;
    }
    const int nrc = (a.R + ROWS - 1) / ROWS;
    dim3 grid(a.B * a.Hkv * nrc, a.nsplit);
    launch_pdl(attn_cc_kernel<T, D, ROWS>, grid, dim3(256), smem, st, a);
    return check_launch("attn_cc_kernel");
}

int launch_attn_cc_f32(const AttnArgs& a, cudaStream_t st) {
    if (a.R <= 16) return a.d == 128 ? launch_cc<float, 128, 16>(a, st) : launch_cc<float, 64, 16>(a, st);
    return a.d == 128 ? launch_cc<float, 128, 64>(a, st) : launch_cc<float, 64, 64>(a, st);
}

}  // namespace gv
