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
// fp32 path: one thread per (sequence, node, frequency) rotates that
// frequency's pair of every query head (into the q_rot workspace, grouped by
// KV head) and of every key head (into the tree K scratch), and copies v.
__global__ void __launch_bounds__(128)
rope_tree_f32_kernel(const float* __restrict__ q, const float* __restrict__ k_new,
                     const float* __restrict__ v_new, const float2* __restrict__ rope, int B, int N,
                     int Hq, int Hkv, int d, float* __restrict__ q_rot, float* __restrict__ treeK,
                     float* __restrict__ treeV, int q_rows_pad) {
    const int half = d >> 1;
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= B * N * half) return;
    const int j = idx % half;
    const int i = (idx / half) % N;
    const int b = idx / (half * N);
    const float2 r = rope[idx];
    const float c = r.x, s = r.y;
    const int G = Hq / Hkv;
    for (int h = 0; h < Hq; ++h) {
        const size_t src = (((size_t)b * N + i) * Hq + h) * d;
        const float x0 = q[src + j], x1 = q[src + j + half];
        const int g = h / G, hl = h % G;
        const size_t dst = (((size_t)b * Hkv + g) * q_rows_pad + (size_t)hl * N + i) * d;
        q_rot[dst + j] = x0 * c - x1 * s;
        q_rot[dst + j + half] = x1 * c + x0 * s;
    }
    for (int g = 0; g < Hkv; ++g) {
        const size_t src = (((size_t)b * N + i) * Hkv + g) * d;
        const size_t dst = (((size_t)b * Hkv + g) * N + i) * d;
        const float x0 = k_new[src + j], x1 = k_new[src + j + half];
        treeK[dst + j] = x0 * c - x1 * s;
        treeK[dst + j + half] = x1 * c + x0 * s;
        treeV[dst + j] = v_new[src + j];
        treeV[dst + j + half] = v_new[src + j + half];
    }
}

int launch_rope_tree_f32(const AttnArgs& a, cudaStream_t st) {
    const int total = a.B * a.N * (a.d / 2);
    rope_tree_f32_kernel<<<(total + 127) / 128, 128, 0, st>>>(
        static_cast<const float*>(a.q), static_cast<const float*>(a.k_new),
        static_cast<const float*>(a.v_new), reinterpret_cast<const float2*>(a.rope), a.B, a.N, a.Hq,
        a.Hkv, a.d, static_cast<float*>(a.q_rot), static_cast<float*>(a.treeK),
        static_cast<float*>(a.treeV), a.q_rows_pad);
    return check_launch("rope_tree_f32_kernel");
}

// ----------------------------------------------------------------- combine --
// One warp per output row (b, node, head): out = sum_s e^{m_s - M} o_s / sum_s e^{m_s - M} l_s.
template <typename T, int D>
__global__ void __launch_bounds__(256)
attn_combine_kernel(const float* __restrict__ part_o, const float* __restrict__ part_ml, int B,
                    int N, int Hq, int Hkv, int nsplit, int R, T* __restrict__ out) {
    const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= B * N * Hq) return;
    const int h = w % Hq, i = (w / Hq) % N, b = w / (Hq * N);
    const int G = Hq / Hkv, g = h / G, hl = h % G;
    const int r = hl * N + i;
    const size_t bg = (size_t)b * Hkv + g;
    float M = -INFINITY;
    for (int s = 0; s < nsplit; ++s) M = fmaxf(M, part_ml[((bg * nsplit + s) * R + r) * 2]);
    float L = 0.f;
    float acc[D / 32] = {};
    for (int s = 0; s < nsplit; ++s) {
        const size_t pr = (bg * nsplit + s) * R + r;
        const float m = part_ml[pr * 2];
        if (m == -INFINITY) continue;
        const float wgt = __expf(m - M);
        L += wgt * part_ml[pr * 2 + 1];
#pragma unroll
        for (int j = 0; j < D / 32; ++j) acc[j] += wgt * part_o[pr * D + lane + 32 * j];
    }
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
        attn_combine_kernel<float, 128><<<blocks, 256, 0, st>>>(a.part_o, a.part_ml, a.B, a.N, a.Hq,
                                                                a.Hkv, a.nsplit, a.R, out);
    else
        attn_combine_kernel<float, 64><<<blocks, 256, 0, st>>>(a.part_o, a.part_ml, a.B, a.N, a.Hq,
                                                               a.Hkv, a.nsplit, a.R, out);
    return check_launch("attn_combine_kernel");
}

// -------------------------------------------------------- CUDA-core splits --
// Block = (sequence, KV head, 64-row chunk of the query rows) x split.
// 4 threads per query row: each scores 8 of a 32-key tile and owns d/4 output
// columns (c = lane_in_row + 4 j, so the 4 threads hit different banks).
constexpr int CC_ROWS = 64;
constexpr int CC_KEYS = 32;

template <typename T, int D>
__global__ void __launch_bounds__(256)
attn_cc_kernel(AttnArgs a) {
    extern __shared__ float smem[];
    float* sQ = smem;                          // [64][D+1]
    float* sK = sQ + CC_ROWS * (D + 1);        // [32][D+1]
    float* sV = sK + CC_KEYS * (D + 1);        // [32][D+1]
    float* sS = sV + CC_KEYS * (D + 1);        // [64][33]
    const int nrc = (a.R + CC_ROWS - 1) / CC_ROWS;
    const int bg = blockIdx.x / nrc, rc = blockIdx.x % nrc;
    const int b = bg / a.Hkv;
    const int split = blockIdx.y;
    const int P = min(max(a.prefix_len[b], 0), a.S_max);
    const bool tree = split == a.nsplit - 1;
    const int k_lo = tree ? 0 : split * a.kps;
    const int k_hi = tree ? a.N : min(P, k_lo + a.kps);
    const int tid = threadIdx.x, row = tid >> 2, kg = tid & 3;
    const int r = rc * CC_ROWS + row;
    float* po = a.part_o + ((size_t)bg * a.nsplit + split) * a.R * D;
    float* pml = a.part_ml + ((size_t)bg * a.nsplit + split) * a.R * 2;
    if (k_lo >= k_hi) {
        if (r < a.R) {
            for (int j = 0; j < D / 4; ++j) po[(size_t)r * D + kg + 4 * j] = 0.f;
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
    for (int e = tid; e < CC_ROWS * D; e += 256) {
        const int rr = e / D, c = e % D;
        const int gr = rc * CC_ROWS + rr;
        sQ[rr * (D + 1) + c] = gr < a.R ? qsrc[(size_t)gr * D + c] : 0.f;
    }
    const T* Kb = tree ? static_cast<const T*>(a.treeK) + (size_t)bg * a.N * D
                       : static_cast<const T*>(a.cacheK) + (size_t)bg * a.S_max * D;
    const T* Vb = tree ? static_cast<const T*>(a.treeV) + (size_t)bg * a.N * D
                       : static_cast<const T*>(a.cacheV) + (size_t)bg * a.S_max * D;
    float m = -INFINITY, l = 0.f;
    float o[D / 4];
#pragma unroll
    for (int j = 0; j < D / 4; ++j) o[j] = 0.f;
    for (int kt = k_lo; kt < k_hi; kt += CC_KEYS) {
        __syncthreads();
        for (int e = tid; e < CC_KEYS * D; e += 256) {
            const int kk = e / D, c = e % D;
            const int key = kt + kk;
            float kv = 0.f, vv = 0.f;
            if (key < k_hi) {
                kv = to_f32(Kb[(size_t)key * D + c]);
                vv = to_f32(Vb[(size_t)key * D + c]);
            }
            sK[kk * (D + 1) + c] = kv;
            sV[kk * (D + 1) + c] = vv;
        }
        __syncthreads();
        float s[8];
        float tmax = -INFINITY;
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
            const int kk = kg * 8 + jj;
            float acc = 0.f;
#pragma unroll 16
            for (int c = 0; c < D; ++c) acc = fmaf(sQ[row * (D + 1) + c], sK[kk * (D + 1) + c], acc);
            const int key = kt + kk;
            const bool ok = key < k_hi && (!tree || ((anc >> key) & 1ull));
            s[jj] = ok ? acc * a.scale : -INFINITY;
            tmax = fmaxf(tmax, s[jj]);
        }
        tmax = fmaxf(tmax, __shfl_xor_sync(FULL, tmax, 1));
        tmax = fmaxf(tmax, __shfl_xor_sync(FULL, tmax, 2));
        const float mnew = fmaxf(m, tmax);
        const float alpha = (mnew == -INFINITY) ? 1.f : __expf(m - mnew);
        float psum = 0.f;
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
            const float p = (s[jj] == -INFINITY) ? 0.f : __expf(s[jj] - mnew);
            sS[row * 33 + kg * 8 + jj] = p;
            psum += p;
        }
        psum += __shfl_xor_sync(FULL, psum, 1);
        psum += __shfl_xor_sync(FULL, psum, 2);
        l = l * alpha + psum;
        m = mnew;
        __syncwarp();
#pragma unroll
        for (int j = 0; j < D / 4; ++j) o[j] *= alpha;
        for (int kk = 0; kk < CC_KEYS; ++kk) {
            const float p = sS[row * 33 + kk];
#pragma unroll
            for (int j = 0; j < D / 4; ++j) o[j] = fmaf(p, sV[kk * (D + 1) + kg + 4 * j], o[j]);
        }
    }
    if (r < a.R) {
#pragma unroll
        for (int j = 0; j < D / 4; ++j) po[(size_t)r * D + kg + 4 * j] = o[j];
        if (kg == 0) {
            pml[r * 2] = m;
            pml[r * 2 + 1] = l;
        }
    }
}

template <typename T, int D>
static int launch_cc(const AttnArgs& a, cudaStream_t st) {
    const size_t smem = sizeof(float) * (CC_ROWS * (D + 1) + 2 * CC_KEYS * (D + 1) + CC_ROWS * 33);
    static thread_local int attr_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (attr_dev != dev) {
        cudaFuncSetAttribute(attn_cc_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        attr_dev = dev;
    }
    const int nrc = (a.R + CC_ROWS - 1) / CC_ROWS;
    dim3 grid(a.B * a.Hkv * nrc, a.nsplit);
    attn_cc_kernel<T, D><<<grid, 256, smem, st>>>(a);
    return check_launch("attn_cc_kernel");
}

int launch_attn_cc_f32(const AttnArgs& a, cudaStream_t st) {
    return a.d == 128 ? launch_cc<float, 128>(a, st) : launch_cc<float, 64>(a, st);
}

}  // namespace gv
