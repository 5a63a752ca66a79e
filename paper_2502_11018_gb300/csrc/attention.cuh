// Internal interface between the attention launchers (not part of the C ABI).
#pragma once

#include "gv_internal.cuh"

namespace gv {

// Everything one attention layer needs, with the workspace already carved.
struct AttnArgs {
    int B, N, Hq, Hkv, d, S_max;
    int G;            // Hq / Hkv
    int R;            // query rows per (sequence, KV head) = G * N
    int q_rows_pad;   // row stride of q_rot per (sequence, KV head)
    float scale;      // 1 / sqrt(d)
    const void* q;
    const void* k_new;
    const void* v_new;
    const void* cacheK;
    const void* cacheV;
    const int32_t* prefix_len;
    const float* rope;   // [B][N][d/2][2] cos, sin per node (gv_rope_table)
    const unsigned long long* anc;
    void* treeK;
    void* treeV;
    void* out;
    // workspace pieces
    void* q_rot;      // [B*Hkv][q_rows_pad][d]  rotated queries          (CUDA-core path)
    float* part_o;    // [B*Hkv][nsplit][R][d]   per-split partial outputs (CUDA-core path)
    float* part_ml;   // [B*Hkv][nsplit][R][2] (m, l)                  (CUDA-core path)
                      // [units][csize][128] lse                       (tensor-core path)
    void* part_o_bf16;  // [units][csize][128][d] bf16 rows, chunks rotated (tensor-core path)
    int nsplit;       // prefix splits + 1 tree split (CUDA-core path)
    int kps;          // prefix keys per split (CUDA-core path)
    int csize;        // key splits (CTAs) per unit (tensor-core path)
    int tiles;        // M tiles of 128 query rows per (sequence, KV head); unit = (b, g, tile)
};

// gv_verify_attention_layers: workspace plan and call (attention_layers_sm103.cu).
struct AttnLayersPlan {
    int T;            // 128-row M tiles per (sequence, KV head): 1 or 2
    int ctas;         // CTAs of the persistent kernel (one per SM)
    int ncnt;         // arrival counters, L * B * Hkv
    size_t q_rot, cnt, part, part_lse, total;   // byte offsets into the workspace
};
struct AttnLayersCall {
    int L, B, N, Hq, Hkv, S_max;
    const void* q;
    long long q_ls;   // layer strides in elements
    const void* k_new;
    long long k_ls;
    const void* v_new;
    long long v_ls;
    const void* cacheK;
    const void* cacheV;
    long long cache_ls;
    const int32_t* prefix_len;
    const float* rope;
    const uint64_t* anc;
    void* treeK;
    void* treeV;
    void* out;
    void* workspace;
};
AttnLayersPlan attn_layers_plan(int L, int B, int N, int Hq, int Hkv);
int launch_attn_layers(const AttnLayersCall& c, cudaStream_t st);

int launch_rope_table(const int32_t* pos, int B, int N, int d, float base, float* rope,
                      cudaStream_t st);
int launch_rope_tree_f32(const AttnArgs& a, cudaStream_t st);
int launch_attn_combine_f32(const AttnArgs& a, cudaStream_t st);
int launch_attn_cc_f32(const AttnArgs& a, cudaStream_t st);
int launch_attn_tc(const AttnArgs& a, cudaStream_t st, int phase);
int launch_rope_apply(const void* x, size_t layer_stride, int L, int B, int N, int H, const float* rope, void* out,
                      cudaStream_t st);   // phase: 1 split kernel, 2 merge, 3 both
int attn_tc_splits(int units, int S_max);

}  // namespace gv
