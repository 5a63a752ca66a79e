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
    float rope_base;
    float scale;      // 1 / sqrt(d)
    const void* q;
    const void* k_new;
    const void* v_new;
    const void* cacheK;
    const void* cacheV;
    const int32_t* prefix_len;
    const int32_t* pos;
    const unsigned long long* anc;
    void* treeK;
    void* treeV;
    void* out;
    // workspace pieces
    void* q_rot;      // [B*Hkv][q_rows_pad][d]  rotated queries (fp32 or bf16)
    float* part_o;    // [B*Hkv][nsplit][R][d]
    float* part_ml;   // [B*Hkv][nsplit][R][2]
    int nsplit;       // prefix splits + 1 tree split
    int kps;          // prefix keys per split
    unsigned* counters;  // [B*Hkv] arrival tickets (tensor-core path)
};

template <typename T, typename TQ> int launch_rope_tree(const AttnArgs& a, cudaStream_t st);
template <typename T> int launch_attn_combine(const AttnArgs& a, cudaStream_t st);
template <typename T> int launch_attn_cc(const AttnArgs& a, cudaStream_t st);

}  // namespace gv
