// extern "C" entry points of libgv.so: argument validation, workspace
// carving, and dispatch to the kernels.  The declarations and the contract of
// every call are in include/gv.h.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <cmath>
#include <mutex>

#include "gv_internal.cuh"
#include "attention.cuh"

namespace gv {

// ------------------------------------------------------------- bookkeeping --
static thread_local char g_err[512];

void set_error(const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
}

void clear_error() { g_err[0] = '\0'; }

int check_launch(const char* what) {
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("%s: %s", what, cudaGetErrorString(e));
        return GV_ERR_CUDA;
    }
    return GV_OK;
}

int sm_count() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (cache[dev] == 0) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        cache[dev] = n > 0 ? n : 148;
    }
    return cache[dev];
}

int device_cc() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    if (cache[dev] == 0) {
        int ma = 0, mi = 0;
        cudaDeviceGetAttribute(&ma, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&mi, cudaDevAttrComputeCapabilityMinor, dev);
        cache[dev] = ma * 10 + mi;
    }
    return cache[dev];
}

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Kernel launchers defined in the other translation units.
int launch_tree_build(const int32_t*, const int32_t*, int, int, int32_t*, int32_t*, uint64_t*,
                      int32_t*, cudaStream_t);
int launch_rmsnorm(const void* x, const void* w, int rows, int H, float eps, void* out, cudaStream_t st);
size_t tgf_workspace_bytes(int rows, int d, int e);
size_t draft_tree_workspace_bytes(int B, int k, int D, int V);
int launch_draft_tree_expand(int B, int k, int D, int V, int step, int dt, const int32_t* root_token,
                             const void* logits, int32_t* exp_token, int32_t* exp_pool, void* ws, cudaStream_t st);
int launch_draft_tree_finish(int B, int k, int D, int N, int32_t* parents, int32_t* tokens, void* ws,
                             cudaStream_t st);
int launch_tgf(const void* F, const void* x, int rows, int d, int e, const void* Wm, const void* bm,
               const void* g_h, const void* b_h, const void* g_x, const void* b_x, const void* Wu, const void* bu,
               const void* Wd, const void* bd, float eps, void* h_out, void* o_out, void* ws, cudaStream_t st);
int launch_tat_loss(const void* logits, int logits_dt, const int32_t* tokens, const void* fd,
                    const void* ft, int feat_dt, int B, int T, int V, int H, int k, int n,
                    const uint8_t* mbar_prev, float lam_tok, float lam_feat, uint8_t* mbar,
                    uint8_t* mask, float* ell, float* seq_loss, cudaStream_t st);
int launch_kv_compact(int, int, int, int, int, int, int, int, const void*, const void*, void*,
                      void*, const int32_t*, const int32_t*, const int32_t*, int32_t*, int32_t*,
                      cudaStream_t);
int launch_accept(int, int, int, int, float, const int32_t*, const uint64_t*, const int32_t*,
                  const int32_t*, const float*, const float*, const float*, const float*,
                  int32_t*, int32_t*, int32_t*, int32_t*, void*, cudaStream_t);
int launch_lmhead_cc(const float*, const float*, int, int, int, int, int, float*, SelectPartials,
                     int32_t*, float*, float*, float*, cudaStream_t);
int launch_lmhead_tc(const void*, const void*, int, int, int, int, int, float*, SelectPartials, int*,
                     cudaStream_t);
int launch_lmhead_merge(SelectPartials, int, int, int32_t*, float*, float*, float*, const int*,
                        cudaStream_t);
int lmhead_tc_grid(int slots_capacity);

// ---------------------------------------------------------- attention plan --
constexpr int KPS_F32 = 64;    // prefix keys per split, CUDA-core path

struct AttnPlan {
    size_t q_rot, part_o, part_ml, total;
    int nsplit, q_rows_pad, kps;
    int tiles, csize;   // tensor-core path: M tiles per (b, g), key splits per unit
};

// Shapes the kernels handle: fp32 with d in {64, 128}; bf16 (tensor cores)
// with d = 128, G = Hq / Hkv dividing 128 and at most 256 query rows (two
// M = 128 tiles) per KV head.
static int attn_shape_status(const gv_attn_shape* s) {
    if (!s || s->B < 1 || s->Hkv < 1 || s->Hq < s->Hkv || s->Hq % s->Hkv != 0 || s->S_max < 1 ||
        (s->dt != GV_BF16 && s->dt != GV_F32))
        return GV_ERR_ARG;
    if (s->N < 1 || s->N > 64) return GV_ERR_UNSUPPORTED;
    if (s->dt == GV_F32 && !(s->d == 64 || s->d == 128)) return GV_ERR_UNSUPPORTED;
    const int G = s->Hq / s->Hkv;
    if (s->dt == GV_BF16 && (s->d != 128 || 128 % G != 0 || G * s->N > 256)) return GV_ERR_UNSUPPORTED;
    return GV_OK;
}

// The fp32 path keeps rotated queries and per-split partials in the
// workspace; the bf16 path keeps one bf16 partial row and one lse per (unit,
// key split, row of the unit's 128-row tile), for its merge kernel.
static AttnPlan attn_plan(const gv_attn_shape* s) {
    AttnPlan p{};
    const int R = (s->Hq / s->Hkv) * s->N;
    p.q_rows_pad = (R + 127) / 128 * 128;
    p.kps = KPS_F32;
    p.nsplit = (s->S_max + KPS_F32 - 1) / KPS_F32 + 1;
    size_t off = 0;
    const size_t bh = (size_t)s->B * s->Hkv;
    if (s->dt == GV_F32) {
        p.q_rot = off;
        off += align256(bh * p.q_rows_pad * s->d * sizeof(float));
        p.part_o = off;
        off += align256(bh * p.nsplit * R * s->d * sizeof(float));
        p.part_ml = off;
        off += align256(bh * p.nsplit * R * 2 * sizeof(float));
    } else {
        p.tiles = (R + 127) / 128;
        const int units = s->B * s->Hkv * p.tiles;
        p.csize = attn_tc_splits(units, s->S_max);
        const size_t nrows = (size_t)units * p.csize * 128;
        p.part_o = off;
        off += align256(nrows * 128 * 2);
        p.part_ml = off;
        off += align256(nrows * sizeof(float));
    }
    p.total = off;
    return p;
}

// ------------------------------------------------------------ lmhead plan --
constexpr int CC_TV = 16;        // vocabulary tile of the CUDA-core (fp32) kernel
constexpr int TC_SLOTS = 256;    // partial slots of the tensor-core kernel (one per CTA)

struct LmPlan {
    size_t val, id, m, s, err, total;
    int slots, K;
};

static LmPlan lm_plan(int rows, int V, int dt, int mode, int k) {
    LmPlan p{};
    p.slots = dt == GV_F32 ? (V + CC_TV - 1) / CC_TV : TC_SLOTS;
    p.K = mode == GV_SELECT_TOPK ? k : 1;
    const size_t n = (size_t)p.slots * rows;
    size_t off = 0;
    p.val = off;
    off += align256(n * p.K * sizeof(float));
    p.id = off;
    off += align256(n * p.K * sizeof(int));
    p.m = off;
    off += align256(n * sizeof(float));
    p.s = off;
    off += align256(n * sizeof(float));
    p.err = off;
    off += align256((size_t)TC_SLOTS * sizeof(int));
    p.total = off;
    return p;
}

// ------------------------------------------- allocation-free LM head scratch --
// gv_lmhead_argmax_noalloc keeps its scratch in the library's own device
// memory: the argmax partials (value, id) of up to GV_NOALLOC_MAX_ROWS rows
// for up to TC_SLOTS CTAs, then the per-CTA status words of the bounded waits.
constexpr size_t NOALLOC_ENTRIES = (size_t)TC_SLOTS * GV_NOALLOC_MAX_ROWS;
constexpr size_t NOALLOC_ID_OFF = NOALLOC_ENTRIES * sizeof(float);
constexpr size_t NOALLOC_ERR_OFF = NOALLOC_ID_OFF + NOALLOC_ENTRIES * sizeof(int);
constexpr size_t NOALLOC_BYTES = NOALLOC_ERR_OFF + (size_t)TC_SLOTS * sizeof(int);
__device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_BYTES];

// Address of the scratch in the current device's context.  Looked up on
// every call (cudaGetSymbolAddress allocates nothing), so a context that was
// reset or replaced since an earlier call gets its own array's address.
static int noalloc_scratch(char** out) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) {
        set_error("gv_lmhead_argmax_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
        return GV_ERR_CUDA;
    }
    *out = static_cast<char*>(p);
    return GV_OK;
}

}  // namespace gv

using namespace gv;

extern "C" {

int gv_version(void) { return 100; }

const char* gv_last_error(void) { return g_err; }

const char* gv_status_string(int status) {
    switch (status) {
        case GV_OK: return "GV_OK";
        case GV_ERR_ARG: return "GV_ERR_ARG";
        case GV_ERR_INVALID_TREE: return "GV_ERR_INVALID_TREE";
        case GV_ERR_CAPACITY: return "GV_ERR_CAPACITY";
        case GV_ERR_UNSUPPORTED: return "GV_ERR_UNSUPPORTED";
        case GV_ERR_CUDA: return "GV_ERR_CUDA";
        case GV_ERR_TIMEOUT: return "GV_ERR_TIMEOUT";
        default: return "GV_ERR_UNKNOWN";
    }
}

int gv_tree_build(const int32_t* parents, const int32_t* prefix_len, int B, int N, int32_t* depth,
                  int32_t* pos, uint64_t* anc, int32_t* seq_status, void* stream) {
    clear_error();
    if (N < 1 || N > 64) {
        set_error("gv_tree_build: N=%d outside 1..64", N);
        return GV_ERR_INVALID_TREE;
    }
    GV_CHECK_ARG(B >= 1, "gv_tree_build: B=%d", B);
    GV_CHECK_ARG(parents && prefix_len && depth && pos && anc && seq_status,
                 "gv_tree_build: null pointer");
    GV_CHECK_ARG(((uintptr_t)anc & 7u) == 0, "gv_tree_build: anc not 8-byte aligned");
    return launch_tree_build(parents, prefix_len, B, N, depth, pos, anc, seq_status,
                             as_stream(stream));
}

int gv_rope_table(const int32_t* pos, int B, int N, int d, float rope_base, float* rope,
                  void* stream) {
    clear_error();
    GV_CHECK_ARG(pos && rope, "gv_rope_table: null pointer");
    GV_CHECK_ARG(B >= 1 && N >= 1 && d >= 2 && d <= 256 && d % 2 == 0,
                 "gv_rope_table: B=%d N=%d d=%d", B, N, d);
    GV_CHECK_ARG(rope_base > 0.0f && std::isfinite(rope_base), "gv_rope_table: rope_base %g",
                 (double)rope_base);
    GV_CHECK_ARG(((uintptr_t)rope & 7u) == 0, "gv_rope_table: rope not 8-byte aligned");
    return launch_rope_table(pos, B, N, d, rope_base, rope, as_stream(stream));
}

size_t gv_verify_attention_workspace(const gv_attn_shape* s) {
    if (attn_shape_status(s) != GV_OK) return 0;
    return attn_plan(s).total;
}

// phase 1: the split kernels (partial rows, or the output when there is one
// split); phase 2: the merge of the splits; 3: both.
static int attention_call(const char* name, int phase, const gv_attn_shape* s, const void* q, const void* k_new,
                          const void* v_new, const void* cacheK, const void* cacheV, const int32_t* prefix_len,
                          const float* rope, const uint64_t* anc, void* treeK, void* treeV, void* out,
                          void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    const int sst = attn_shape_status(s);
    if (sst == GV_ERR_UNSUPPORTED) {
        set_error("%s: unsupported shape (N=%d d=%d G*N=%d dt=%d); fp32 needs "
                  "d in {64,128}, bf16 needs d=128 and G*N <= 256, N <= 64",
                  name, s->N, s->d, (s->Hq / s->Hkv) * s->N, (int)s->dt);
        return GV_ERR_UNSUPPORTED;
    }
    GV_CHECK_ARG(sst == GV_OK, "%s: invalid shape", name);
    GV_CHECK_ARG(out && aligned16(out), "%s: out null or not 16-byte aligned", name);
    if (phase & 1) {
        const void* ptrs[] = {q, k_new, v_new, cacheK, cacheV, treeK, treeV};
        for (const void* p : ptrs) GV_CHECK_ARG(p && aligned16(p), "%s: tensor null or not 16-byte aligned", name);
        GV_CHECK_ARG(prefix_len && anc, "%s: null index pointer", name);
        // no table: q and k_new arrive rotated (bf16 path only)
        GV_CHECK_ARG(rope ? aligned16(rope) : s->dt == GV_BF16,
                     "%s: rope not 16-byte aligned, or NULL on the fp32 path", name);
    }
    const AttnPlan plan = attn_plan(s);
    GV_CHECK_ARG(workspace && ((uintptr_t)workspace & 255u) == 0, "%s: workspace null or not 256-byte aligned",
                 name);
    GV_CHECK_ARG(ws_bytes >= plan.total, "%s: workspace %zu < %zu bytes", name, ws_bytes, plan.total);
    char* ws = static_cast<char*>(workspace);
    AttnArgs a{};
    a.B = s->B;
    a.N = s->N;
    a.Hq = s->Hq;
    a.Hkv = s->Hkv;
    a.d = s->d;
    a.S_max = s->S_max;
    a.G = s->Hq / s->Hkv;
    a.R = a.G * s->N;
    a.q_rows_pad = plan.q_rows_pad;
    a.scale = 1.0f / sqrtf((float)s->d);
    a.q = q;
    a.k_new = k_new;
    a.v_new = v_new;
    a.cacheK = cacheK;
    a.cacheV = cacheV;
    a.prefix_len = prefix_len;
    a.rope = rope;
    a.anc = reinterpret_cast<const unsigned long long*>(anc);
    a.treeK = treeK;
    a.treeV = treeV;
    a.out = out;
    a.q_rot = ws + plan.q_rot;
    a.part_o = reinterpret_cast<float*>(ws + plan.part_o);
    a.part_ml = reinterpret_cast<float*>(ws + plan.part_ml);
    a.part_o_bf16 = ws + plan.part_o;
    a.tiles = plan.tiles;
    a.csize = plan.csize;
    a.nsplit = plan.nsplit;
    a.kps = plan.kps;
    cudaStream_t st = as_stream(stream);
    int rc;
    if (s->dt == GV_F32) {
        if (phase & 1) {
            if ((rc = launch_rope_tree_f32(a, st)) != GV_OK) return rc;
            if ((rc = launch_attn_cc_f32(a, st)) != GV_OK) return rc;
        }
        return (phase & 2) ? launch_attn_combine_f32(a, st) : GV_OK;
    }
    return launch_attn_tc(a, st, phase);
}

int gv_verify_attention(const gv_attn_shape* s, const void* q, const void* k_new,
                        const void* v_new, const void* cacheK, const void* cacheV,
                        const int32_t* prefix_len, const float* rope, const uint64_t* anc,
                        void* treeK, void* treeV, void* out, void* workspace, size_t ws_bytes,
                        void* stream) {
    return attention_call("gv_verify_attention", 3, s, q, k_new, v_new, cacheK, cacheV, prefix_len, rope, anc,
                          treeK, treeV, out, workspace, ws_bytes, stream);
}

int gv_verify_attention_split(const gv_attn_shape* s, const void* q, const void* k_new, const void* v_new,
                              const void* cacheK, const void* cacheV, const int32_t* prefix_len, const float* rope,
                              const uint64_t* anc, void* treeK, void* treeV, void* out, void* workspace,
                              size_t ws_bytes, void* stream) {
    return attention_call("gv_verify_attention_split", 1, s, q, k_new, v_new, cacheK, cacheV, prefix_len, rope, anc,
                          treeK, treeV, out, workspace, ws_bytes, stream);
}

int gv_verify_attention_merge(const gv_attn_shape* s, void* out, void* workspace, size_t ws_bytes, void* stream) {
    return attention_call("gv_verify_attention_merge", 2, s, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr,
                          nullptr, nullptr, nullptr, nullptr, out, workspace, ws_bytes, stream);
}

int gv_rope_apply(const gv_attn_shape* s, int L, const void* q, size_t q_layer_stride, const void* k_new,
                  size_t k_layer_stride, const float* rope, void* q_out, void* k_out, void* stream) {
    clear_error();
    GV_CHECK_ARG(s && s->dt == GV_BF16 && s->d == 128 && s->B >= 1 && s->N >= 1 && s->Hq >= 1 && s->Hkv >= 1,
                 "gv_rope_apply: bf16 with d = 128 only");
    GV_CHECK_ARG(L >= 1, "gv_rope_apply: L=%d", L);
    const size_t nq = (size_t)s->B * s->N * s->Hq * 128, nk = (size_t)s->B * s->N * s->Hkv * 128;
    GV_CHECK_ARG((L == 1 || (q_layer_stride >= nq && k_layer_stride >= nk)) && q_layer_stride % 8 == 0 &&
                     k_layer_stride % 8 == 0,
                 "gv_rope_apply: layer strides %zu, %zu (elements; >= one layer, multiples of 8)", q_layer_stride,
                 k_layer_stride);
    const void* ptrs[] = {q, k_new, rope, q_out, k_out};
    for (const void* p : ptrs) GV_CHECK_ARG(p && aligned16(p), "gv_rope_apply: tensor null or not 16-byte aligned");
    cudaStream_t st = as_stream(stream);
    int rc = launch_rope_apply(q, q_layer_stride, L, s->B, s->N, s->Hq, rope, q_out, st);
    if (rc != GV_OK) return rc;
    return launch_rope_apply(k_new, k_layer_stride, L, s->B, s->N, s->Hkv, rope, k_out, st);
}

static int attn_layers_shape_ok(const gv_attn_shape* s, int L) {
    return s && s->dt == GV_BF16 && s->d == 128 && L >= 1 && s->B >= 1 && s->B <= 64 && s->N >= 1 &&
           s->N <= 64 && s->Hkv >= 1 && s->Hq >= s->Hkv && s->Hq % s->Hkv == 0 &&
           (s->Hq / s->Hkv) * s->N <= 256 && s->S_max >= 1 &&
           8LL * L * s->B * s->N * (s->Hq + 2LL * s->Hkv) <= (1LL << 30);
}

size_t gv_verify_attention_layers_workspace(const gv_attn_shape* s, int L) {
    if (!attn_layers_shape_ok(s, L)) return 0;
    return attn_layers_plan(L, s->B, s->N, s->Hq, s->Hkv).total;
}

int gv_verify_attention_layers(const gv_attn_shape* s, int L, const void* q, int64_t q_layer_stride,
                               const void* k_new, int64_t k_layer_stride, const void* v_new, int64_t v_layer_stride,
                               const void* cacheK, const void* cacheV, int64_t cache_layer_stride,
                               const int32_t* prefix_len, const float* rope, const uint64_t* anc, void* treeK,
                               void* treeV, void* out, void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    if (!attn_layers_shape_ok(s, L)) {
        set_error("gv_verify_attention_layers: unsupported shape (bf16, d = 128, L >= 1, 1 <= B <= 64, "
                  "1 <= N <= 64, G * N <= 256, 8 L B N (Hq + 2 Hkv) <= 2^30 needed)");
        return s ? GV_ERR_UNSUPPORTED : GV_ERR_ARG;
    }
    const long long nq = (long long)s->B * s->N * s->Hq * 128, nk = (long long)s->B * s->N * s->Hkv * 128;
    const long long nc = (long long)s->B * s->Hkv * s->S_max * 128;
    GV_CHECK_ARG((L == 1 || (q_layer_stride >= nq && k_layer_stride >= nk && v_layer_stride >= nk &&
                             cache_layer_stride >= nc)) &&
                     q_layer_stride % 8 == 0 && k_layer_stride % 8 == 0 && v_layer_stride % 8 == 0 &&
                     cache_layer_stride % 8 == 0 && q_layer_stride >= 0 && k_layer_stride >= 0 &&
                     v_layer_stride >= 0 && cache_layer_stride >= 0,
                 "gv_verify_attention_layers: layer strides (elements) must cover a layer and be multiples of 8");
    const void* ptrs[] = {q, k_new, v_new, cacheK, cacheV, rope, treeK, treeV, out};
    for (const void* p : ptrs)
        GV_CHECK_ARG(p && aligned16(p), "gv_verify_attention_layers: tensor null or not 16-byte aligned");
    GV_CHECK_ARG(prefix_len && anc && ((uintptr_t)anc & 7u) == 0, "gv_verify_attention_layers: null index pointer");
    const AttnLayersPlan plan = attn_layers_plan(L, s->B, s->N, s->Hq, s->Hkv);
    GV_CHECK_ARG(workspace && ((uintptr_t)workspace & 255u) == 0,
                 "gv_verify_attention_layers: workspace null or not 256-byte aligned");
    GV_CHECK_ARG(ws_bytes >= plan.total, "gv_verify_attention_layers: workspace %zu < %zu bytes", ws_bytes,
                 plan.total);
    AttnLayersCall c{};
    c.L = L;
    c.B = s->B;
    c.N = s->N;
    c.Hq = s->Hq;
    c.Hkv = s->Hkv;
    c.S_max = s->S_max;
    c.q = q;
    c.q_ls = L == 1 ? nq : q_layer_stride;
    c.k_new = k_new;
    c.k_ls = L == 1 ? nk : k_layer_stride;
    c.v_new = v_new;
    c.v_ls = L == 1 ? nk : v_layer_stride;
    c.cacheK = cacheK;
    c.cacheV = cacheV;
    c.cache_ls = L == 1 ? nc : cache_layer_stride;
    c.prefix_len = prefix_len;
    c.rope = rope;
    c.anc = anc;
    c.treeK = treeK;
    c.treeV = treeV;
    c.out = out;
    c.workspace = workspace;
    return launch_attn_layers(c, as_stream(stream));
}

size_t gv_lmhead_workspace(int rows, int H, int V, int dt, int mode, int k) {
    if (rows < 1 || H < 1 || V < 1 || mode < 0 || mode > 2) return 0;
    if (mode == GV_SELECT_TOPK && (k < 1 || k > 16)) return 0;
    if (dt != GV_BF16 && dt != GV_F32) return 0;
    return lm_plan(rows, V, dt, mode, k).total;
}

int gv_lmhead_select(const void* h, const void* W, int rows, int H, int V, int dt, int mode, int k,
                     int32_t* ids, float* vals, float* logits, float* row_max, float* row_lse,
                     void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    GV_CHECK_ARG(rows >= 1 && H >= 1 && V >= 1, "gv_lmhead_select: rows=%d H=%d V=%d", rows, H, V);
    GV_CHECK_ARG(dt == GV_BF16 || dt == GV_F32, "gv_lmhead_select: dtype %d", dt);
    GV_CHECK_ARG(mode >= 0 && mode <= 2, "gv_lmhead_select: mode %d", mode);
    GV_CHECK_ARG(mode != GV_SELECT_TOPK || (k >= 1 && k <= 16), "gv_lmhead_select: k=%d", k);
    GV_CHECK_ARG(h && W && aligned16(h) && aligned16(W), "gv_lmhead_select: h/W null or unaligned");
    if (mode == GV_SELECT_LOGITS)
        GV_CHECK_ARG(logits, "gv_lmhead_select: logits output is null");
    else
        GV_CHECK_ARG(ids, "gv_lmhead_select: ids output is null");
    if (dt == GV_BF16)
        GV_CHECK_ARG(H % 8 == 0, "gv_lmhead_select: bf16 rows need H %% 8 == 0 (16-byte rows), H=%d", H);
    if (mode == GV_SELECT_LOGITS)
        GV_CHECK_ARG(aligned16(logits), "gv_lmhead_select: logits not 16-byte aligned");
    const LmPlan plan = lm_plan(rows, V, dt, mode, k);
    GV_CHECK_ARG(workspace && ((uintptr_t)workspace & 255u) == 0,
                 "gv_lmhead_select: workspace null or not 256-byte aligned");
    GV_CHECK_ARG(ws_bytes >= plan.total, "gv_lmhead_select: workspace %zu < %zu bytes", ws_bytes,
                 plan.total);
    char* ws = static_cast<char*>(workspace);
    SelectPartials part;
    part.val = reinterpret_cast<float*>(ws + plan.val);
    part.id = reinterpret_cast<int*>(ws + plan.id);
    part.m = reinterpret_cast<float*>(ws + plan.m);
    part.s = reinterpret_cast<float*>(ws + plan.s);
    part.slots = plan.slots;
    part.rows = rows;
    part.K = plan.K;
    cudaStream_t st = as_stream(stream);
    if (dt == GV_F32)
        return launch_lmhead_cc(static_cast<const float*>(h), static_cast<const float*>(W), rows, H,
                                V, mode, plan.K, logits, part, ids, vals, row_max, row_lse, st);
    int* err = reinterpret_cast<int*>(ws + plan.err);
    part.slots = lmhead_tc_grid(TC_SLOTS);
    int rc = launch_lmhead_tc(h, W, rows, H, V, mode, plan.K, logits, part, err, st);
    if (rc != GV_OK) return rc;
    return launch_lmhead_merge(part, mode, plan.K, ids, vals, row_max, row_lse, err, st);
}

int gv_lmhead_argmax_noalloc(const void* h, const void* W, int rows, int H, int V, int32_t* ids,
                             float* vals, void* stream) {
    clear_error();
    GV_CHECK_ARG(rows >= 1 && H >= 1 && V >= 1, "gv_lmhead_argmax_noalloc: rows=%d H=%d V=%d",
                 rows, H, V);
    if (rows > GV_NOALLOC_MAX_ROWS) {
        set_error("gv_lmhead_argmax_noalloc: rows=%d exceeds the fixed scratch (at most %d rows); "
                  "use gv_lmhead_select with a workspace", rows, GV_NOALLOC_MAX_ROWS);
        return GV_ERR_UNSUPPORTED;
    }
    GV_CHECK_ARG(h && W && aligned16(h) && aligned16(W),
                 "gv_lmhead_argmax_noalloc: h/W null or not 16-byte aligned");
    GV_CHECK_ARG(ids, "gv_lmhead_argmax_noalloc: ids output is null");
    GV_CHECK_ARG(H % 8 == 0, "gv_lmhead_argmax_noalloc: H %% 8 != 0 (16-byte rows), H=%d", H);
    char* ws = nullptr;
    int rc = noalloc_scratch(&ws);
    if (rc != GV_OK) return rc;
    SelectPartials part;
    part.val = reinterpret_cast<float*>(ws);
    part.id = reinterpret_cast<int*>(ws + NOALLOC_ID_OFF);
    part.m = nullptr;     // read and written only in GV_SELECT_LOGITS mode
    part.s = nullptr;
    part.slots = lmhead_tc_grid(TC_SLOTS);   // <= TC_SLOTS, so slots * rows fits
    part.rows = rows;
    part.K = 1;
    int* err = reinterpret_cast<int*>(ws + NOALLOC_ERR_OFF);
    cudaStream_t st = as_stream(stream);
    rc = launch_lmhead_tc(h, W, rows, H, V, GV_SELECT_ARGMAX, 1, nullptr, part, err, st);
    if (rc != GV_OK) return rc;
    return launch_lmhead_merge(part, GV_SELECT_ARGMAX, 1, ids, vals, nullptr, nullptr, err, st);
}

size_t gv_accept_workspace(int B, int V, float temperature) {
    if (B < 1) return 0;
    if (temperature == 0.0f) return 0;
    return align256((size_t)B * 2 * (size_t)V * sizeof(float));
}

int gv_accept(int B, int N, int D, int V, float temperature, const int32_t* tokens,
              const uint64_t* anc, const int32_t* depth, const int32_t* choice,
              const float* target_logits, const float* draft_logits, const float* u_acc,
              const float* u_res, int32_t* path, int32_t* accept_len, int32_t* out_tokens,
              int32_t* seq_status, void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    if (N < 1 || N > 64) {
        set_error("gv_accept: N=%d outside 1..64", N);
        return GV_ERR_INVALID_TREE;
    }
    GV_CHECK_ARG(B >= 1 && D >= 0, "gv_accept: B=%d D=%d", B, D);
    GV_CHECK_ARG(std::isfinite(temperature) && temperature >= 0.0f, "gv_accept: temperature %g",
                 (double)temperature);
    GV_CHECK_ARG(tokens && anc && depth && path && accept_len && out_tokens && seq_status,
                 "gv_accept: null pointer");
    if (temperature == 0.0f) {
        GV_CHECK_ARG(choice, "gv_accept: greedy acceptance needs choice");
    } else {
        GV_CHECK_ARG(V >= 1, "gv_accept: V=%d", V);
        GV_CHECK_ARG(target_logits && u_acc && u_res,
                     "gv_accept: sampling needs target logits and uniforms");
        GV_CHECK_ARG(workspace && ws_bytes >= gv_accept_workspace(B, V, temperature),
                     "gv_accept: workspace too small");
    }
    return launch_accept(B, N, D, V, temperature, tokens, anc, depth, choice, target_logits,
                         draft_logits, u_acc, u_res, path, accept_len, out_tokens, seq_status,
                         workspace, as_stream(stream));
}

int gv_kv_compact(int L, int B, int N, int D, int Hkv, int d, int S_max, int dt, const void* treeK,
                  const void* treeV, void* cacheK, void* cacheV, const int32_t* path,
                  const int32_t* accept_len, const int32_t* prefix_len, int32_t* new_len,
                  int32_t* seq_status, void* stream) {
    clear_error();
    GV_CHECK_ARG(L >= 1 && B >= 1 && N >= 1 && N <= 64 && D >= 0 && Hkv >= 1 && d >= 1 &&
                     S_max >= 1,
                 "gv_kv_compact: bad sizes");
    GV_CHECK_ARG(dt == GV_BF16 || dt == GV_F32, "gv_kv_compact: dtype %d", dt);
    const int esize = dt == GV_BF16 ? 2 : 4;
    GV_CHECK_ARG((d * esize) % 16 == 0, "gv_kv_compact: row of %d bytes is not a 16-byte multiple",
                 d * esize);
    const void* ptrs[] = {treeK, treeV, cacheK, cacheV};
    for (const void* p : ptrs)
        GV_CHECK_ARG(p && aligned16(p), "gv_kv_compact: tensor null or not 16-byte aligned");
    GV_CHECK_ARG(path && accept_len && prefix_len && new_len && seq_status,
                 "gv_kv_compact: null index pointer");
    return launch_kv_compact(L, B, N, D, Hkv, d, S_max, esize, treeK, treeV, cacheK, cacheV, path,
                             accept_len, prefix_len, new_len, seq_status, as_stream(stream));
}

size_t gv_linear_workspace(int rows, int K, int n_out, int epilogue) {
    if (rows < 1 || rows > 256 || K < 8 || n_out < 8) return 0;
    if (epilogue < GV_LINEAR_STORE || epilogue > GV_LINEAR_SILU) return 0;
    const int N = epilogue == GV_LINEAR_SWIGLU ? 2 * n_out : n_out;
    return align256(linear_workspace_bytes(rows, K, N));
}

int gv_linear(const void* x, const void* W, int rows, int K, int n_out, int epilogue,
              const void* residual, void* out, void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    GV_CHECK_ARG(rows >= 1 && rows <= 256, "gv_linear: rows=%d outside 1..256", rows);
    GV_CHECK_ARG(K >= 8 && K % 8 == 0 && n_out >= 8 && n_out % 8 == 0,
                 "gv_linear: K=%d and n_out=%d must be positive multiples of 8", K, n_out);
    GV_CHECK_ARG(epilogue >= GV_LINEAR_STORE && epilogue <= GV_LINEAR_SILU, "gv_linear: epilogue %d",
                 epilogue);
    GV_CHECK_ARG(x && W && out && workspace, "gv_linear: null pointer");
    GV_CHECK_ARG(aligned16(x) && aligned16(W) && aligned16(out), "gv_linear: pointers not 16-byte aligned");
    GV_CHECK_ARG((epilogue == GV_LINEAR_ADD) == (residual != nullptr),
                 "gv_linear: residual is required by GV_LINEAR_ADD and only by it");
    GV_CHECK_ARG(!residual || aligned16(residual), "gv_linear: residual not 16-byte aligned");
    GV_CHECK_ARG(ws_bytes >= gv_linear_workspace(rows, K, n_out, epilogue) && aligned16(workspace),
                 "gv_linear: workspace too small or misaligned");
    LinearOp op;
    op.x = x;
    op.W = W;
    op.rows = rows;
    op.K = K;
    op.n_out = n_out;
    op.epi = epilogue;
    op.residual = residual;
    op.out = out;
    op.ws = workspace;
    return launch_linear(op, as_stream(stream));
}

size_t gv_linear_qkv_workspace(int rows, int K, int n_q, int n_kv) {
    return gv_linear_workspace(rows, K, n_q + 2 * n_kv, GV_LINEAR_STORE);
}

int gv_linear_qkv(const void* x, const void* Wqkv, int rows, int K, int n_q, int n_kv, void* q, void* k, void* v,
                  void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    GV_CHECK_ARG(rows >= 1 && rows <= 256, "gv_linear_qkv: rows=%d outside 1..256", rows);
    GV_CHECK_ARG(K >= 8 && K % 8 == 0 && n_q >= 8 && n_q % 8 == 0 && n_kv >= 8 && n_kv % 8 == 0,
                 "gv_linear_qkv: K=%d, n_q=%d, n_kv=%d must be positive multiples of 8", K, n_q, n_kv);
    GV_CHECK_ARG(x && Wqkv && q && k && v && workspace, "gv_linear_qkv: null pointer");
    GV_CHECK_ARG(aligned16(x) && aligned16(Wqkv) && aligned16(q) && aligned16(k) && aligned16(v) &&
                     aligned16(workspace),
                 "gv_linear_qkv: pointers not 16-byte aligned");
    GV_CHECK_ARG(ws_bytes >= gv_linear_qkv_workspace(rows, K, n_q, n_kv), "gv_linear_qkv: workspace too small");
    LinearOp op;
    op.x = x;
    op.W = Wqkv;
    op.rows = rows;
    op.K = K;
    op.n_out = n_q + 2 * n_kv;
    op.out = q;
    op.out1 = k;
    op.out2 = v;
    op.n0 = n_q;
    op.n1 = n_kv;
    op.ws = workspace;
    return launch_linear(op, as_stream(stream));
}

int gv_linear_add_rmsnorm(const void* x, const void* W, int rows, int K, int n_out, const void* residual,
                          void* out, const void* norm_w, float eps, void* norm_out, void* workspace, size_t ws_bytes,
                          void* stream) {
    clear_error();
    GV_CHECK_ARG(rows >= 1 && rows <= 256, "gv_linear_add_rmsnorm: rows=%d outside 1..256", rows);
    GV_CHECK_ARG(K >= 8 && K % 8 == 0 && n_out >= 8 && n_out % 8 == 0 && n_out <= 8192,
                 "gv_linear_add_rmsnorm: K=%d, n_out=%d (multiples of 8, n_out <= 8192)", K, n_out);
    GV_CHECK_ARG(std::isfinite(eps) && eps >= 0.0f, "gv_linear_add_rmsnorm: eps %g", (double)eps);
    GV_CHECK_ARG(x && W && residual && out && norm_w && norm_out && workspace, "gv_linear_add_rmsnorm: null pointer");
    GV_CHECK_ARG(aligned16(x) && aligned16(W) && aligned16(residual) && aligned16(out) && aligned16(norm_w) &&
                     aligned16(norm_out) && aligned16(workspace),
                 "gv_linear_add_rmsnorm: pointers not 16-byte aligned");
    GV_CHECK_ARG(norm_out != out && norm_out != residual, "gv_linear_add_rmsnorm: norm_out must be its own buffer");
    GV_CHECK_ARG(ws_bytes >= gv_linear_workspace(rows, K, n_out, GV_LINEAR_ADD),
                 "gv_linear_add_rmsnorm: workspace too small");
    LinearOp op;
    op.x = x;
    op.W = W;
    op.rows = rows;
    op.K = K;
    op.n_out = n_out;
    op.epi = GV_LINEAR_ADD;
    op.residual = residual;
    op.out = out;
    op.norm_w = norm_w;
    op.eps = eps;
    op.norm_out = norm_out;
    op.ws = workspace;
    return launch_linear(op, as_stream(stream));
}

int gv_rmsnorm(const void* x, const void* w, int rows, int H, float eps, void* out, void* stream) {
    clear_error();
    GV_CHECK_ARG(rows >= 1 && H >= 8 && H % 8 == 0, "gv_rmsnorm: rows=%d H=%d (H a multiple of 8)", rows, H);
    GV_CHECK_ARG(std::isfinite(eps) && eps >= 0.0f, "gv_rmsnorm: eps %g", (double)eps);
    GV_CHECK_ARG(x && w && out, "gv_rmsnorm: null pointer");
    GV_CHECK_ARG(aligned16(x) && aligned16(w) && aligned16(out), "gv_rmsnorm: pointers not 16-byte aligned");
    return launch_rmsnorm(x, w, rows, H, eps, out, as_stream(stream));
}

size_t gv_tgf_workspace(int rows, int d, int e) {
    if (rows < 1 || rows > 256 || d < 64 || d % 64 != 0 || d > 8192 || e < 8 || e % 8 != 0) return 0;
    return align256(tgf_workspace_bytes(rows, d, e));
}

int gv_tgf(const void* F, const void* x, int rows, int d, int e, const void* Wm, const void* bm, const void* g_h,
           const void* b_h, const void* g_x, const void* b_x, const void* Wu, const void* bu, const void* Wd,
           const void* bd, float eps, void* h_out, void* o_out, void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    GV_CHECK_ARG(rows >= 1 && rows <= 256, "gv_tgf: rows=%d outside 1..256", rows);
    GV_CHECK_ARG(d >= 64 && d % 64 == 0 && d <= 8192, "gv_tgf: d=%d (a multiple of 64, at most 8192)", d);
    GV_CHECK_ARG(e >= 8 && e % 8 == 0, "gv_tgf: e=%d (a positive multiple of 8)", e);
    GV_CHECK_ARG(std::isfinite(eps) && eps >= 0.0f, "gv_tgf: eps %g", (double)eps);
    const void* ptrs[] = {F, x, Wm, bm, g_h, b_h, g_x, b_x, Wu, bu, Wd, bd, h_out, o_out, workspace};
    for (const void* p : ptrs) GV_CHECK_ARG(p && aligned16(p), "gv_tgf: tensor null or not 16-byte aligned");
    GV_CHECK_ARG(h_out != o_out, "gv_tgf: h_out and o_out must be separate buffers");
    GV_CHECK_ARG(ws_bytes >= gv_tgf_workspace(rows, d, e), "gv_tgf: workspace too small");
    return launch_tgf(F, x, rows, d, e, Wm, bm, g_h, b_h, g_x, b_x, Wu, bu, Wd, bd, eps, h_out, o_out, workspace,
                      as_stream(stream));
}

static bool draft_tree_shape_ok(int B, int k, int D, int V) {
    if (B < 1 || k < 1 || k > 16 || D < 1 || D > 16 || V < k || V > 262144) return false;
    return 1 + k + (long)(D - 1) * k * k <= 4096;
}

size_t gv_draft_tree_workspace(int B, int k, int D, int V) {
    if (!draft_tree_shape_ok(B, k, D, V)) return 0;
    return align256(draft_tree_workspace_bytes(B, k, D, V));
}

int gv_draft_tree_expand(int B, int k, int D, int V, int step, int dt, const int32_t* root_token,
                         const void* logits, int32_t* exp_token, int32_t* exp_pool, void* workspace,
                         size_t ws_bytes, void* stream) {
    clear_error();
    GV_CHECK_ARG(draft_tree_shape_ok(B, k, D, V),
                 "gv_draft_tree_expand: B=%d k=%d D=%d V=%d (1 <= k <= 16, 1 <= D <= 16, k <= V <= 262144, "
                 "1 + k + (D-1) k^2 <= 4096)", B, k, D, V);
    GV_CHECK_ARG(step >= 0 && step < D, "gv_draft_tree_expand: step %d outside 0..%d", step, D - 1);
    GV_CHECK_ARG(dt == GV_F32 || dt == GV_BF16, "gv_draft_tree_expand: logits dtype %d", dt);
    GV_CHECK_ARG(logits && workspace, "gv_draft_tree_expand: null pointer");
    GV_CHECK_ARG(step > 0 || root_token, "gv_draft_tree_expand: step 0 needs root_token");
    GV_CHECK_ARG(ws_bytes >= gv_draft_tree_workspace(B, k, D, V) && aligned16(workspace),
                 "gv_draft_tree_expand: workspace too small or misaligned");
    return launch_draft_tree_expand(B, k, D, V, step, dt, root_token, logits, exp_token, exp_pool, workspace,
                                    as_stream(stream));
}

int gv_draft_tree_finish(int B, int k, int D, int V, int N, int32_t* parents, int32_t* tokens, void* workspace,
                         size_t ws_bytes, void* stream) {
    clear_error();
    GV_CHECK_ARG(draft_tree_shape_ok(B, k, D, V), "gv_draft_tree_finish: B=%d k=%d D=%d V=%d", B, k, D, V);
    const int P = 1 + k + (D - 1) * k * k;
    GV_CHECK_ARG(N >= 1 && N <= P && N <= 64, "gv_draft_tree_finish: N=%d outside 1..min(64, %d)", N, P);
    GV_CHECK_ARG(parents && tokens && workspace, "gv_draft_tree_finish: null pointer");
    GV_CHECK_ARG(ws_bytes >= gv_draft_tree_workspace(B, k, D, V), "gv_draft_tree_finish: workspace too small");
    return launch_draft_tree_finish(B, k, D, N, parents, tokens, workspace, as_stream(stream));
}

int gv_tat_loss(const void* logits, int logits_dt, const int32_t* tokens, const void* feat_draft,
                const void* feat_target, int feat_dt, int B, int T, int V, int H, int k, int n,
                const uint8_t* mbar_prev, float lambda_tok, float lambda_feat, uint8_t* mbar,
                uint8_t* mask, float* ell, float* seq_loss, void* stream) {
    clear_error();
    GV_CHECK_ARG(B >= 1 && T >= 1 && V >= 1 && H >= 0 && n >= 1 && k >= 1 && k <= V,
                 "gv_tat_loss: bad sizes (B %d, T %d, V %d, H %d, k %d, n %d)", B, T, V, H, k, n);
    GV_CHECK_ARG((long long)B * T <= 0x7fffffffLL, "gv_tat_loss: B * T too large");
    GV_CHECK_ARG(logits_dt == GV_BF16 || logits_dt == GV_F32, "gv_tat_loss: logits dtype %d", logits_dt);
    GV_CHECK_ARG(feat_dt == GV_BF16 || feat_dt == GV_F32, "gv_tat_loss: feature dtype %d", feat_dt);
    GV_CHECK_ARG(logits && tokens && mbar && mask && ell && seq_loss, "gv_tat_loss: null pointer");
    GV_CHECK_ARG(H == 0 || (feat_draft && feat_target), "gv_tat_loss: null feature pointer");
    GV_CHECK_ARG((n == 1) == (mbar_prev == nullptr), "gv_tat_loss: mbar_prev must be NULL iff n == 1");
    return launch_tat_loss(logits, logits_dt, tokens, feat_draft, feat_target, feat_dt, B, T, V, H, k, n,
                           mbar_prev, lambda_tok, lambda_feat, mbar, mask, ell, seq_loss, as_stream(stream));
}

}  // extern "C"
