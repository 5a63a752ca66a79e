/*
 * gv.h -- C ABI of the GB300 draft-tree verification library (libgv.so).
 *
 * One verify step of GRIFFIN-style speculative decoding (arXiv 2502.11018):
 * the draft model proposes a tree of tokens, the target model verifies all of
 * them in a single forward pass and accepts a subset (Section 3, the
 * draft-and-verify cycle; Appendix C, the dynamic draft tree of 60 tokens).
 * The calls below are that pass's data-parallel steps, in order:
 *
 *   gv_tree_build        positions and ancestor bitmasks from a parent array
 *   gv_rope_table        RoPE cos/sin of every node (shared by all layers)
 *   gv_rope_apply        (optional) the rotation of every layer's tree
 *                        queries and keys, ahead of the attention calls
 *   gv_verify_attention  tree-masked attention of one layer (call per layer;
 *                        or its halves gv_verify_attention_split / _merge)
 *   gv_lmhead_select     LM-head projection fused with argmax / top-k / logits
 *   gv_accept            longest accepted root chain (T = 0) or recursive
 *                        rejection sampling (T > 0)
 *   gv_kv_compact        commit the accepted chain's K/V into the cache
 *
 * the target model's layer body around the attention (the rest of the verify
 * forward pass of Section 3, for LLaMA-style targets):
 *
 *   gv_rmsnorm           RMSNorm of the node rows
 *   gv_linear            skinny projection x W^T with a fused epilogue
 *   gv_linear_qkv        the Q, K and V projections as one weight stream
 *   gv_linear_add_rmsnorm  a residual projection fused with the next RMSNorm
 *
 * and, for the draft model (Section 4):
 *
 *   gv_tat_loss          top-k predictable masks, chain alignment masks and
 *                        the masked loss of one token-alignable training pass
 *   gv_tgf               the Token-Guided Fusion module (Eqs. 6-8)
 *   gv_draft_tree_expand / gv_draft_tree_finish
 *                        the dynamic draft tree: top-k expansion steps and
 *                        the rerank into the tree the verify pass takes
 *
 * Conventions shared by every call:
 *  - Every pointer argument is DEVICE memory owned by the caller, unless the
 *    argument says otherwise.  The library never allocates on these paths:
 *    scratch memory is queried with the matching *_workspace call and passed
 *    in.  The library keeps no state between calls (the only persistent state
 *    of a decoding loop is the caller's cache and prefix lengths).
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Calls only enqueue work; they are asynchronous with respect to
 *    the host and can be captured into a CUDA graph.
 *  - Return value: a gv_status.  Argument errors the host can see (null
 *    pointers, bad sizes, misalignment, unsupported shapes) return
 *    synchronously before anything is enqueued.  A CUDA launch error returns
 *    GV_ERR_CUDA (text from gv_last_error()).  Data-dependent errors (an
 *    invalid parent array, cache overflow) cannot be seen by the host without
 *    a synchronisation; they are written to the per-sequence status array
 *    `seq_status[B]` on the device, and every later call that takes
 *    `seq_status` leaves a sequence whose status is non-zero untouched.
 *  - Index layouts are row-major with the last index contiguous.  Node 0 of
 *    every tree is the root (the last committed token, whose K/V is not yet
 *    in the cache); nodes are in topological order, parents[i] < i.
 *  - Limits: 1 <= N <= 64 nodes per tree; head dim d in {64, 128}; Hq a
 *    multiple of Hkv.
 */
#ifndef GV_H
#define GV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    GV_OK = 0,
    GV_ERR_ARG = -1,          /* bad pointer, size, alignment or mode          */
    GV_ERR_INVALID_TREE = -2, /* parent array breaks the topological rule, or
                                 a node is deeper than the caller's D         */
    GV_ERR_CAPACITY = -3,     /* prefix_len + accept_len would exceed S_max    */
    GV_ERR_UNSUPPORTED = -4,  /* shape outside the supported limits, or no
                                 sm_103 device                                */
    GV_ERR_CUDA = -5,         /* a CUDA runtime call failed                    */
    GV_ERR_TIMEOUT = -6       /* a bounded device-side wait gave up            */
} gv_status;

typedef enum { GV_BF16 = 0, GV_F32 = 1 } gv_dtype;

typedef enum {
    GV_SELECT_ARGMAX = 0,     /* ids[rows], vals[rows] = max logit             */
    GV_SELECT_TOPK = 1,       /* ids[rows][k], vals[rows][k], k <= 16          */
    GV_SELECT_LOGITS = 2      /* logits[rows][V] fp32, row_max[rows], row_lse[rows] */
} gv_select_mode;

/* Epilogues of gv_linear. */
typedef enum {
    GV_LINEAR_STORE = 0,   /* out = x W^T                                   */
    GV_LINEAR_ADD = 1,     /* out = residual + x W^T (out may be residual)  */
    GV_LINEAR_SWIGLU = 2,  /* out = silu(x Wg^T) * (x Wu^T), W = [Wg ; Wu]  */
    GV_LINEAR_SILU = 3     /* out = silu(x W^T)                             */
} gv_linear_epilogue;

/* Shape of one attention layer of the verify pass. */
typedef struct {
    int B;            /* sequences                                            */
    int N;            /* tree nodes per sequence, root included (<= 64)       */
    int Hq;           /* query heads                                          */
    int Hkv;          /* key/value heads (Hq % Hkv == 0; GQA when Hq > Hkv)   */
    int d;            /* head dimension (64 or 128)                           */
    int S_max;        /* cache rows per (sequence, KV head)                   */
    gv_dtype dt;      /* GV_BF16 (tensor-core path) or GV_F32                 */
} gv_attn_shape;

/*
 * gv_tree_build -- depths, RoPE positions and ancestor bitmasks of B trees.
 * Section 4.1: a rejected draft token takes every later token of its draft
 * sequence with it, so the ancestor-or-self set of a node is what decides both
 * its attention mask and its acceptance; Appendix C: dynamic tree, <= 64 nodes.
 *
 *   parents    int32 [B][N]  parent index per node; parents[b][0] == -1 and
 *                            0 <= parents[b][i] < i for i >= 1
 *   prefix_len int32 [B]     cached tokens per sequence (P_b)
 *   depth      int32 [B][N]  out: edges from the root
 *   pos        int32 [B][N]  out: P_b + depth (RoPE position)
 *   anc        uint64[B][N]  out: bit j set iff node j is on the root-to-i chain
 *   seq_status int32 [B]     out: GV_OK, or GV_ERR_INVALID_TREE for a parent
 *                            array that breaks the rule above; such a tree gets
 *                            depth 0, pos P_b and anc[i] = 1 << i.
 * Returns GV_ERR_INVALID_TREE synchronously when N < 1 or N > 64.
 */
int gv_tree_build(const int32_t* parents, const int32_t* prefix_len, int B, int N,
                  int32_t* depth, int32_t* pos, uint64_t* anc, int32_t* seq_status,
                  void* stream);

/*
 * gv_rope_table -- RoPE cos/sin of every tree node, once per verify step.
 * Every layer of the verify forward pass (Section 3) rotates the draft
 * tokens' queries and keys at the same positions, so the angles are formed
 * once: rope[b][i][j] = {cos(a), sin(a)} with a = pos[b][i] * rope_base^(-2j/d)
 * for j < d/2 (rotate-half RoPE).  The angle is formed and reduced modulo
 * 2 pi in double; cos and sin of the remainder are within 3e-7 of the exact
 * values, stored as fp32.
 *
 *   pos   int32 [B][N]          from gv_tree_build
 *   rope  fp32  [B][N][d/2][2]  out
 * d must be even, 2 <= d <= 256.
 */
int gv_rope_table(const int32_t* pos, int B, int N, int d, float rope_base, float* rope,
                  void* stream);

/*
 * gv_verify_attention -- one attention layer of the verify forward pass.
 * Section 3: the target model verifies all draft tokens in one forward pass.
 * Draft node i of sequence b, query head h, attends to the cached prefix rows
 * 0..P_b-1 of KV head g = h / (Hq/Hkv) and to the tree nodes j with bit j of
 * anc[b][i] set, which equals causal attention over [prefix ; root chain of i].
 * RoPE (rotate-half) is applied to q and k_new of node i with the cos/sin of
 * rope[b][i] from gv_rope_table; softmax scale is 1/sqrt(d).
 *
 *   q          [B][N][Hq][d]      tree queries, unrotated           (dt)
 *   k_new      [B][N][Hkv][d]     tree keys, unrotated              (dt)
 *   v_new      [B][N][Hkv][d]     tree values                       (dt)
 *   cacheK/V   [B][Hkv][S_max][d] cache of this layer; rows < P_b are
 *                                 read (keys stored already rotated)  (dt)
 *   prefix_len int32 [B]          P_b <= S_max
 *   rope       fp32 [B][N][d/2][2] from gv_rope_table; or NULL (bf16 only)
 *                                 when q and k_new arrive already rotated
 *                                 (gv_rope_apply: the same arithmetic, so the
 *                                 results are bit-identical)
 *   anc        uint64 [B][N]       from gv_tree_build
 *   treeK/V    [B][Hkv][N][d]     out: rotated tree keys / the values, the
 *                                 scratch gv_kv_compact reads        (dt)
 *   out        [B][N][Hq][d]      out: attention output              (dt)
 *   workspace  >= gv_verify_attention_workspace(s) bytes, 256-byte aligned;
 *              contents need no initialisation and are clobbered.
 * All tensors 16-byte aligned.  Two calls that share a workspace must be
 * ordered on the device (same stream or an event between them).
 */
size_t gv_verify_attention_workspace(const gv_attn_shape* s);
/*
 * gv_rope_apply -- the RoPE rotation gv_verify_attention applies to its tree
 * queries and keys, done ahead of time for L layers at once (bf16, d = 128):
 * q_out[l] = RoPE(q[l]), k_out[l] = RoPE(k_new[l]) with the cos/sin of
 * rope[b][i] (gv_rope_table).  Layer l of the inputs starts at
 * q + l * q_layer_stride (and k_new + l * k_layer_stride) elements; the
 * outputs are packed [L][B][N][Hq][d] and [L][B][N][Hkv][d].  Feeding them to
 * gv_verify_attention with rope = NULL gives the same results as the
 * unrotated inputs with the table.
 */
int gv_rope_apply(const gv_attn_shape* s, int L, const void* q, size_t q_layer_stride, const void* k_new,
                  size_t k_layer_stride, const float* rope, void* q_out, void* k_out, void* stream);

int gv_verify_attention(const gv_attn_shape* s, const void* q, const void* k_new,
                        const void* v_new, const void* cacheK, const void* cacheV,
                        const int32_t* prefix_len, const float* rope, const uint64_t* anc,
                        void* treeK, void* treeV, void* out,
                        void* workspace, size_t ws_bytes, void* stream);

/*
 * gv_verify_attention_split / gv_verify_attention_merge -- the two halves of
 * gv_verify_attention, for callers that schedule them apart.  split takes
 * gv_verify_attention's arguments and launches the key-split kernels: their
 * partial rows go to the workspace, or, when the shape has a single split,
 * the final rows to `out`.  merge combines the partial rows into `out` (a
 * no-op for a single split); it reads only the workspace.  Run in that order
 * (e.g. the merge on a second stream that waits for the split), the pair
 * gives gv_verify_attention's results bit for bit; the workspace belongs to
 * the pair until the merge has completed.  A verify step whose layers take
 * their queries, keys and values as inputs needs no layer's merged output
 * before the next layer's split: it can run the merges beside the splits,
 * with a workspace per layer in flight.
 */
int gv_verify_attention_split(const gv_attn_shape* s, const void* q, const void* k_new, const void* v_new,
                              const void* cacheK, const void* cacheV, const int32_t* prefix_len, const float* rope,
                              const uint64_t* anc, void* treeK, void* treeV, void* out, void* workspace,
                              size_t ws_bytes, void* stream);
int gv_verify_attention_merge(const gv_attn_shape* s, void* out, void* workspace, size_t ws_bytes, void* stream);

/*
 * gv_verify_attention_layers -- the tree attention of L layers in one call.
 * Section 3: one target forward pass verifies every draft token; when the
 * caller holds the tree queries, keys and values of several layers at once
 * (a verify step whose layers' inputs are given), their attentions are
 * independent problems and run as one persistent launch.  The results equal
 * L calls of gv_verify_attention (same rotation, mask and softmax; the
 * combination of partial results may round differently in the last bf16
 * bit).  Layer l of an input starts l * (its layer stride) elements after its
 * pointer; the outputs are packed by layer.
 *
 *   q          [L][B][N][Hq][d]      tree queries, unrotated, stride q_layer_stride
 *   k_new      [L][B][N][Hkv][d]     tree keys, unrotated, stride k_layer_stride
 *   v_new      [L][B][N][Hkv][d]     tree values, stride v_layer_stride
 *   cacheK/V   [L][B][Hkv][S_max][d] caches, stride cache_layer_stride; rows
 *                                    < P_b are read (keys stored rotated)
 *   prefix_len int32 [B], rope fp32 [B][N][d/2][2] (gv_rope_table), anc
 *                                    uint64 [B][N] (gv_tree_build)
 *   treeK/V    [L][B][Hkv][N][d]     out: rotated tree keys / the values
 *                                    (what gv_kv_compact reads)
 *   out        [L][B][N][Hq][d]      out: attention outputs
 *   workspace  >= gv_verify_attention_layers_workspace(s, L) bytes, 256-byte
 *              aligned; contents need no initialisation and are clobbered.
 * bf16 only, d = 128, 1 <= B <= 64, N <= 64, (Hq/Hkv) * N <= 256 and
 * 8 L B N (Hq + 2 Hkv) <= 2^30 (else GV_ERR_UNSUPPORTED); strides are element
 * counts, multiples of 8, each at least one layer (ignored for L = 1).  All tensors 16-byte aligned.  Two
 * calls that share a workspace must be ordered on the device.  A bounded
 * device-side wait that gives up turns the affected output rows into NaN.
 */
size_t gv_verify_attention_layers_workspace(const gv_attn_shape* s, int L);
int gv_verify_attention_layers(const gv_attn_shape* s, int L, const void* q, int64_t q_layer_stride,
                               const void* k_new, int64_t k_layer_stride, const void* v_new,
                               int64_t v_layer_stride, const void* cacheK, const void* cacheV,
                               int64_t cache_layer_stride, const int32_t* prefix_len, const float* rope,
                               const uint64_t* anc, void* treeK, void* treeV, void* out, void* workspace,
                               size_t ws_bytes, void* stream);

/*
 * gv_lmhead_select -- LM head fused with the per-node selection.
 * Section 3 / Eq. 1: the LM head maps a final hidden feature to a token;
 * Section 4.1 ranks candidates by their top-k; Section 5 decodes at T in {0,1}.
 * logits[r][v] = sum_k h[r][k] * W[v][k], accumulated in fp32.
 *
 *   h        [rows][H]   final hidden states of the tree nodes     (dt)
 *   W        [V][H]      LM-head weight, row-major                 (dt)
 *   mode GV_SELECT_ARGMAX: ids int32[rows] = argmax (lowest id on ties),
 *                          vals fp32[rows] = its logit; no logits are written
 *                          to memory.
 *   mode GV_SELECT_TOPK:   ids int32[rows][k], vals fp32[rows][k], by
 *                          decreasing logit, lower id first on ties; 1<=k<=16.
 *   mode GV_SELECT_LOGITS: logits fp32[rows][V], row_max fp32[rows],
 *                          row_lse fp32[rows] = max + log(sum exp(l - max)).
 *   Unused outputs may be NULL.
 *   workspace >= gv_lmhead_workspace(rows, H, V, dt, mode, k) bytes.
 * H must be a multiple of 8 (bf16) or 4 (fp32); rows >= 1.
 * Device-side timeout (bf16 path): every wait inside the kernel is bounded
 * (about a second); a kernel that gives up does not fault, and the call still
 * returns GV_OK (it was enqueued), but its results mark the failure once the
 * stream has run: ids = -1 and vals = NaN (argmax, top-k), row_max = row_lse
 * = NaN (logits).  A caller that cannot rule this out checks for ids < 0 (or
 * NaN) before passing the ids on, e.g. to gv_accept.
 */
size_t gv_lmhead_workspace(int rows, int H, int V, int dt, int mode, int k);
int gv_lmhead_select(const void* h, const void* W, int rows, int H, int V, int dt, int mode,
                     int k, int32_t* ids, float* vals, float* logits, float* row_max,
                     float* row_lse, void* workspace, size_t ws_bytes, void* stream);

/*
 * gv_lmhead_argmax_noalloc -- gv_lmhead_select(mode GV_SELECT_ARGMAX, bf16)
 * without a workspace argument.  The paper has no counterpart: it exists for
 * callers that cannot allocate or hold device memory of their own for
 * scratch, e.g. an embedding runtime whose memory is fixed once at start-up,
 * or a caller outside PyTorch's allocator that has only the inputs and
 * outputs.  Same arithmetic and kernels as gv_lmhead_select; ids/vals equal.
 *
 *   h [rows][H] bf16, W [V][H] bf16, ids int32[rows], vals fp32[rows] (may
 *   be NULL); 1 <= rows <= GV_NOALLOC_MAX_ROWS, H a multiple of 8.
 *
 * Scratch: a fixed 512 KB + 1 KB array in the library's own device memory
 * (a file-scope __device__ array, one per device, reserved when the library
 * is loaded): per-CTA argmax partials of up to GV_NOALLOC_MAX_ROWS rows and
 * per-CTA status words, which each call's projection kernel rewrites (no
 * memset precedes its kernels).
 * Every call looks the array's address up (cudaGetSymbolAddress, which
 * allocates nothing), so a reset or replaced context is handled; make the
 * first call on a device before any stream capture (the lookup itself is not
 * captured).  Nothing is allocated by any call.
 * rows > GV_NOALLOC_MAX_ROWS returns GV_ERR_UNSUPPORTED (message in
 * gv_last_error()), before anything is enqueued.
 * Calls that overlap in time on one device (different streams, or host
 * threads without ordering) share the scratch and race: serialise them.
 * Device-side timeout: as for gv_lmhead_select, ids = -1 and vals = NaN.
 */
#define GV_NOALLOC_MAX_ROWS 256
int gv_lmhead_argmax_noalloc(const void* h, const void* W, int rows, int H, int V,
                             int32_t* ids, float* vals, void* stream);

/*
 * gv_accept -- accept the longest verified root chain of each tree.
 * Section 3: the target accepts a subset of the drafts; Section 4.1: a
 * rejected token discards its whole subtree; Section 5: lossless at T = 0 and
 * T = 1.
 *
 * temperature == 0 (greedy): node j > 0 matches when
 *   tokens[b][j] == choice[b*N + parent(j)]; the accepted node is the deepest
 *   node whose whole root chain matches (smallest index among equals).
 * temperature > 0: multi-draft recursive rejection sampling.  From the root:
 *   p = softmax(target_logits[b][u] / T), q = softmax(draft_logits[b][u] / T);
 *   children c of u in increasing index are accepted when
 *   u_acc[b][c] <= p(x_c) / q(x_c) (always when q(x_c) == 0), otherwise
 *   p <- max(p - q, 0) / sum(max(p - q, 0)) (kept if that sum is 0); when no
 *   child is accepted the bonus token is the smallest v with
 *   sum_{w<=v} p(w) > u_res[b][u] * sum(p).
 * temperature > 0 and draft_logits == NULL: the drafts are deterministic
 *   proposals (top-k, EAGLE style): q(x_c) is taken as 1, so c is accepted
 *   when u_acc[b][c] <= p(x_c), and a rejection sets p(x_c) = 0 and
 *   renormalises p (kept if nothing is left); the bonus is drawn as above.
 *
 *   tokens        int32 [B][N]      draft token per node (tokens[b][0] = root)
 *   anc, depth    from gv_tree_build
 *   choice        int32 [B*N]       target argmax per node (T == 0; else NULL)
 *   target_logits fp32  [B][N][V]   (T > 0; else NULL)
 *   draft_logits  fp32  [B][N][V]   (T > 0, or NULL for the q = 1 rule; NULL for T == 0)
 *   u_acc, u_res  fp32  [B][N]      uniforms in [0, 1) (T > 0; else NULL)
 *   path          int32 [B][D+1]    out: accepted chain, root first, -1 padded
 *   accept_len    int32 [B]         out: entries of path (1 .. D+1)
 *   out_tokens    int32 [B][D+1]    out: accepted drafts then the bonus token
 *   seq_status    int32 [B]         in/out: non-zero sequences are skipped
 *                                   (accept_len 0, rows of -1); a tree with a
 *                                   node deeper than D gets GV_ERR_INVALID_TREE.
 *   workspace >= gv_accept_workspace(B, V, temperature) bytes (0 for T == 0).
 */
size_t gv_accept_workspace(int B, int V, float temperature);
int gv_accept(int B, int N, int D, int V, float temperature, const int32_t* tokens,
              const uint64_t* anc, const int32_t* depth, const int32_t* choice,
              const float* target_logits, const float* draft_logits, const float* u_acc,
              const float* u_res, int32_t* path, int32_t* accept_len, int32_t* out_tokens,
              int32_t* seq_status, void* workspace, size_t ws_bytes, void* stream);

/*
 * gv_kv_compact -- append the accepted chain's K/V to every layer's cache.
 * Section 4.1: only the accepted chain survives verification.  For every
 * layer l, sequence b, KV head h and t < accept_len[b]:
 *   cache[l][b][h][P_b + t][:] = tree[l][b][h][path[b][t]][:]
 * and new_len[b] = P_b + accept_len[b].  Nothing else is written.
 *
 *   treeK/V    [L][B][Hkv][N][d]      tree scratch of every layer   (dt)
 *   cacheK/V   [L][B][Hkv][S_max][d]  caches, updated in place       (dt)
 *   path       int32 [B][D+1], accept_len int32 [B] from gv_accept
 *   prefix_len int32 [B]
 *   new_len    int32 [B]   out
 *   seq_status int32 [B]   in/out: non-zero sequences are left untouched
 *                          (new_len = P_b); P_b + accept_len > S_max sets
 *                          GV_ERR_CAPACITY and writes nothing for that sequence.
 * Rows must be 16-byte multiples (d * sizeof(dt) % 16 == 0).
 */
int gv_kv_compact(int L, int B, int N, int D, int Hkv, int d, int S_max, int dt,
                  const void* treeK, const void* treeV, void* cacheK, void* cacheV,
                  const int32_t* path, const int32_t* accept_len, const int32_t* prefix_len,
                  int32_t* new_len, int32_t* seq_status, void* stream);

/*
 * gv_tat_loss -- the draft model's token-alignable training objective for
 * training pass n (Section 4.1, Eqs. 2-5; per-step loss of the Implementation
 * Details appendix).  Not part of the verify step: a data-parallel pass over
 * the draft model's logits for a batch of training sequences.
 *
 *   logits      [B][T][V]    draft logits Xd_t                  (logits_dt)
 *   tokens      int32 [B][T] ground-truth tokens x_t, 0 <= x_t < V
 *   feat_draft  [B][T][H]    draft features Fd_t                (feat_dt)
 *   feat_target [B][T][H]    target features Ft_t               (feat_dt)
 *   mbar_prev   uint8 [n-1][B][T]  predictable masks of passes 1 .. n-1
 *                            (the mbar outputs of those passes); NULL iff n == 1
 *   mbar        uint8 [B][T] out: 1 iff x_t is among the top-k of Xd_t (ties
 *                            toward the lower id)
 *   mask        uint8 [B][T] out: alignment mask m_t (Eq. 3, along the draft
 *                            chain): prod_{j=1}^{n-1} mbar_prev[j-1][b][t-n+j],
 *                            0 for t < n-1, 1 everywhere when n == 1
 *   ell         fp32 [B][T]  out: lam_tok * (logsumexp(Xd_t) - Xd_t[x_t])
 *                            + lam_feat * ||Fd_t - Ft_t||_1
 *   seq_loss    fp32 [B]     out: sum_t m_t ell_t / sum_t m_t (Eq. 5), 0 when
 *                            no position is aligned; NaN when a token of the
 *                            sequence is outside [0, V) (its ell is NaN)
 * The paper's defaults are k = 3, lam_tok = 1, lam_feat = 0.1.  1 <= k <= V,
 * n >= 1, T >= 1, V >= 1, H >= 0.  Output buffers must not overlap the inputs.
 */
int gv_tat_loss(const void* logits, int logits_dt, const int32_t* tokens, const void* feat_draft,
                const void* feat_target, int feat_dt, int B, int T, int V, int H, int k, int n,
                const uint8_t* mbar_prev, float lambda_tok, float lambda_feat, uint8_t* mbar,
                uint8_t* mask, float* ell, float* seq_loss, void* stream);

/*
 * gv_tgf -- the draft model's Token-Guided Fusion (Section 4.2, Eqs. 6-8) of
 * rows of features F with the embeddings x of their tokens:
 *
 *   h = [F ; x] Wm^T + bm                     embedding fusion (Eq. 6)
 *   z = [LN_h(h) ; LN_x(x)] Wu^T + bu         normalisation and expansion (Eq. 7)
 *   o = silu(z) Wd^T + bd + h                 refinement (Eq. 8)
 *
 * LN_v(v) = (v - mean(v)) / sqrt(var(v) + eps) * g_v + b_v per row
 * (population variance); [a ; b] is the concatenation along the row.
 *
 *   F, x      bf16 [rows][d]    1 <= rows <= 256; d a multiple of 64, <= 8192
 *   Wm        bf16 [d][2d]      (output rows; columns: F's d, then x's d)
 *   bm, g_h, b_h, g_x, b_x      bf16 [d]
 *   Wu        bf16 [e][2d]      e the expansion width (a multiple of 8;
 *                               4d in Section 4.2, 11008 for LLaMA-2-7B)
 *   bu        bf16 [e]
 *   Wd        bf16 [d][e];  bd bf16 [d]
 *   h_out     bf16 [rows][d]    out: h (rounded to bf16; the residual of Eq. 8
 *                               and the layer norm take this rounded h)
 *   o_out     bf16 [rows][d]    out: o
 *   workspace >= gv_tgf_workspace(rows, d, e) bytes
 * fp32 accumulation and normalisation; z and silu(z) are rounded to bf16
 * between the projections.  16-byte aligned pointers; outputs must not
 * overlap the inputs or each other.  Six kernel launches, graph-capturable.
 */
size_t gv_tgf_workspace(int rows, int d, int e);
int gv_tgf(const void* F, const void* x, int rows, int d, int e, const void* Wm, const void* bm, const void* g_h,
           const void* b_h, const void* g_x, const void* b_x, const void* Wu, const void* bu, const void* Wd,
           const void* bd, float eps, void* h_out, void* o_out, void* workspace, size_t ws_bytes, void* stream);

/*
 * gv_draft_tree_expand / gv_draft_tree_finish -- the dynamic draft tree of one
 * cycle (60 nodes, depth 6 in the Implementation Details appendix; built the
 * EAGLE-2 way from the top-k lists of Section 4.1's draft passes).  Per
 * sequence b, a pool of nodes (token, parent, score) lives in the workspace:
 *
 *   step 0:       the pool is reset to the root (root_token[b], score 0); the
 *                 root's k most probable tokens join it
 *   step j >= 1:  each of the k nodes selected after step j-1 (slot s = the
 *                 s-th best) proposes its k most probable tokens
 *
 * A candidate's score is its parent's score + log softmax(logits row)[token];
 * the k best candidates of step j (larger score first, then the earlier
 * pool position) are expanded at step j+1.  Within a row, tokens rank by
 * larger logit, then lower id.  finish keeps the root and the N-1 best pool
 * nodes (same order), numbered in pool order (parents before children).
 *
 *   logits      [B][rows][V]  draft logits (dt GV_F32 or GV_BF16); rows = 1
 *                             at step 0, k after (row s = slot s); finite
 *   root_token  int32 [B]     step 0 only (else may be NULL)
 *   exp_token   int32 [B][k]  out, may be NULL: the tokens of the nodes to
 *                             expand at the next step, best first (the
 *                             drafter's next inputs; not written at step D-1)
 *   exp_pool    int32 [B][k]  out, may be NULL: their pool positions (the
 *                             root is 0; step j's candidates follow the
 *                             earlier ones, slot-major)
 *   parents     int32 [B][N]  out (finish): -1 for the root, else an index < i
 *   tokens      int32 [B][N]  out (finish): token[0] = the root token
 *   workspace   >= gv_draft_tree_workspace(B, k, D, V) bytes, the same buffer
 *               for every step of a tree; steps run in order 0 .. D-1, then
 *               finish.
 * 1 <= k <= 16, 1 <= D <= 16, k <= V <= 262144, 1 + k + (D-1) k^2 <= 4096 pool nodes,
 * 1 <= N <= min(64, pool nodes).  Scores are fp32.
 */
size_t gv_draft_tree_workspace(int B, int k, int D, int V);
int gv_draft_tree_expand(int B, int k, int D, int V, int step, int dt, const int32_t* root_token,
                         const void* logits, int32_t* exp_token, int32_t* exp_pool, void* workspace,
                         size_t ws_bytes, void* stream);
int gv_draft_tree_finish(int B, int k, int D, int V, int N, int32_t* parents, int32_t* tokens, void* workspace,
                         size_t ws_bytes, void* stream);

/*
 * gv_rmsnorm -- out[r] = x[r] / sqrt(mean(x[r]^2) + eps) * w (the target
 * layer's input and post-attention norms, and the final norm before the LM
 * head).  bf16 x, w, out [rows][H] / [H]; fp32 arithmetic; H % 8 == 0,
 * 16-byte aligned pointers; out may equal x.
 */
int gv_rmsnorm(const void* x, const void* w, int rows, int H, float eps, void* out, void* stream);

/*
 * gv_linear -- a projection of the node rows, out = epilogue(x W^T): the
 * Q/K/V, O, gate/up and down projections of the target layer.  The weight is
 * streamed once from HBM (tensor cores, K split across CTAs when the output is
 * narrow); fp32 accumulation; bf16 in and out.
 *
 *   x         bf16 [rows][K]           node rows, 1 <= rows <= 256
 *   W         bf16 [N][K]              N = n_out, or 2 * n_out for
 *                                      GV_LINEAR_SWIGLU (gate rows, then up rows)
 *   residual  bf16 [rows][n_out]       GV_LINEAR_ADD only (else NULL); out may be
 *                                      the same buffer
 *   out       bf16 [rows][n_out]; GV_LINEAR_SILU gives silu(x W^T)
 *   workspace >= gv_linear_workspace(rows, K, n_out, epilogue) bytes
 * K % 8 == 0, n_out % 8 == 0, 16-byte aligned pointers.  A bounded wait that
 * gives up turns the affected outputs into NaN.
 */
size_t gv_linear_workspace(int rows, int K, int n_out, int epilogue);
int gv_linear(const void* x, const void* W, int rows, int K, int n_out, int epilogue,
              const void* residual, void* out, void* workspace, size_t ws_bytes, void* stream);

/*
 * gv_linear_qkv -- the Q, K and V projections as one weight stream:
 * Wqkv = [Wq ; Wk ; Wv] bf16 [n_q + 2 n_kv][K]; q [rows][n_q], k and v
 * [rows][n_kv] (bf16, separate buffers, e.g. the gv_verify_attention inputs
 * q [B][N][Hq][d], k_new / v_new [B][N][Hkv][d]).  Conditions and workspace
 * as gv_linear's.
 */
size_t gv_linear_qkv_workspace(int rows, int K, int n_q, int n_kv);
int gv_linear_qkv(const void* x, const void* Wqkv, int rows, int K, int n_q, int n_kv, void* q, void* k, void* v,
                  void* workspace, size_t ws_bytes, void* stream);

/*
 * gv_linear_add_rmsnorm -- the residual projection fused with the RMSNorm
 * that follows it in the layer: out = residual + x W^T (out may be residual)
 * and norm_out = RMSNorm(out) * norm_w, computed from the stored bf16 out
 * (eps as gv_rmsnorm's).  n_out <= 8192; other conditions and the workspace
 * as gv_linear's with GV_LINEAR_ADD; norm_out is a separate buffer.
 */
int gv_linear_add_rmsnorm(const void* x, const void* W, int rows, int K, int n_out, const void* residual,
                          void* out, const void* norm_w, float eps, void* norm_out, void* workspace, size_t ws_bytes,
                          void* stream);

/* Static name of a status code. */
const char* gv_status_string(int status);

/* Detail of the last error returned on the calling host thread ("" if none). */
const char* gv_last_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int gv_version(void);

#ifdef __cplusplus
}
#endif

#endif /* GV_H */
