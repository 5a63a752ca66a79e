// gv_verify_attention_layers: the tree attention of L layers of one verify
// step in one persistent launch (bf16, d = 128, G * N <= 256).
//
// GRIFFIN Section 3: the target model verifies every draft token of the tree
// in one forward pass; in each attention layer node i attends to the cached
// prefix and to the nodes on its own root chain (Section 4.1: a rejected
// token drops its subtree, so the ancestor set is what node i may see).  The
// arithmetic per (layer, node, head) is that of gv_verify_attention.
//
// Work decomposition.  A unit is (layer l, sequence b, KV head g): its G * N
// query rows (row r = i * G + hl holds node i and query head g * G + hl; one
// or two 128-row M tiles, T) against its keys, cut into 128-key blocks.
// Block 0 of a unit holds the N tree keys (masked per query row by its
// ancestor bitmask), blocks 1 .. ceil(P_b / 128) the cached prefix.  The
// blocks of all units, in (l, b, g, block) order, each unit's blocks between
// AL_DSTART and AL_DEND positions without a block (the weights of a unit's
// start and end: pipeline restarts and epilogues for the CTAs that hold
// them), form one sequence of W
// positions that is cut into gridDim.x contiguous ranges of equal length
// (stream-K): CTA c takes the blocks at positions [c W / C, (c + 1) W / C).
// A unit inside one range is a whole piece, whose rows go straight to the
// output.  A unit cut by range ends has pieces in consecutive CTAs; a piece
// either combines with the unit's other piece if that one has arrived, or
// writes its normalised partial rows and their log2-sum-exp to a slot of the
// workspace (slot 2c for the first piece of CTA c, 2c + 1 for its last) and
// counts itself in the unit's arrival counter; the last of three or more
// pieces combines them all into the output.  No CTA waits for another.
//
// Both tiles of a unit share each staged K/V block (GQA: the G heads of a KV
// head read one K/V stream): per block, S_t = Q_t K^T and O_t += P_t V for
// t < T, so every K/V row is read once.  With one tile the two softmax
// streams take alternate halves of the blocks, each with its own O, and a
// piece's rows combine the two.  The K and V rings, the queries and
// the MMAs run ahead across piece boundaries: the next piece's blocks stream
// in while the current one finishes, its queries land once the last S of the
// current piece has read the old ones, and its first S is computed while the
// softmax warps write the current piece's rows.
//
// Warp roles: warp 0 issues TMA (lane 0 the K halves of every block, lane 1
// the V halves, lane 2 the queries of every piece); warp 1 owns TMEM and
// issues the MMAs from a polling loop (S first, then O += P V, whichever is
// ready); warps 4..7 and 8..11 are the two softmax streams (one thread per
// query row) and write the rows.  A job is 64 keys (one half of a block) of
// one tile: job k = (block, half, tile) in that order belongs to stream k & 1,
// and halves without keys (the tree block's second, the second of a last
// prefix block of <= 64 keys) are skipped.  TMEM: four S buffers of 64
// columns, job k in buffer k & 3 (so each stream computes its next S while
// its softmax runs; P overwrites the buffer's first half as bf16 pairs and
// feeds the PV MMA from TMEM), the O accumulator of stream s at columns
// 256 + 128 s.
//
// The queries and the tree keys arrive rotated (tree_prep_kernel, launched
// right before by the same call, rotates the queries into the workspace and
// writes the rotated tree keys and the values to the tree K/V scratch, the
// rows gv_kv_compact reads).  Every mbarrier wait is bounded; a CTA that gives
// up writes NaN for the rows of every piece it has not finished.
#include "gv_internal.cuh"
#include "attention.cuh"
#include "attn_common.cuh"
#include "sm103.cuh"

namespace gv {
using namespace sm103;

namespace {

constexpr int AL_BK = 128;                 // keys per block
constexpr int AL_HALF = 128 * 128;         // 128 rows x 64 d bf16 (one 128B-swizzled column block)
constexpr int AL_TILE = 2 * AL_HALF;       // 128 rows x 128 d
constexpr int AL_KST = 3;                  // K ring stages (32 KB each)
constexpr int AL_VST = 2;                  // V ring stages
constexpr int AL_NSM = 256;                // softmax threads (warps 4..11)
constexpr int AL_SM0 = 128;                // first softmax thread
constexpr int AL_NTH = AL_SM0 + AL_NSM;
// Registers per thread: launched with 168 (the most 384 threads get), then
// warpgroup 0 (TMA, MMA, two idle warps) gives 64 back and the two softmax
// warpgroups take 32 more each: 128 * 104 + 256 * 200 = 384 * 168.
constexpr int AL_REG_LOW = 104, AL_REG_HIGH = 200;
static_assert(128 * AL_REG_LOW + 256 * AL_REG_HIGH <= 384 * 168, "register split");
constexpr uint32_t AL_OCOL = 256;          // O of tile t at columns 256 + 128 t
constexpr uint32_t AL_TMEM_COLS = 512;
constexpr int AL_MAXB = 64;                // sequences per call
constexpr int AL_DSTART = 3;               // positions without a block before each unit's blocks (see Walk)
constexpr int AL_DEND = 0;                 // ... and after them

// Shared memory: Q tiles | K ring | V ring | barriers | misc | the two
// streams' row maxima and sums | blocks per unit and prefix length of each
// sequence.
constexpr int AL_OFF_K = 2 * AL_TILE;
constexpr int AL_OFF_V = AL_OFF_K + AL_KST * AL_TILE;
constexpr int AL_OFF_BAR = AL_OFF_V + AL_VST * AL_TILE;
constexpr int AL_NBAR = 3 * AL_KST + 3 * AL_VST + 12 + 5;
constexpr int AL_OFF_MISC = AL_OFF_BAR + 8 * AL_NBAR;
constexpr int AL_OFF_ML = AL_OFF_MISC + 32;            // float2 (m, l) [2 streams][128 rows]
constexpr int AL_OFF_NB = AL_OFF_ML + 2 * 128 * 8;     // int [AL_MAXB]
constexpr int AL_OFF_P = AL_OFF_NB + 4 * AL_MAXB;      // int [AL_MAXB] prefix lengths
constexpr int AL_SMEM = AL_OFF_P + 4 * AL_MAXB;
static_assert(AL_SMEM <= 232448, "shared memory of the multi-layer attention kernel");

}  // namespace

struct AttnLayersArgs {
    int L, B, N, Hq, Hkv, G, T, S_max;
    int boxn;                        // nodes per Q box: min(128 / G, N)
    float scale;                     // 1 / sqrt(d)
    const int32_t* prefix_len;
    const unsigned long long* anc;
    __nv_bfloat16* out;              // [L][B][N][Hq][128]
    __nv_bfloat16* part;             // [2 C][T][128][128] normalised partial rows
    float* part_lse;                 // [2 C][T][128]
    int* cnt;                        // [L][B][Hkv] arrival counters (zero between calls)
};

namespace {

// One piece: blocks [j0, j1) of unit (l, b, g), in the CTA's range.
struct Piece {
    int l, b, g, j0, j1, nb, unit;
    long long u0;    // the unit's first position in the (weighted) sequence
    bool direct;     // the whole unit
    int slot;        // partial slot (split pieces)
};

// Walks the pieces of the range [w, w_end) of CTA c.  Positions: a unit of
// sequence b spans AL_DSTART + nb[b] + AL_DEND positions: AL_DSTART without a
// block, its blocks, AL_DEND without a block (a unit's start and end cost
// the CTAs that hold them a pipeline restart and an epilogue; weighting them
// evens the CTAs' times).
struct Walk {
    long long w, w_end, w_begin, Wl;
    int B, Hkv, c;
    const int* nb;   // blocks per unit of sequence b
    __device__ __forceinline__ bool next(Piece& p) {
        while (w < w_end) {
            const long long l = w / Wl;
            long long r = w - l * Wl;
            int b = 0;
            while (b < B - 1 && r >= (long long)Hkv * (nb[b] + AL_DSTART + AL_DEND)) {
                r -= (long long)Hkv * (nb[b] + AL_DSTART + AL_DEND);
                ++b;
            }
            const int n = nb[b], vn = AL_DSTART + n + AL_DEND;
            const int g = (int)(r / vn);
            const int j0 = (int)(r - (long long)g * vn) - AL_DSTART;
            if (j0 < 0) {                  // (before the unit's blocks)
                w -= j0;
                continue;
            }
            if (j0 >= n) {                 // (past the unit's blocks)
                w += n + AL_DEND - j0;
                continue;
            }
            const long long len = min((long long)(n - j0), w_end - w);
            p.l = (int)l;
            p.b = b;
            p.g = g;
            p.j0 = j0;
            p.j1 = j0 + (int)len;
            p.nb = n;
            p.unit = ((int)l * B + b) * Hkv + g;
            p.u0 = w - j0;
            p.direct = j0 == 0 && len == n;
            // (the CTA's first piece when its unit starts at or before the
            // range, the rule the combining CTA applies to find the slot)
            p.slot = 2 * c + (p.u0 <= w_begin ? 0 : 1);
            w += len;
            return true;
        }
        return false;
    }
};

// Halves (64 keys each) of block j that hold keys: the tree block's N <= 64
// keys and a last prefix block of at most 64 keys are one half, every other
// block two.
__device__ __forceinline__ int halves_of(int j, int P) {
    return (j == 0 || P - AL_BK * (j - 1) <= AL_BK / 2) ? 1 : 2;
}

// The blocks of a CTA in order and, in each, the jobs of one stream: with two
// tiles stream s has the block's halves of tile s, with one tile it has half
// s of a block that has it.  m counts the stream's jobs (mp: at the piece's
// start); piece_ok / stage_ok record the waits the issuer passed for the
// current piece and block.
struct Cursor {
    Walk wk;
    Piece pc;
    const int* sP;   // prefix length of each sequence
    bool valid, piece_ok, stage_ok;
    int T, s, P, jp, nh, nj, jh, pidx, gb, m, mp;
    __device__ __forceinline__ void set_block() {
        nh = halves_of(pc.j0 + jp, P);
        nj = T == 2 ? nh : (s < nh ? 1 : 0);
    }
    __device__ __forceinline__ void start(const Walk& w, const int* sp, int T_, int s_) {
        wk = w;
        sP = sp;
        T = T_;
        s = s_;
        jp = jh = pidx = gb = m = mp = 0;
        piece_ok = stage_ok = false;
        valid = wk.next(pc);
        if (valid) {
            P = sP[pc.b];
            set_block();
        }
    }
    __device__ __forceinline__ int half() const { return T == 2 ? jh : s; }
    __device__ __forceinline__ bool last_block() const { return jp == pc.j1 - pc.j0 - 1; }
    __device__ __forceinline__ void next_block() {
        jh = 0;
        stage_ok = false;
        ++gb;
        if (++jp < pc.j1 - pc.j0) {
            set_block();
            return;
        }
        jp = 0;
        ++pidx;
        mp = m;
        piece_ok = false;
        valid = wk.next(pc);
        if (valid) {
            P = sP[pc.b];
            set_block();
        }
    }
};

// CTA whose range holds block w: the largest c with floor(c W / C) <= w.
__device__ __forceinline__ int cta_of(long long w, long long W, int C) {
    return (int)(((w + 1) * C - 1) / W);
}

// The tile count of a unit as a type (the piece epilogue is compiled per count).
template <int V>
struct AlTiles {
    static constexpr int value = V;
};

// 32-byte store of 8 words (sm_100+).
__device__ __forceinline__ void st_global_v8(void* p, const uint32_t (&r)[8]) {
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(r[0]), "r"(r[1]),
                 "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
                 : "memory");
}

}  // namespace

// The last piece of a unit to arrive combines the unit's pieces: for every
// query row, o = sum_p 2^(lse_p - M) o_p / sum_p 2^(lse_p - M) over the pieces'
// normalised partial rows o_p and log2-sum-exps lse_p (M their maximum),
// online over the pieces.  Thread (row, 16-byte chunk), chunks fastest, so a
// warp reads and writes two whole rows; four items per thread are in flight.
__device__ __forceinline__ void merge_unit(const AttnLayersArgs& a, const Piece& pc, long long U0, int cf, int cl,
                                           long long W, int C, int t_id) {
    const int nitems = a.G * a.N * 16;
    for (int e0 = t_id; e0 < nitems; e0 += 4 * AL_NSM) {
        float M[4], wsum[4], acc[4][8];
        bool bad[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            M[q] = -INFINITY;
            wsum[q] = 0.f;
            bad[q] = false;
#pragma unroll
            for (int u = 0; u < 8; ++u) acc[q][u] = 0.f;
        }
        for (int cc = cf; cc <= cl; ++cc) {
            const long long sc = (long long)cc * W / C;
            if (sc == (long long)(cc + 1) * W / C) continue;        // (an empty range holds no piece)
            const int slot = 2 * cc + (U0 <= sc ? 0 : 1);
            float ls[4];
            uint4 v[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int e = e0 + q * AL_NSM;
                ls[q] = -INFINITY;
                v[q] = make_uint4(0, 0, 0, 0);
                if (e < nitems) {
                    const int qr = e >> 4, ch = e & 15;
                    const size_t prow = ((size_t)slot * a.T + (qr >> 7)) * 128 + (qr & 127);
                    ls[q] = __ldcg(a.part_lse + prow);
                    v[q] = __ldcg(reinterpret_cast<const uint4*>(a.part + prow * 128) + ch);
                }
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                bad[q] |= ls[q] != ls[q];
                const float m_new = fmaxf(M[q], ls[q]);
                const float sa = M[q] == -INFINITY ? 0.f : fast_exp2(M[q] - m_new);
                const float wq = ls[q] == -INFINITY ? 0.f : fast_exp2(ls[q] - m_new);
                M[q] = m_new;
                wsum[q] = wsum[q] * sa + wq;
                const uint32_t u4[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
#pragma unroll
                for (int h2 = 0; h2 < 4; ++h2) {
                    const float2 f = unpack_bf16(u4[h2]);
                    acc[q][2 * h2] = fmaf(wq, f.x, acc[q][2 * h2] * sa);
                    acc[q][2 * h2 + 1] = fmaf(wq, f.y, acc[q][2 * h2 + 1] * sa);
                }
            }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int e = e0 + q * AL_NSM;
            if (e >= nitems) continue;
            const int qr = e >> 4, ch = e & 15;
            const float inv = bad[q] ? NAN : 1.0f / wsum[q];
            const int i = qr / a.G, h = pc.g * a.G + qr % a.G;
            uint4* o = reinterpret_cast<uint4*>(a.out + ((((size_t)pc.l * a.B + pc.b) * a.N + i) * a.Hq + h) * 128);
            o[ch] = make_uint4(pack_bf16(acc[q][0] * inv, acc[q][1] * inv), pack_bf16(acc[q][2] * inv, acc[q][3] * inv),
                               pack_bf16(acc[q][4] * inv, acc[q][5] * inv), pack_bf16(acc[q][6] * inv, acc[q][7] * inv));
        }
    }
}

__global__ void __launch_bounds__(AL_NTH, 1)
attn_layers_kernel(const __grid_constant__ CUtensorMap map_ck, const __grid_constant__ CUtensorMap map_cv,
                   const __grid_constant__ CUtensorMap map_tk, const __grid_constant__ CUtensorMap map_tv,
                   const __grid_constant__ CUtensorMap map_q, AttnLayersArgs a) {
    extern __shared__ __align__(1024) uint8_t smem[];
    uint8_t* sQ = smem;
    uint8_t* sK = smem + AL_OFF_K;
    uint8_t* sV = smem + AL_OFF_V;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + AL_OFF_BAR);
    uint64_t* k_full = bars;
    uint64_t* k_empty = k_full + AL_KST;     // [2 streams][AL_KST]
    uint64_t* v_full = k_empty + 2 * AL_KST;
    uint64_t* v_empty = v_full + AL_VST;     // [2 streams][AL_VST]
    // S buffer b = 2 s + (m & 1) holds job m of stream s
    uint64_t* s_full = v_empty + 2 * AL_VST; // [4]
    uint64_t* p_full = s_full + 4;           // [4]
    // [4] the PV of buffer b has completed (with every MMA its issuer issued
    // before it).  A parity wait on an mbarrier is unambiguous only while the
    // barrier is at most one phase behind.  A softmax thread waits for the PV
    // of its stream's job m only after it has seen S_m (or a later S of its
    // stream) complete, and S_m was issued after the PV of job m - 2 (the
    // buffer's previous phase) by the same thread: in-order MMAs, so that PV
    // is done.
    uint64_t* pv_done = p_full + 4;
    uint64_t* q_full = pv_done + 4;
    uint64_t* q_empty = q_full + 1;          // one arrival per stream
    uint64_t* o_free = q_empty + 1;
    uint64_t* drain = o_free + 1;            // [2] one per issuer
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(smem + AL_OFF_MISC);
    volatile int* abort = reinterpret_cast<volatile int*>(smem + AL_OFF_MISC + 4);
    volatile int* last_flag = reinterpret_cast<volatile int*>(smem + AL_OFF_MISC + 8);
    // [2] a split piece's decision to combine, published by thread 0 with the
    // piece-end vote (two words, alternating by piece: a word is rewritten
    // only after every thread has passed the next piece's vote)
    volatile int* cmb_flag = reinterpret_cast<volatile int*>(smem + AL_OFF_MISC + 12);
    int* snb = reinterpret_cast<int*>(smem + AL_OFF_NB);
    int* sP = reinterpret_cast<int*>(smem + AL_OFF_P);

    const int T = a.T, N = a.N, G = a.G;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < AL_KST; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
            mbar_init(&k_empty[AL_KST + s], 1);
        }
        for (int s = 0; s < AL_VST; ++s) {
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], 1);
            mbar_init(&v_empty[AL_VST + s], 1);
        }
        for (int c = 0; c < 4; ++c) {
            mbar_init(&s_full[c], 1);
            mbar_init(&p_full[c], AL_NSM / 64);     // the four warps of one stream
            mbar_init(&pv_done[c], 1);
        }
        mbar_init(q_full, 1);
        mbar_init(q_empty, 2);
        mbar_init(o_free, AL_NSM / 32);
        mbar_init(&drain[0], 1);
        mbar_init(&drain[1], 1);
        // (the 128B-swizzled tiles need a 1024-byte aligned base)
        *abort = (smem_u32(smem) & 1023u) != 0 ? 1 : 0;
        *last_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&map_ck);
        prefetch_tmap(&map_cv);
        prefetch_tmap(&map_tk);
        prefetch_tmap(&map_tv);
        prefetch_tmap(&map_q);
    }
    // Blocks per unit of every sequence: the tree block and the prefix blocks.
    // prefix_len is a step input no kernel of the step writes, so it may be
    // read before griddepcontrol.wait.
    if (threadIdx.x < a.B) {
        const int P = min(max(a.prefix_len[threadIdx.x], 0), a.S_max);
        snb[threadIdx.x] = 1 + (P + AL_BK - 1) / AL_BK;
        sP[threadIdx.x] = P;
    }
    if (warp == 1) tmem_alloc(tmem_holder, AL_TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    pdl_trigger();

    // This CTA's block range.
    long long Wl = 0;
    for (int b = 0; b < a.B; ++b) Wl += snb[b] + AL_DSTART + AL_DEND;
    Wl *= a.Hkv;
    const long long W = Wl * a.L;
    const int C = gridDim.x, c = blockIdx.x;
    const long long w_begin = (long long)c * W / C, w_end = (long long)(c + 1) * W / C;
    Walk walk0;
    walk0.w = w_begin;
    walk0.w_end = w_end;
    walk0.w_begin = w_begin;
    walk0.Wl = Wl;
    walk0.B = a.B;
    walk0.Hkv = a.Hkv;
    walk0.c = c;
    walk0.nb = snb;

    // (each register split sits in the branch whose code runs under it)
    if (warp < 4) {
      asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(AL_REG_LOW));
      if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane < 2) {
            // Lane 0 streams the K halves of every block, lane 1 the V halves,
            // each as soon as its ring stage is free.  The prefix blocks of the
            // first fill stream before griddepcontrol.wait (the cache is not
            // written by the kernels this one follows); the tree block reads
            // the scratch the preceding kernel wrote, after it.
            const bool isk = lane == 0;
            const int NS = isk ? AL_KST : AL_VST;
            uint64_t* full = isk ? k_full : v_full;
            uint64_t* empty = isk ? k_empty : v_empty;
            uint8_t* ring = isk ? sK : sV;
            const CUtensorMap* mc = isk ? &map_ck : &map_cv;
            const CUtensorMap* mt = isk ? &map_tk : &map_tv;
            const uint64_t pol = policy_evict_first();
            Walk wk = walk0;
            Piece pc;
            int gb = 0, last = -1;
            bool waited = false, go = *abort == 0;
            while (go && wk.next(pc)) {
                for (int j = pc.j0; j < pc.j1; ++j, ++gb) {
                    const int s = gb % NS;
                    const uint32_t ph = (uint32_t)(gb / NS) & 1u;
                    if (!waited && (j == 0 || gb >= NS)) {
                        pdl_wait();
                        waited = true;
                    }
                    // (each stream's issuer releases the stage once it is done with the block)
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort) || !mbar_wait(&empty[NS + s], ph ^ 1u, abort)) {
                        go = false;
                        break;
                    }
                    uint8_t* st = ring + s * AL_TILE;
                    if (j == 0) {
                        mbar_arrive_expect_tx(&full[s], (uint32_t)(2 * N * 128));
                        const int y = pc.unit * N;
                        tma_load_2d(st, mt, &full[s], 0, y, pol);
                        tma_load_2d(st + AL_HALF, mt, &full[s], 64, y, pol);
                    } else {
                        mbar_arrive_expect_tx(&full[s], (uint32_t)(2 * AL_HALF));
                        const int y = (pc.b * a.Hkv + pc.g) * a.S_max + (j - 1) * AL_BK;
                        tma_load_3d(st, mc, &full[s], 0, y, pc.l, pol);
                        tma_load_3d(st + AL_HALF, mc, &full[s], 64, y, pc.l, pol);
                    }
                    last = gb;
                }
            }
            if (*abort && last >= 0) {
                // Drain: the newest load of every stage lands before the CTA exits.
                for (int s = 0; s < NS; ++s) {
                    if (last < s) continue;
                    const int gs = last - ((last - s) % NS);
                    mbar_wait_timeout_only(&full[s], (uint32_t)(gs / NS) & 1u);
                }
            }
        } else if (lane == 2) {
            // The queries of every piece (both tiles), once the last S of the
            // previous piece has read the old ones.  4-D map over the rotated
            // queries [L * B][N][Hq][128]: box {64 d, G heads, boxn nodes}, so a
            // tile lands as node-major, head-minor rows; nodes past N read 0.
            const uint64_t pol = policy_evict_first();
            pdl_wait();
            Walk wk = walk0;
            Piece pc;
            int pidx = 0;
            const uint32_t bytes = (uint32_t)(T * 2 * 64 * G * a.boxn * 2);
            while (*abort == 0 && wk.next(pc)) {
                if (pidx > 0 && !mbar_wait(q_empty, (uint32_t)(pidx - 1) & 1u, abort)) break;
                mbar_arrive_expect_tx(q_full, bytes);
                const int z4 = pc.l * a.B + pc.b;
                for (int t = 0; t < T; ++t) {
                    const int n0 = t * (128 / G);
                    tma_load_4d(sQ + t * AL_TILE, &map_q, q_full, 0, pc.g * G, n0, z4, pol);
                    tma_load_4d(sQ + t * AL_TILE + AL_HALF, &map_q, q_full, 64, pc.g * G, n0, z4, pol);
                }
                ++pidx;
            }
            if (*abort && pidx > 0) mbar_wait_timeout_only(q_full, (uint32_t)(pidx - 1) & 1u);
        }
    } else if (warp == 1 || warp == 2) {
        // ------------------------------------------------- MMA issuers (one per stream)
        // One thread issues a stream's MMAs (a single thread reaches about half
        // the tensor pipe's rate with these 128-row shapes, two reach it); the
        // whole warp walks the jobs, so that its other lanes can zero V rows.
        const int st = warp - 1;                             // stream
        const uint32_t idesc_s = idesc_bf16(128, AL_BK / 2);
        const uint32_t idesc_o = idesc_bf16(128, 128, /*b_mn_major=*/true);
        const uint32_t ocol = tmem + AL_OCOL + 128u * (uint32_t)st;
        const uint32_t qbase = smem_u32(sQ + (T == 2 ? st : 0) * AL_TILE);
        uint64_t* kemp = k_empty + st * AL_KST;
        uint64_t* vemp = v_empty + st * AL_VST;
        // (lane 0's view of a barrier, the same for the whole warp)
        auto wtest = [&](uint64_t* bar, uint32_t parity) -> bool {
            return __shfl_sync(FULL, mbar_test_wait(bar, parity) ? 1 : 0, 0) != 0;
        };
        Cursor cs, cp;
        cs.start(walk0, sP, T, st);
        cp.start(walk0, sP, T, st);
        bool mok = *abort == 0;
        bool o_ok = false;                                  // o_free passed for cp's piece
        unsigned long long t_last = globaltimer();
        while (mok && (cs.valid || cp.valid)) {
            bool prog = false;
            // S of the stream's job m = Q K_{half}^T (64 keys) into buffer
            // 2 st + (m & 1), once the piece's queries and the block's K have
            // landed and the PV of job m - 2 (the last reader of that buffer's
            // P) has been issued: a thread's MMAs run in issue order.  After its
            // jobs of a block the stream releases the block's K stage (and, at a
            // piece's end, the queries); a block without a job of this stream is
            // waited for and released all the same, so that every barrier
            // advances one phase per block.
            if (cs.valid) {
                bool go = true;
                if (!cs.piece_ok) go = cs.piece_ok = wtest(q_full, (uint32_t)cs.pidx & 1u);
                const int ks = cs.gb % AL_KST;
                if (go && !cs.stage_ok) go = cs.stage_ok = wtest(&k_full[ks], (uint32_t)(cs.gb / AL_KST) & 1u);
                if (go && cs.jh < cs.nj && cs.m - cp.m < 2) {
                    const int buf = 2 * st + (cs.m & 1);
                    if (lane == 0) {
                        tc_fence_after();
                        // keys 64 hh .. of the stage: 64 rows of 128 B = 8 swizzle atoms on
                        const uint32_t kbase = smem_u32(sK + ks * AL_TILE) + (uint32_t)cs.half() * (64u * 128u);
#pragma unroll
                        for (int kb = 0; kb < 2; ++kb) {
                            const uint64_t qdesc = sdesc_kmajor_sw128(qbase + kb * AL_HALF);
                            const uint64_t kdesc = sdesc_kmajor_sw128(kbase + kb * AL_HALF);
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                mma_bf16(tmem + (uint32_t)(buf * 64), qdesc + 2u * kk, kdesc + 2u * kk, idesc_s,
                                         (kb | kk) != 0);
                        }
                        mma_commit(&s_full[buf]);
                    }
                    ++cs.m;
                    ++cs.jh;
                    prog = true;
                }
                if (go && cs.jh == cs.nj) {
                    if (lane == 0) {
                        mma_commit(&kemp[ks]);
                        if (cs.last_block()) mma_commit(q_empty);
                    }
                    cs.next_block();
                    prog = true;
                }
            }
            // O_st += P V_{half} once the softmax has written P of job m and the
            // block's V has landed.  The stream's first PV of a piece overwrites
            // O_st, after the softmax warps have read the previous piece's O
            // (o_free; tested only by a stream that has a PV in the piece, the
            // one that can hold the barrier back).  V rows past the valid keys
            // of a block's last half (past the prefix end, or past the N tree
            // rows the copy wrote) may hold anything, and P = 0 times a NaN would
            // still be NaN: the warp zeroes them before the PV that reads them
            // (with two tiles both streams do, each before its own PV).
            if (cp.valid) {
                bool go = true;
                const int vs = cp.gb % AL_VST;
                if (!cp.stage_ok) {
                    go = cp.stage_ok = wtest(&v_full[vs], (uint32_t)(cp.gb / AL_VST) & 1u);
                    const int j = cp.pc.j0 + cp.jp;
                    const int nvalid = j == 0 ? N : min(AL_BK, cp.P - (j - 1) * AL_BK);
                    if (go && nvalid < 64 * cp.nh && (T == 2 || st == cp.nh - 1)) {
                        uint8_t* vt = sV + vs * AL_TILE;
                        for (int e = lane; e < (64 * cp.nh - nvalid) * 16; e += 32) {
                            const int key = nvalid + (e >> 4), ch = e & 15;
                            *reinterpret_cast<uint4*>(vt + (ch >> 3) * AL_HALF + sw128(key, ch & 7)) =
                                make_uint4(0, 0, 0, 0);
                        }
                        __syncwarp();
                        if (lane == 0) fence_proxy_async_smem();   // the zeros, for the MMA
                    }
                }
                if (go && cp.jh < cp.nj) {
                    const int buf = 2 * st + (cp.m & 1);
                    const bool fresh = cp.m == cp.mp;
                    if (fresh && !o_ok) o_ok = cp.pidx == 0 || wtest(o_free, (uint32_t)(cp.pidx - 1) & 1u);
                    if ((!fresh || o_ok) && cp.m < cs.m && wtest(&p_full[buf], (uint32_t)(cp.m >> 1) & 1u)) {
                        if (lane == 0) {
                            tc_fence_after();
                            // V as the MN-major B operand: rows = keys (128 B apart,
                            // SBO = 1 KB per 8 keys), the two 64-wide halves of d
                            // (LBO) one half-tile apart; a K step is 16 keys = 2 KB.
                            uint64_t vdesc = sdesc_kmajor_sw128(smem_u32(sV + vs * AL_TILE));
                            vdesc = (vdesc & ~(0x3FFFull << 16)) | ((uint64_t)(AL_HALF >> 4) << 16);
                            // P: 8 TMEM columns (bf16 pairs) per K step of 16 keys.
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                mma_bf16_ta(ocol, tmem + (uint32_t)(buf * 64 + 8 * kk),
                                            vdesc + (uint64_t)((4 * cp.half() + kk) * 128), idesc_o,
                                            !fresh || (kk != 0));
                            mma_commit(&pv_done[buf]);
                        }
                        ++cp.m;
                        ++cp.jh;
                        prog = true;
                    } else {
                        go = false;
                    }
                }
                if (go && cp.jh == cp.nj) {
                    if (lane == 0) mma_commit(&vemp[vs]);
                    const int pidx0 = cp.pidx;
                    cp.next_block();
                    if (cp.pidx != pidx0) o_ok = false;
                    prog = true;
                }
            }
            if (prog) {
                t_last = globaltimer();
            } else if (__shfl_sync(FULL, (*abort || globaltimer() - t_last > WAIT_TIMEOUT_NS) ? 1 : 0, 0)) {
                *abort = 1;
                mok = false;
            }
        }
        if (lane == 0) {
            mma_commit(&drain[st]);
            mbar_wait_timeout_only(&drain[st], 0);
        }
        __syncwarp();
      }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(AL_REG_HIGH));
        // ------------------------------------------- softmax, rows, merges
        // Two warp groups, one per stream: job k belongs to stream k & 1,
        // whose O accumulator is O_{k & 1}; its S arrives in buffer k & 3.
        // With two tiles a stream is a tile (both streams read every half
        // block); with one tile the streams take alternate halves of the same
        // rows, and the piece's rows combine both accumulators.  One thread
        // per query row holds the job's 64 scores, so the row max needs no
        // exchange, and the two groups hide each other's latencies.
        const int t_id = threadIdx.x - AL_SM0;
        const int s = (warp - 4) >> 2;                       // stream (warp group)
        const int sub = warp & 3;                            // TMEM lane quarter
        const int row = sub * 32 + lane;                     // row within the tile
        const int tile = T == 2 ? s : 0;
        const int qr = 128 * tile + row;                     // query row of the unit
        const bool rv = qr < G * N;
        const uint32_t lane_base = tmem + ((uint32_t)(sub * 32) << 16);
        const uint32_t ocol = lane_base + AL_OCOL + 128u * (uint32_t)s;  // this stream's O
        const float sl2 = a.scale * 1.4426950408889634f;    // scale * log2(e)
        float2* sML = reinterpret_cast<float2*>(smem + AL_OFF_ML);        // [2 streams][128 rows]
        // (one vote, so that every softmax thread starts from the same answer)
        bool ok = bar_and(1, AL_NSM, *abort == 0 ? 1 : 0);
        bool waited = false;
        Walk wk = walk0;
        Piece pc;
        int npc = 0;           // pieces so far
        int m0 = 0;            // this stream's jobs before the piece
        while (wk.next(pc)) {
            const int P = min(max(a.prefix_len[pc.b], 0), a.S_max);
            const int nbk = pc.j1 - pc.j0;
            float m_run = -INFINITY, l_run = 0.f;
            // (the ancestor masks were written two launches before this one)
            const unsigned long long anc_r = (rv && pc.j0 == 0) ? __ldg(a.anc + (size_t)pc.b * N + qr / G) : 0ull;
            // Walk this stream's jobs of the piece in the order its MMA issuer
            // does (with two tiles every half of a block, else half s of a
            // block that has it); m counts the stream's jobs.  A thread whose
            // wait failed stops working (no barrier inside the loop), and the
            // piece-wide vote below makes it every thread's answer.
            int m = m0, nmine = 0, nother = 0;
            for (int jp = 0; jp < nbk; ++jp) {
                const int j = pc.j0 + jp;
                const int nvalid = j == 0 ? N : min(AL_BK, P - (j - 1) * AL_BK);
                const int nh = halves_of(j, P);
                const int nj = T == 2 ? nh : (s < nh ? 1 : 0);
                nother += T == 2 ? nh : (1 - s < nh ? 1 : 0);
                {
                    for (int jh = 0; jh < nj; ++jh, ++m, ++nmine) {
                        if (!ok) continue;
                        const int hh = T == 2 ? jh : s;
                        const int buf = 2 * s + (m & 1);
                        const uint32_t scol = lane_base + (uint32_t)(buf * 64);
                        int w = 1;
                        if (lane == 0) w = mbar_wait(&s_full[buf], (uint32_t)(m >> 1) & 1u, abort);
                        if (!__shfl_sync(FULL, w, 0)) {
                            ok = false;
                            continue;
                        }
                        tc_fence_after();
                        uint32_t sv[64];
                        tmem_ld32(scol, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
                        tmem_ld32(scol + 32u, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
                        tmem_wait_ld();
#pragma unroll
                        for (int cc = 0; cc < 64; ++cc) asm volatile("" : "+r"(sv[cc]));   // uses stay after the wait
                        // Keys of this half this row may see: all of them (the
                        // common, unmasked path), else a branch-free mask (the
                        // row's ancestor bitmask on the tree block, whose keys
                        // are nodes 0..N-1 <= 63; the prefix end on the last
                        // block); masked scores become -inf, and their exp2 is 0.
                        const int nv = nvalid - 64 * hh;
                        if (j == 0 || nv < 64) {
                            const unsigned long long vbits = j == 0 ? anc_r : ((1ull << nv) - 1ull);
                            const uint32_t vlo = (uint32_t)vbits, vhi = (uint32_t)(vbits >> 32);
#pragma unroll
                            for (int cc = 0; cc < 64; ++cc)
                                sv[cc] = ((cc < 32 ? vlo >> cc : vhi >> (cc - 32)) & 1u) ? sv[cc]
                                                                                       : __float_as_uint(-INFINITY);
                        }
                        float mxs[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                        for (int cc = 0; cc < 64; cc += 2)
                            mxs[(cc >> 1) & 3] =
                                max3(mxs[(cc >> 1) & 3], __uint_as_float(sv[cc]), __uint_as_float(sv[cc + 1]));
                        const float mx = max3(mxs[0], mxs[1], fmaxf(mxs[2], mxs[3])) * sl2;   // sl2 > 0
                        const float m_new = fmaxf(m_run, mx);
                        const bool need = m_new > m_run + 8.0f;      // also true the first time
                        float alpha = 1.0f;
                        if (need) {
                            alpha = fast_exp2(m_run - m_new);         // 0 when m_run = -inf
                            m_run = m_new;
                        }
                        // p = 2^(s * sl2 - m); a row with no visible key so far
                        // keeps m = -inf and all its p are 0.  P as bf16 pairs over
                        // the first 32 of the buffer's 64 columns.
                        const float nmv = m_run == -INFINITY ? 0.f : -m_run;
                        const uint64_t sc2 = f32x2(sl2, sl2), nm2 = f32x2(nmv, nmv);
                        uint64_t ps[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
                        for (int c0 = 0; c0 < 32; c0 += 16) {
                            uint32_t pk[16];
#pragma unroll
                            for (int u = 0; u < 16; ++u) {
                                const int cc = c0 + u;
                                const float2 xa = split_f32x2(ffma_f32x2(
                                    f32x2(__uint_as_float(sv[2 * cc]), __uint_as_float(sv[2 * cc + 1])), sc2, nm2));
                                const float p0 = fast_exp2(xa.x), p1 = fast_exp2(xa.y);
                                ps[cc & 3] = fadd_f32x2(ps[cc & 3], f32x2(p0, p1));
                                pk[u] = pack_bf16(p0, p1);
                            }
                            tmem_st16(scol + (uint32_t)c0, pk);
                        }
                        const float2 psum =
                            split_f32x2(fadd_f32x2(fadd_f32x2(ps[0], ps[1]), fadd_f32x2(ps[2], ps[3])));
                        l_run = l_run * alpha + (psum.x + psum.y);
                        if (m > m0 && __any_sync(FULL, need)) {
                            // Rescale this row of O_s: this stream's previous PV
                            // must have landed first.
                            const int mq = m - 1;
                            if (lane == 0)
                                w = mbar_wait(&pv_done[2 * s + (mq & 1)], (uint32_t)(mq >> 1) & 1u, abort);
                            if (!__shfl_sync(FULL, w, 0)) {
                                ok = false;
                                continue;
                            }
                            tc_fence_after();
#pragma unroll
                            for (int c0 = 0; c0 < 128; c0 += 32) {
                                uint32_t ov[32];
                                tmem_ld32(ocol + c0, ov);
                                tmem_wait_ld();
                                uint32_t lo[16], hi[16];
#pragma unroll
                                for (int e = 0; e < 16; ++e) {
                                    lo[e] = __float_as_uint(__uint_as_float(ov[e]) * alpha);
                                    hi[e] = __float_as_uint(__uint_as_float(ov[16 + e]) * alpha);
                                }
                                tmem_st16(ocol + c0, lo);
                                tmem_st16(ocol + c0 + 16, hi);
                            }
                        }
                        tmem_wait_st();
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&p_full[buf]);
                    }
                }
            }
            // ------------------------------------------------- the piece's rows
            // The output and the workspace may still be read by the grid this
            // one follows (an earlier call's), and the arrival counters are
            // zeroed by the one right before: wait for it first.
            if (!waited) {
                pdl_wait();
                waited = true;
            }
            // A piece of a unit cut between CTAs: the unit's pieces are one in
            // every CTA of [cf, cl] whose range is not empty (ranges are empty
            // when there are fewer blocks than CTAs).  When the unit has two
            // pieces and the other one has already arrived (an acquiring read
            // of the unit's counter, taken by thread 0 while the last PV lands
            // and published with the vote), this piece combines the two
            // straight from its accumulators and the other's partial rows;
            // otherwise it writes its own partial rows and counts itself
            // (below).
            const long long U0 = pc.u0;
            int cf = 0, cl = -1, npieces = 0, other_slot = -1;
            if (!pc.direct) {
                cf = cta_of(U0, W, C);
                cl = cta_of(U0 + pc.nb - 1, W, C);
                for (int cc = cf; cc <= cl; ++cc) {
                    const long long sc = (long long)cc * W / C;
                    if (sc == (long long)(cc + 1) * W / C) continue;
                    ++npieces;
                    if (cc != c) other_slot = 2 * cc + (U0 <= sc ? 0 : 1);
                }
                if (t_id == 0) {
                    const bool ready = npieces == 2 && atomicAdd(a.cnt + pc.unit, 0) == 1;
                    __threadfence();
                    cmb_flag[npc & 1] = ready ? 1 : 0;
                }
            }
            // This stream's last PV has landed; every softmax thread agrees on
            // whether the piece completed.
            int w = ok ? 1 : 0;
            if (w && nmine > 0 && lane == 0) {
                const int ml = m - 1;   // this stream's last job
                w = mbar_wait(&pv_done[2 * s + (ml & 1)], (uint32_t)(ml >> 1) & 1u, abort);
            }
            w = __shfl_sync(FULL, w, 0);
            ok = bar_and(1, AL_NSM, w);
            const bool combine = !pc.direct && cmb_flag[npc & 1] != 0;
            ++npc;
            // Rows of this piece: with two tiles each stream writes its tile's
            // rows; with one tile the two accumulators (disjoint key sets of
            // the same rows) combine, and stream s writes d columns 64 s ..
            // Whether each accumulator holds this piece's sums is the same for
            // every thread (a stream without jobs in the piece holds a stale
            // O), so the TMEM loads below, which the whole warp must issue,
            // never diverge.
            const bool has_self = nmine > 0, has_other = T == 1 && nother > 0;
            float M = m_run, ltot = l_run;
            float w_self = 1.f, w_other = 0.f;
            if (T == 1) {
                sML[s * 128 + row] = make_float2(m_run, l_run);
                named_bar_sync(1, AL_NSM);
                const float2 o2 = sML[(1 - s) * 128 + row];
                M = fmaxf(m_run, o2.x);
                w_self = m_run == -INFINITY ? 0.f : fast_exp2(m_run - M);
                w_other = o2.x == -INFINITY ? 0.f : fast_exp2(o2.x - M);
                ltot = w_self * l_run + w_other * o2.y;
                named_bar_sync(1, AL_NSM);
            }
            // The rows out, compiled once per tile count: with two tiles a
            // thread writes all 128 d columns of its tile's row from one
            // accumulator, with one tile 64 columns (64 s ..) from two.
            auto rows_out = [&](auto tiles) {
                constexpr int TT = decltype(tiles)::value;
                constexpr int CN = TT == 2 ? 128 : 64;       // d columns this thread writes
                const int c_lo = TT == 2 ? 0 : 64 * s;
                __nv_bfloat16* dst = nullptr;
                if (rv) {
                    if (pc.direct || combine) {
                        const int i = qr / G, h = pc.g * G + qr % G;
                        dst = a.out + ((((size_t)pc.l * a.B + pc.b) * N + i) * a.Hq + h) * 128;
                    } else {
                        dst = a.part + (((size_t)pc.slot * TT + tile) * 128 + row) * 128;
                    }
                }
                const uint32_t o_other = lane_base + AL_OCOL + 128u * (uint32_t)(1 - s);
                // (combining: the other piece's log2-sum-exp and partial
                // columns, loaded 64 columns ahead of their use into a ring of
                // eight 16-byte chunks)
                uint4 pr[8];
                const uint4* psrc = nullptr;
                float a_self = 1.f, a_part = 0.f;
                if (combine && rv) {
                    const size_t prow = ((size_t)other_slot * TT + tile) * 128 + row;
                    const float lse_o = __ldcg(a.part_lse + prow);
                    psrc = reinterpret_cast<const uint4*>(a.part + prow * 128 + c_lo);
#pragma unroll
                    for (int q = 0; q < 8; ++q) pr[q] = __ldcg(psrc + q);
                    const float lse_s = ltot > 0.f ? M + log2f(ltot) : -INFINITY;
                    const float Mc = fmaxf(lse_s, lse_o);
                    const float es = lse_s == -INFINITY ? 0.f : fast_exp2(lse_s - Mc);
                    const float eo = lse_o == -INFINITY ? 0.f : fast_exp2(lse_o - Mc);
                    a_self = es / (es + eo);
                    a_part = eo / (es + eo);                     // (NaN when the other gave up)
                }
                if (ok) {
                    tc_fence_after();
                    const float inv = ltot > 0.f ? 1.0f / ltot : 0.f;
                    const float fs = w_self * inv * a_self, fo = w_other * inv * a_self;
                    // 16 columns at a time; after each step the two ring
                    // chunks it used are reloaded with those 64 columns on
#pragma unroll
                    for (int qt = 0; qt < CN / 16; ++qt) {
                        const int cq = c_lo + 16 * qt;       // (the columns of O this thread writes)
                        uint32_t os[16], oo[16];
                        if (has_self) tmem_ld16(ocol + (uint32_t)cq, os);
                        if (TT == 1 && has_other) tmem_ld16(o_other + (uint32_t)cq, oo);
                        tmem_wait_ld();
                        if (dst) {
                            uint32_t pv[8];
#pragma unroll
                            for (int u = 0; u < 8; ++u) {
                                const int e = 2 * u;     // column pair within the 16
                                float v0 = 0.f, v1 = 0.f;
                                if (has_self) {
                                    v0 = __uint_as_float(os[e]) * fs;
                                    v1 = __uint_as_float(os[e + 1]) * fs;
                                }
                                if (TT == 1 && has_other) {
                                    v0 = fmaf(__uint_as_float(oo[e]), fo, v0);
                                    v1 = fmaf(__uint_as_float(oo[e + 1]), fo, v1);
                                }
                                if (combine) {
                                    const uint4 q4 = pr[(2 * qt + (e >> 3)) & 7];
                                    const int wd = (e >> 1) & 3;
                                    const uint32_t pw = wd == 0 ? q4.x : wd == 1 ? q4.y : wd == 2 ? q4.z : q4.w;
                                    const float2 f = unpack_bf16(pw);
                                    v0 = fmaf(f.x, a_part, v0);
                                    v1 = fmaf(f.y, a_part, v1);
                                }
                                pv[u] = pack_bf16(v0, v1);
                            }
                            st_global_v8(dst + cq, pv);
                        }
                        if (psrc && qt + 4 < CN / 16) {
                            pr[(2 * qt) & 7] = __ldcg(psrc + 2 * (qt + 4));
                            pr[(2 * qt + 1) & 7] = __ldcg(psrc + 2 * (qt + 4) + 1);
                        }
                    }
                } else if (dst) {
                    // Gave up: NaN rows (whole piece, or combined) or an invalid partial.
                    const uint32_t fill = (pc.direct || combine) ? pack_bf16(NAN, NAN) : 0u;
                    const uint32_t pv[8] = {fill, fill, fill, fill, fill, fill, fill, fill};
                    for (int e = 0; e < CN; e += 16) st_global_v8(dst + c_lo + e, pv);
                }
            };
            if (T == 2)
                rows_out(AlTiles<2>{});
            else
                rows_out(AlTiles<1>{});
            if (!pc.direct && !combine && rv && (T == 2 || s == 0))
                a.part_lse[((size_t)pc.slot * T + tile) * 128 + row] =
                    ok ? (ltot > 0.f ? M + log2f(ltot) : -INFINITY) : NAN;
            // O has been read: the next piece's PV may overwrite it.
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(o_free);
            if (combine) {
                // (the other piece had arrived: the unit is done)
                if (t_id == 0) a.cnt[pc.unit] = 0;   // ready for the next call
            } else if (!pc.direct) {
                // Count this piece in the unit's arrivals; the last piece to
                // arrive combines the unit's pieces into the output.
                __threadfence();
                named_bar_sync(1, AL_NSM);
                if (t_id == 0) {
                    const int old = atomicAdd(a.cnt + pc.unit, 1);
                    __threadfence();
                    *last_flag = old == npieces - 1 ? 1 : 0;
                }
                named_bar_sync(1, AL_NSM);
                if (*last_flag) {
                    merge_unit(a, pc, U0, cf, cl, W, C, t_id);
                    if (t_id == 0) a.cnt[pc.unit] = 0;   // ready for the next call
                }
                named_bar_sync(1, AL_NSM);                // (last_flag is reused)
            }
            m0 = m;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, AL_TMEM_COLS);
}

// Rotates the queries of L layers into q_rot [L][B][N][Hq][128], writes the
// rotated tree keys and the values to treeK / treeV [L][B][Hkv][N][128] (the
// scratch gv_kv_compact reads, and the tree block of attn_layers_kernel), and
// zeroes the arrival counters.  One thread per (row, 16-byte chunk of the low
// half); the rotation is rope8, the arithmetic of the per-layer kernel.
__global__ void __launch_bounds__(256)
tree_prep_kernel(const __nv_bfloat16* __restrict__ q, long long q_ls, const __nv_bfloat16* __restrict__ k,
                 long long k_ls, const __nv_bfloat16* __restrict__ v, long long v_ls, int L, int B, int N, int Hq,
                 int Hkv, const float* __restrict__ rope, __nv_bfloat16* __restrict__ q_rot,
                 __nv_bfloat16* __restrict__ treeK, __nv_bfloat16* __restrict__ treeV, int* __restrict__ cnt,
                 int ncnt) {
    pdl_wait();
    pdl_trigger();
    // (32-bit index arithmetic: the host bounds 8 L B N (Hq + 2 Hkv) by 2^30)
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t < ncnt) cnt[t] = 0;
    const int nqr = B * N * Hq, nkr = B * N * Hkv;
    const int nq = L * nqr, nk = L * nkr;
    const int c = t & 7;
    if (t < 8 * nq) {
        const int row = t >> 3;
        const int l = row / nqr, r = row - l * nqr;
        const int bn = r / Hq;
        const uint4* src = reinterpret_cast<const uint4*>(q + l * q_ls + (long long)r * 128);
        const uint4 lo = __ldg(src + c), hi = __ldg(src + 8 + c);
        const float4* cs = reinterpret_cast<const float4*>(rope) + bn * 32 + c * 4;
        float4 c4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) c4[e] = __ldg(cs + e);
        uint4 olo, ohi;
        rope8(lo, hi, c4, olo, ohi);
        uint4* dst = reinterpret_cast<uint4*>(q_rot) + (long long)row * 16;
        dst[c] = olo;
        dst[8 + c] = ohi;
        return;
    }
    const int u = t - 8 * nq;
    if (u >= 16 * nk) return;
    const bool isk = u < 8 * nk;
    const int row = (isk ? u : u - 8 * nk) >> 3;
    const int l = row / nkr, r = row - l * nkr;               // r = (b * N + n) * Hkv + h
    const int bn = r / Hkv;
    const int h = r - bn * Hkv;
    const int b = bn / N, n = bn - b * N;
    const long long drow = ((long long)(l * B + b) * Hkv + h) * N + n;   // [L][B][Hkv][N]
    if (isk) {
        const uint4* src = reinterpret_cast<const uint4*>(k + l * k_ls + (long long)r * 128);
        const uint4 lo = __ldg(src + c), hi = __ldg(src + 8 + c);
        const float4* cs = reinterpret_cast<const float4*>(rope) + bn * 32 + c * 4;
        float4 c4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) c4[e] = __ldg(cs + e);
        uint4 olo, ohi;
        rope8(lo, hi, c4, olo, ohi);
        uint4* dst = reinterpret_cast<uint4*>(treeK) + drow * 16;
        dst[c] = olo;
        dst[8 + c] = ohi;
    } else {
        const uint4* src = reinterpret_cast<const uint4*>(v + l * v_ls + (long long)r * 128);
        uint4* dst = reinterpret_cast<uint4*>(treeV) + drow * 16;
        dst[c] = __ldg(src + c);
        dst[8 + c] = __ldg(src + 8 + c);
    }
}

// ----------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();

// bf16 tensor map of `rank` dims (dims[0] = 128 d elements, contiguous),
// 128-byte swizzle, box {64, box[1..]}.
static int make_map(CUtensorMap* map, const void* base, int rank, const cuuint64_t* dims,
                    const cuuint64_t* strides_bytes, const cuuint32_t* box, const char* what) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled unavailable");
        return GV_ERR_CUDA;
    }
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), dims,
                     strides_bytes, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled (%s) failed (%d)", what, (int)r);
        return GV_ERR_CUDA;
    }
    return GV_OK;
}

AttnLayersPlan attn_layers_plan(int L, int B, int N, int Hq, int Hkv) {
    AttnLayersPlan p{};
    const int G = Hq / Hkv;
    p.T = (G * N + 127) / 128;
    p.ctas = sm_count();
    auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
    p.q_rot = 0;
    size_t off = up((size_t)L * B * N * Hq * 128 * 2);
    p.cnt = off;
    p.ncnt = L * B * Hkv;
    off += up((size_t)p.ncnt * 4);
    p.part = off;
    off += up((size_t)2 * p.ctas * p.T * 128 * 128 * 2);
    p.part_lse = off;
    off += up((size_t)2 * p.ctas * p.T * 128 * 4);
    p.total = off;
    return p;
}

int launch_attn_layers(const AttnLayersCall& c, cudaStream_t st) {
    const int G = c.Hq / c.Hkv;
    const AttnLayersPlan plan = attn_layers_plan(c.L, c.B, c.N, c.Hq, c.Hkv);
    char* ws = static_cast<char*>(c.workspace);
    __nv_bfloat16* q_rot = reinterpret_cast<__nv_bfloat16*>(ws + plan.q_rot);
    int* cnt = reinterpret_cast<int*>(ws + plan.cnt);
    // 1. rotation of the queries and tree keys, the tree K/V scratch, counters
    {
        const long long nq = (long long)c.L * c.B * c.N * c.Hq, nk = (long long)c.L * c.B * c.N * c.Hkv;
        const long long threads = 8 * nq + 16 * nk;
        cudaError_t e = launch_pdl(tree_prep_kernel, dim3((unsigned)((threads + 255) / 256)), dim3(256), 0, st,
                                   static_cast<const __nv_bfloat16*>(c.q), c.q_ls,
                                   static_cast<const __nv_bfloat16*>(c.k_new), c.k_ls,
                                   static_cast<const __nv_bfloat16*>(c.v_new), c.v_ls, c.L, c.B, c.N, c.Hq, c.Hkv,
                                   c.rope, q_rot, static_cast<__nv_bfloat16*>(c.treeK),
                                   static_cast<__nv_bfloat16*>(c.treeV), cnt, plan.ncnt);
        if (e != cudaSuccess) {
            set_error("tree_prep_kernel launch: %s", cudaGetErrorString(e));
            return GV_ERR_CUDA;
        }
    }
    // 2. the attention of every layer
    CUtensorMap mck, mcv, mtk, mtv, mq;
    {
        const cuuint64_t dims[3] = {128, (cuuint64_t)c.B * c.Hkv * c.S_max, (cuuint64_t)c.L};
        const cuuint64_t str[2] = {256, (cuuint64_t)c.cache_ls * 2};
        const cuuint32_t box[3] = {64, 128, 1};
        int rc = make_map(&mck, c.cacheK, 3, dims, str, box, "cacheK");
        if (rc != GV_OK) return rc;
        rc = make_map(&mcv, c.cacheV, 3, dims, str, box, "cacheV");
        if (rc != GV_OK) return rc;
    }
    {
        const cuuint64_t dims[2] = {128, (cuuint64_t)c.L * c.B * c.Hkv * c.N};
        const cuuint64_t str[1] = {256};
        const cuuint32_t box[2] = {64, (cuuint32_t)c.N};
        int rc = make_map(&mtk, c.treeK, 2, dims, str, box, "treeK");
        if (rc != GV_OK) return rc;
        rc = make_map(&mtv, c.treeV, 2, dims, str, box, "treeV");
        if (rc != GV_OK) return rc;
    }
    const int boxn = 128 / G < c.N ? 128 / G : c.N;
    {
        const cuuint64_t dims[4] = {128, (cuuint64_t)c.Hq, (cuuint64_t)c.N, (cuuint64_t)c.L * c.B};
        const cuuint64_t str[3] = {256, (cuuint64_t)c.Hq * 256, (cuuint64_t)c.N * c.Hq * 256};
        const cuuint32_t box[4] = {64, (cuuint32_t)G, (cuuint32_t)boxn, 1};
        int rc = make_map(&mq, q_rot, 4, dims, str, box, "q_rot");
        if (rc != GV_OK) return rc;
    }
    AttnLayersArgs a{};
    a.L = c.L;
    a.B = c.B;
    a.N = c.N;
    a.Hq = c.Hq;
    a.Hkv = c.Hkv;
    a.G = G;
    a.T = plan.T;
    a.S_max = c.S_max;
    a.boxn = boxn;
    a.scale = 1.0f / sqrtf(128.0f);
    a.prefix_len = c.prefix_len;
    a.anc = reinterpret_cast<const unsigned long long*>(c.anc);
    a.out = static_cast<__nv_bfloat16*>(c.out);
    a.part = reinterpret_cast<__nv_bfloat16*>(ws + plan.part);
    a.part_lse = reinterpret_cast<float*>(ws + plan.part_lse);
    a.cnt = cnt;
    cudaFuncSetAttribute(attn_layers_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, AL_SMEM);
    cudaError_t e = launch_pdl(attn_layers_kernel, dim3((unsigned)plan.ctas), dim3(AL_NTH), (size_t)AL_SMEM, st, mck,
                               mcv, mtk, mtv, mq, a);
    if (e != cudaSuccess) {
        set_error("attn_layers_kernel launch: %s", cudaGetErrorString(e));
        return GV_ERR_CUDA;
    }
    return GV_OK;
}

}  // namespace gv
