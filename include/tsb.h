/*
 * tsb.h -- C ABI of libtsb, a GB300 (sm_103a) library for the per-step logit path of
 * Tsubame's two-pass tree speculative decoding (Weng, Hu & Yairi, "Tsubame: Tree Replay for
 * Diffusion-Based Speculative Decoding").
 *
 * One decoding step on B independent trees:
 *
 *   tsb_row_stats   draft rows            -> chunk statistics (max, sum of exp)
 *   tsb_plan        draft rows + stats    -> frozen topology T (first pass, Sec. 3.1)
 *   tsb_plan_rows   draft rows            -> their statistics + T, in one pass over the rows
 *   tsb_replay      q rows + stats + T    -> one fresh token per node (second pass, Sec. 3.2)
 *   tsb_verify      target rows + q rows + T + tokens -> accepted path and final token
 *                   (recursive rejection sampling, Sec. 2.3 and App. A; block verification
 *                   of a sampled chain, Sun et al. 2025 as cited in Sec. 1 and App. A; or
 *                   target-sample matching, Table 2)
 *   tsb_replay_verify  tsb_replay + tsb_verify (recursive rejection sampling) in one call, the
 *                   verifier's target-row pre-pass running beside the replay draws
 *
 * and the paper's other choices for each pass:
 *
 *   tsb_plan_expand, tsb_plan_rows_expand   expand-then-prune first pass (Sec. 3.1, App. B.3)
 *   tsb_replay_mixed                        mixed sampling in the second pass (App. A)
 *   tsb_plan_pooled, tsb_replay_pooled,     draft laws restricted to per-position pools of the
 *   tsb_verify_pooled                       P most probable tokens (Sec. 3.1-3.3)
 *
 * Conventions
 *   - Every tensor pointer is a DEVICE pointer owned by the caller. The library never
 *     allocates, frees or synchronises; the only call that waits is tsb_device_status.
 *   - Calls are asynchronous on the given stream (NULL = legacy default stream).
 *   - Host validation runs before anything is launched; on any error status nothing has
 *     been launched and no output was touched.
 *   - Problems that only the device can see (non-finite logits, an index out of range in a
 *     caller-supplied array) set bits in a sticky status word kept in the caller's workspace;
 *     tsb_device_status reads and clears it. Outputs of a call that set a bit are undefined.
 *   - Functions keep no global state and are safe to call from several host threads on
 *     different workspaces. The one exception is tsb_plan_noalloc, whose scratch is a
 *     static device array (see there).
 *   - Logits: element (b, r, v) is at data[b*batch_stride + r*row_stride + v], in elements.
 *     batch_stride may be 0 (every tree shares the same rows). Every row must start on a
 *     16-byte boundary (data, batch_stride*elem_size and row_stride*elem_size multiples of 16).
 *     Values must be finite. A logit z is used as x = fp32(z) * fp32(1/T), one fp32 multiply.
 *   - Randomness is Philox4x32-10 (Salmon et al., SC 2011) with key {seed lo32, seed hi32} and
 *     counter {draw/4, node, batch, purpose}, word draw%4, uniform U = (w>>8 + 1/2) * 2^-24.
 *     Every draw is keyed by what it is, so results do not depend on launch geometry.
 */
#ifndef TSB_H
#define TSB_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *tsb_stream; /* the same type as cudaStream_t */

typedef enum {
    TSB_OK = 0,
    TSB_ERR_ARG = 1,       /* NULL pointer, bad enum, non-positive or non-finite temperature */
    TSB_ERR_SHAPE = 2,     /* sizes out of range or inconsistent between arguments */
    TSB_ERR_DTYPE = 3,     /* logits dtype not TSB_F32 / TSB_BF16 */
    TSB_ERR_ALIGN = 4,     /* a row does not start on a 16-byte boundary */
    TSB_ERR_WORKSPACE = 5, /* workspace or stats buffer too small or misaligned */
    TSB_ERR_CUDA = 6,      /* a CUDA runtime call or kernel launch failed */
    TSB_ERR_DEVICE = 7     /* tsb_device_status found device-side status bits set */
} tsb_status;

/* Device status bits (sticky, in the workspace). */
#define TSB_DEV_NONFINITE 0x1u /* a logit was NaN or infinite after the temperature multiply */
#define TSB_DEV_BAD_INDEX 0x2u /* a token, row index or child index was out of range */
#define TSB_DEV_BAD_TREE 0x4u  /* tree arrays inconsistent (e.g. block verification on a non-chain) */
#define TSB_DEV_CHECK 0x8u     /* libtsb_checked.so: a bounds check of a data-dependent index failed */

typedef enum { TSB_F32 = 0, TSB_BF16 = 1 } tsb_dtype;

typedef enum {
    TSB_VERIFY_RRS = 0,   /* recursive rejection sampling, WoR candidates, any topology */
    TSB_VERIFY_BLOCK = 1, /* block verification; the topology must be the chain 0->1->...->N */
    TSB_VERIFY_NAIVE = 2, /* target-sample matching: any topology, any way of filling it */
    TSB_VERIFY_TRAVERSAL = 3 /* traversal verification, WoR candidates, any topology */
} tsb_verify_mode;

/* Limits (validated). */
#define TSB_MAX_WIDTH 1024              /* frontier width of the expand-then-prune first pass */
#define TSB_MAX_POOL 64                 /* tokens in a pooled draft law (one warp, two per lane) */
#define TSB_MAX_EXPAND_CANDIDATES 8192  /* candidates it may generate: K + (L-1) layers of <= W*K */
#define TSB_CHUNK 256 /* fixed chunk of the chunk statistics and of the replay sampler */
#define TSB_MAX_K 32
#define TSB_MAX_L 64
#define TSB_MAX_N 1024
#define TSB_MAX_B 1048576
#define TSB_MAX_V 409600 /* the verifier keeps one target and one q row slice per CTA in shared memory */

typedef struct {
    const void *data;     /* device pointer */
    int32_t dtype;        /* tsb_dtype */
    int32_t B, R, V;      /* trees, rows per tree, vocabulary */
    int64_t batch_stride; /* elements between trees (0 = shared rows) */
    int64_t row_stride;   /* elements between rows, >= V */
} tsb_logits;

typedef struct {
    int32_t B;         /* trees in the batch, 1..TSB_MAX_B */
    int32_t L;         /* draft block length = depth cap, 1..TSB_MAX_L */
    int32_t N;         /* planned nodes besides the root, 1..TSB_MAX_N, N <= K + K^2 + ... + K^L */
    int32_t K;         /* candidates per draft row = maximum children per node, 1..TSB_MAX_K, K <= V */
    int32_t V;         /* vocabulary, 1..TSB_MAX_V */
    float temperature; /* T > 0 and finite; applied to draft, q and target rows alike */
} tsb_cfg;

/* Frozen topology, device arrays. Node 0 is the root; nodes 1..N are numbered in the order
 * the first pass pops them, so parent[i] < i. The children of u, in slot (rank) order, are
 * child_ids[child_off[u] .. child_off[u+1]). */
typedef struct {
    int32_t *parent;     /* [B, N+1], parent[0] = -1 */
    int32_t *depth;      /* [B, N+1], depth[0] = 0 */
    int32_t *rank;       /* [B, N+1], slot among siblings; rank[0] = -1 */
    int32_t *plan_token; /* [B, N+1], first-pass token (discarded by replay); -1 at the root */
    float *score;        /* [B, N+1], draft path log-probability; 0 at the root */
    int32_t *child_off;  /* [B, N+2] */
    int32_t *child_ids;  /* [B, N] */
} tsb_tree;

/* Library version, major*10000 + minor*100 + patch. */
int32_t tsb_version(void);

/* Human-readable name of a status. Never NULL. */
const char *tsb_status_str(tsb_status status);

/* Bytes of the chunk-statistics buffer for B*R rows of V logits: one (max, sum exp) float
 * pair per chunk of TSB_CHUNK logits, [B][R][ceil(V/TSB_CHUNK)]. 0 if the sizes are invalid. */
size_t tsb_stats_bytes(int32_t B, int32_t R, int32_t V);

/* Bytes of the workspace for a configuration: a status word (256 bytes), per-(tree, node)
 * scalars of the verifiers (B*(N+1)*32), the partial row normalisers of the recursive
 * rejection pre-pass (B*1024) and the first pass's per-draft-row results (B*L*(8 + 8*K)). The
 * workspace must be 256-byte aligned; tsb_row_stats needs only the first 256 bytes. 0 if the
 * configuration is invalid. */
size_t tsb_workspace_bytes(const tsb_cfg *cfg);

/* Zero the workspace's status word on the stream. Call once before first use. */
tsb_status tsb_workspace_init(void *ws, size_t ws_bytes, tsb_stream stream);

/* Waits for the stream, then returns the device status bits in *bits and clears them.
 * Returns TSB_OK if no bit was set, TSB_ERR_DEVICE if some were, TSB_ERR_CUDA if the CUDA
 * context reported an error. */
tsb_status tsb_device_status(void *ws, tsb_stream stream, uint32_t *bits);

/* Chunk statistics of every row (the streaming pass over the logits): for chunk
 * c = [c*TSB_CHUNK, min(V, (c+1)*TSB_CHUNK)) of row (b, r) it writes
 * stats[(b*R + r)*C + c] = { m_c = max x_v, s_c = sum exp(x_v - m_c) }, x = fp32(z)*fp32(1/T).
 * They give every row's log-normaliser, the per-position candidate pools of the first pass
 * (Sec. 3.1) and the chunk log-masses of the replay sampler. stats: float2-aligned device
 * buffer of tsb_stats_bytes(B, R, V). */
tsb_status tsb_row_stats(const tsb_logits *rows, float temperature, void *stats, size_t stats_bytes, void *ws,
                         size_t ws_bytes, tsb_stream stream);

/* First pass (Sec. 3.1, App. B.3): per draft row d the top-K tokens by (x desc, id asc),
 * then best-first (max-heap) expansion by cumulative draft path log-probability, popping N
 * nodes. Candidates pop in the order (path log-probability desc, depth asc, parent asc,
 * rank asc), where parent is the parent's node number; two candidates of the same depth
 * compare their path log-probabilities exactly (they share the depth's log-normaliser
 * prefix, so only their sums of x differ). A node at depth d takes its token from draft row
 * d-1; a node at depth L gets no children. draft: [B, >=L, V]; draft_stats: tsb_row_stats of the same rows
 * and temperature. Writes every array of *out. */
tsb_status tsb_plan(const tsb_cfg *cfg, const tsb_logits *draft, const void *draft_stats, size_t stats_bytes,
                    const tsb_tree *out, void *ws, size_t ws_bytes, tsb_stream stream);

/* tsb_row_stats of draft rows 0..L-1 and tsb_plan in one pass over those rows: each draft
 * row is streamed once by one CTA, which writes the row's chunk statistics to draft_stats
 * (layout and bits exactly as tsb_row_stats writes them; rows L..R-1 are not written) and then
 * runs the first pass's top-K on them while the candidate chunks are still in L2; then the
 * best-first expansion as in tsb_plan (Sec. 3.1, App. B.3). draft_stats: float2-aligned
 * device buffer of tsb_stats_bytes(B, R, V), an output here. Other arguments and errors as in
 * tsb_plan; non-finite logits set TSB_DEV_NONFINITE. */
tsb_status tsb_plan_rows(const tsb_cfg *cfg, const tsb_logits *draft, void *draft_stats, size_t stats_bytes,
                         const tsb_tree *out, void *ws, size_t ws_bytes, tsb_stream stream);

/* First pass by expand-then-prune (Sec. 3.1 and App. B.3: the EAGLE-2-style planner the paper
 * uses for drafters that correct logits per prefix). Depth by depth, the `width` best
 * candidates of the newest layer (its frontier) get their K children each (a node at depth L
 * gets none); after the last depth the N best of all generated candidates are the nodes,
 * numbered in the order (path log-probability desc, depth asc, parent's position in its layer
 * asc, rank asc). Path scores, tokens and output layout are those of tsb_plan; with width >= N
 * the tree is the max-heap tree of tsb_plan. Inside a layer the order is the same one, and a
 * frontier is a prefix of its sorted layer.
 * width: 1..TSB_MAX_WIDTH. The number of generated candidates, K + sum over depths 2..L of
 * min(width, previous layer) * K, must be at least N and at most TSB_MAX_EXPAND_CANDIDATES,
 * else TSB_ERR_SHAPE. A child whose rounded score came out above its parent's (a draft row
 * with all its mass on one token) sets TSB_DEV_BAD_TREE.
 * tsb_plan_expand takes the draft statistics as input like tsb_plan; tsb_plan_rows_expand
 * computes and writes them in the same pass over the rows like tsb_plan_rows. Other arguments
 * and errors as in tsb_plan / tsb_plan_rows. */
tsb_status tsb_plan_expand(const tsb_cfg *cfg, int32_t width, const tsb_logits *draft, const void *draft_stats,
                           size_t stats_bytes, const tsb_tree *out, void *ws, size_t ws_bytes, tsb_stream stream);
tsb_status tsb_plan_rows_expand(const tsb_cfg *cfg, int32_t width, const tsb_logits *draft, void *draft_stats,
                                size_t stats_bytes, const tsb_tree *out, void *ws, size_t ws_bytes,
                                tsb_stream stream);

/* Pooled draft laws (Sec. 3.1: the draft law of a position is restricted to a pool of its P
 * most probable tokens and normalised within it; Sec. 3.2: replay uses the same pools; Sec. 3.3:
 * verification uses the pooled probabilities, the target law and the residual stay
 * full-vocabulary). The pool of the tokens at depth d+1 is the P most probable tokens of draft
 * row d by (x desc, id asc); it serves every node at depth d, whatever its q row.
 *
 * tsb_plan_pooled: tsb_plan with each depth's law normalised over its pool; the candidates are
 *   the pool's first K tokens (K <= P <= TSB_MAX_POOL, P <= V, else TSB_ERR_SHAPE). Writes the
 *   pools to pool_ids (device, caller-owned, [B, L, P] int32, sorted by (x desc, id asc)) and
 *   *out as tsb_plan does. draft_stats: tsb_row_stats of the draft rows.
 * tsb_replay_pooled: for every parent u with m_u children, the m_u ordered draws without
 *   replacement from q_u restricted to pool row depth[u] and renormalised there: the top-m_u
 *   Gumbel keys x_v + G(U[replay element, u, v]) over the P pool tokens. qrows / qrow_of_node
 *   as in tsb_replay (no statistics needed).
 * tsb_verify_pooled: recursive rejection sampling as tsb_verify's TSB_VERIFY_RRS with q_u the
 *   pooled law; a child token outside the pool has draft probability 0 and is accepted.
 * Other arguments, layouts and errors as in tsb_plan / tsb_replay / tsb_verify; a pool token
 * out of range sets TSB_DEV_BAD_INDEX. */
tsb_status tsb_plan_pooled(const tsb_cfg *cfg, int32_t P, const tsb_logits *draft, const void *draft_stats,
                           size_t stats_bytes, int32_t *pool_ids, const tsb_tree *out, void *ws, size_t ws_bytes,
                           tsb_stream stream);
tsb_status tsb_replay_pooled(const tsb_cfg *cfg, int32_t P, const tsb_logits *qrows, const int32_t *qrow_of_node,
                             const int32_t *pool_ids, const tsb_tree *tree, uint64_t seed, int32_t *token, void *ws,
                             size_t ws_bytes, tsb_stream stream);
tsb_status tsb_verify_pooled(const tsb_cfg *cfg, int32_t P, const tsb_logits *target, const tsb_logits *qrows,
                             const int32_t *qrow_of_node, const int32_t *pool_ids, const tsb_tree *tree,
                             const int32_t *token, uint64_t seed, int32_t *out_tokens, int32_t *out_nodes,
                             int32_t *out_len, void *ws, size_t ws_bytes, tsb_stream stream);

/* Size of the device scratch array behind tsb_plan_noalloc (1 MiB per device). */
#define TSB_NOALLOC_SCRATCH_BYTES ((size_t)1 << 20)

/* tsb_plan without a workspace and without any allocation. The paper has no counterpart:
 * this is a calling convention, not a step of the method. It is for callers that cannot
 * call cudaMalloc: a plug-in whose host program owns all device memory and hands it only
 * its input and output tensors; a serving engine that reserves the device's memory up
 * front for its own pool; a hot loop that cannot pay cudaMalloc's implicit device-wide
 * synchronisation. It computes exactly what tsb_plan computes, with the same kernels,
 * and writes the same *out.
 *
 * Scratch: a single static device array of TSB_NOALLOC_SCRATCH_BYTES that every device
 * loading this library holds until the process exits. A configuration needs
 * 256 + B*L*(8 + 8*K) bytes of it; larger ones return TSB_ERR_SHAPE before anything is
 * launched (for example B <= 910 trees at L = 16, K = 8). All calls on a device share the
 * array and it keeps the last call's contents, so calls whose kernels may overlap on the
 * GPU (different streams, or different host threads, without ordering between them) race
 * and give undefined outputs: order them on one stream or with events.
 *
 * Set-up: every call looks up the array's device address on the current device with
 * cudaGetSymbolAddress (nothing is cached, so a cudaDeviceReset leaves no stale address);
 * the first call on a device may load the library's module there, so make that first call
 * before any stream capture on the device. The call allocates and frees nothing and calls
 * no allocating library routine.
 *
 * dev_status: optional 4-byte aligned device word, owned by the caller, into which the
 * device status bits (TSB_DEV_*) are OR-ed; the caller clears it (it may be the status
 * word of a workspace set up by tsb_workspace_init, which tsb_device_status then reads).
 * With NULL the bits go to a word inside the scratch that each call clears first and that
 * nothing reads. Other arguments and errors as in tsb_plan. */
tsb_status tsb_plan_noalloc(const tsb_cfg *cfg, const tsb_logits *draft, const void *draft_stats, size_t stats_bytes,
                            const tsb_tree *out, uint32_t *dev_status, tsb_stream stream);

/* Second pass (Sec. 3.2, Eq. replay-distribution; WoR as in App. A): for every parent u
 * with m_u children, draws m_u tokens without replacement from q_u = softmax(x of row
 * qrow(u)) and writes the j-th draw to child slot j: token[b, child_ids[child_off[u]+j]].
 * token[b, 0] = -1. qrows: [B, Rq, V] with its stats (same temperature); qrow_of_node:
 * [B, N+1] row index per node, or NULL for per-depth rows (qrow(u) = depth[u]). The draws
 * are the top-m_u Gumbel keys, built top-down over chunks of TSB_CHUNK tokens. */
tsb_status tsb_replay(const tsb_cfg *cfg, const tsb_logits *qrows, const void *qstats, size_t stats_bytes,
                      const int32_t *qrow_of_node, const tsb_tree *tree, uint64_t seed, int32_t *token, void *ws,
                      size_t ws_bytes, tsb_stream stream);

/* Second pass with mixed sampling (Sec. 3.2 and App. A; the greedy draft sampling of Hu et
 * al. 2025): for every parent u with m_u children, child slots 0..m_u-2 take the m_u-1 most
 * probable tokens of q_u in order, by (x desc, id asc), and slot m_u-1 takes one draw from q_u
 * renormalised over the other tokens: the largest Gumbel key among them, with the keys of
 * tsb_replay's top-down construction (so with m_u = 1 the token is tsb_replay's). Arguments,
 * layout and errors as in tsb_replay. Pair it with TSB_VERIFY_NAIVE: recursive rejection
 * sampling assumes WoR candidates and is not lossless for these. */
tsb_status tsb_replay_mixed(const tsb_cfg *cfg, const tsb_logits *qrows, const void *qstats, size_t stats_bytes,
                            const int32_t *qrow_of_node, const tsb_tree *tree, uint64_t seed, int32_t *token,
                            void *ws, size_t ws_bytes, tsb_stream stream);

/* Verification on the frozen topology with the replayed tokens (Prop. 1).
 * TSB_VERIFY_RRS: from the root, test the children in slot order, accept child i iff
 *   U * q'(y_i) < p'(y_i) with q' the draft law renormalised over tokens not yet drawn and
 *   p' the current residual target law; on rejection p' <- max(p' - q', 0) normalised over
 *   the full vocabulary. An accepted child is emitted and the walk continues there; when all
 *   children are rejected the final token is drawn from the last residual; at a leaf the
 *   bonus token is drawn from the node's target row.
 * TSB_VERIFY_BLOCK: block verification of the chain 0->1->...->N (requires N <= L).
 * TSB_VERIFY_TRAVERSAL: traversal verification (Sec. 2.3, Table 2 "Traversal" and App. A:
 *   recursive rejection sampling lifted to sequences, for WoR candidates; UniVer reduces to it
 *   under WoR). The tree is traversed depth first, children in slot order, and a node is tried
 *   only once every child subtree below it has been rejected; it is accepted iff
 *   U[accept, node] < p_a(node), the root always. Entering child c (token y) of u gives
 *   p_a(c) = min(p_a(u) Mb_u(y) / Ms_u(y), 1) with p_a(root) = 1, Mb_u = softmax(target row u)
 *   and Ms_u = q_u renormalised over tokens of u's children not yet rejected. After the subtree
 *   of a child is rejected: R = max(p_a(u) Mb_u - Ms_u, 0), p_a(u) <- sum R / (sum R + 1 -
 *   p_a(u)), Mb_u <- R / sum R. Accepting u emits the path to u and a final token: from the last
 *   R if u had children, the bonus from u's target row otherwise. On a chain this is block
 *   verification, at the root recursive rejection sampling. Every internal node's target row is
 *   normalised (one parallel pass), so the call reads each internal node's row at least once.
 * TSB_VERIFY_NAIVE: target-sample matching (Sec. 2.3, "Naive" in Table 2): from the root, draw
 *   y from the node's target law (the two-level Gumbel-max of the bonus token); the first child
 *   carrying y is accepted and the walk continues there, otherwise y is the final token. Each
 *   emitted token is a draw from the target law, whatever the children hold, so it verifies the
 *   first-pass tokens (plan_token) as well as WoR or mixed replays; a child with token v is
 *   accepted with probability p(v). qrows, qstats and qrow_of_node are not used and may be
 *   NULL. Only the visited nodes' target rows are read (one cluster of CTAs walks each tree);
 *   a visited row holding a NaN or +inf logit sets TSB_DEV_NONFINITE.
 * target: [B, N+1, V], row u = target logits after the path to node u. qrows / qstats /
 * qrow_of_node as in tsb_replay. Outputs: out_tokens [B, L+1] (accepted tokens then the
 * final token, -1 after), out_nodes [B, L] (accepted node ids, -1 after), out_len [B]
 * (number of emitted tokens = accepted + 1). */
tsb_status tsb_verify(const tsb_cfg *cfg, int32_t mode, const tsb_logits *target, const tsb_logits *qrows,
                      const void *qstats, size_t stats_bytes, const int32_t *qrow_of_node, const tsb_tree *tree,
                      const int32_t *token, uint64_t seed, int32_t *out_tokens, int32_t *out_nodes,
                      int32_t *out_len, void *ws, size_t ws_bytes, tsb_stream stream);

/* tsb_replay followed by tsb_verify with TSB_VERIFY_RRS, same seed, in one call: the same
 * tokens and outputs bit for bit. The verifier's pass over the target rows that it normalises
 * ahead of the walk (the first internal nodes of each tree's first-child chain) reads only the
 * tree and the target rows, so it runs in the same grid as the replay draws instead of after
 * them. token [B, N+1] is written as by tsb_replay; the other arguments, layouts and errors are
 * those of tsb_replay and tsb_verify. */
tsb_status tsb_replay_verify(const tsb_cfg *cfg, const tsb_logits *target, const tsb_logits *qrows, const void *qstats,
                             size_t stats_bytes, const int32_t *qrow_of_node, const tsb_tree *tree, uint64_t seed,
                             int32_t *token, int32_t *out_tokens, int32_t *out_nodes, int32_t *out_len, void *ws,
                             size_t ws_bytes, tsb_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* TSB_H */
