/*
 * libraspec — the LibraSpec verify round on NVIDIA GB300 (sm_103a).
 *
 * One decoding round of diffusion-drafted speculative decoding with the
 * LibraSpec length controller (arxiv 2608.08721), as four device steps:
 *
 *   1. libraspec_confidence      drafter confidence q of every drafted token
 *   2. libraspec_select_lengths  per-sequence speculative length L_b
 *   3. libraspec_verify_attn     block-causal GQA verify attention (per layer)
 *   4. libraspec_accept          greedy / rejection-sampling acceptance
 *
 * libraspec_verify_round runs all four on one stream.
 *
 * Conventions shared by every call
 * --------------------------------
 * - Every tensor pointer is a DEVICE pointer owned by the caller, contiguous
 *   and row-major in the layout stated (last index fastest). The library
 *   never frees or keeps them.
 * - bf16 tensors are passed as uint16_t bit patterns.
 * - `stream` is a cudaStream_t (NULL = the legacy default stream). Calls only
 *   enqueue work on it and return without synchronising, except
 *   libraspec_get_status.
 * - The library allocates no device memory. Calls that need scratch space
 *   take a caller-provided `workspace` of at least libraspec_workspace_size()
 *   bytes, 256-byte aligned and zero-filled once before first use
 *   (libraspec_workspace_init). Every call leaves its counters at zero again,
 *   so a workspace can be reused by any number of calls in stream order.
 *   Calls sharing one workspace must not overlap on the GPU.
 * - Return value: LIBRASPEC_OK, or a negative status (below). Arguments are
 *   checked on the host before anything is enqueued. Conditions only the
 *   device can see (a selected length out of range, a non-positive cost, a
 *   KV cache too short for the block) set a status word in the workspace,
 *   read by libraspec_get_status. Kernels never trap and never spin without
 *   a bound.
 * - Logits must be finite. Vocabulary sizes need not be multiples of 4, but
 *   rows whose byte length is a multiple of 16 use the vectorised path.
 *
 * Batch sharding: `seq_offset` is added to the batch index b wherever a
 * random number is drawn, so a batch split over several GPUs draws exactly
 * the numbers the unsplit batch would.
 */
#ifndef LIBRASPEC_H
#define LIBRASPEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LIBRASPEC_OK 0
#define LIBRASPEC_EINVAL (-1)       /* null pointer, bad shape or alignment     */
#define LIBRASPEC_EUNSUPPORTED (-2) /* valid but not supported (e.g. head dim)  */
#define LIBRASPEC_ECUDA (-3)        /* a CUDA runtime call or launch failed     */
#define LIBRASPEC_EDEVICE (-4)      /* a kernel reported a violation (status)   */

/* Device status bits (libraspec_get_status). */
#define LIBRASPEC_ST_BAD_LENGTH 0x1  /* L_b outside [0, K]                       */
#define LIBRASPEC_ST_BAD_COST 0x2    /* cost_table entry not positive and finite */
#define LIBRASPEC_ST_KV_OVERFLOW 0x4 /* kv_len_b + L_b + 1 > S_cap or kv_len < 0 */
#define LIBRASPEC_ST_BAD_TOKEN 0x8   /* draft token outside [0, V)               */
#define LIBRASPEC_ST_TIMEOUT 0x10    /* a bounded wait (async copy, grid barrier) expired */
#define LIBRASPEC_ST_MISSING_INPUT 0x20 /* sampling sequence but conf/dstat NULL  */
#define LIBRASPEC_ST_BAD_PAGE 0x40   /* a block-table entry outside [0, n_pages)  */
#define LIBRASPEC_ST_BAD_TREE 0x80   /* a draft-tree parent outside [0, t)        */

/* Limits of the library. */
#define LIBRASPEC_MAX_K 64           /* drafter block length / d_max             */
#define LIBRASPEC_MAX_B 4096         /* sequences per call                       */
#define LIBRASPEC_MAX_TREE_NODES 512 /* nodes below the root of a draft tree      */

/* Version string of the library. */
const char* libraspec_version(void);

/* Human-readable name of a status code returned by any call. */
const char* libraspec_status_string(int status);

/*
 * Bytes of workspace a round with these shapes needs (all calls of the
 * round may share it). B sequences, K drafter block length (the node
 * budget N for the draft-tree calls, up to LIBRASPEC_MAX_TREE_NODES), V
 * vocabulary, Hq / Hkv query / kv heads, head_dim, S_cap cache capacity per
 * (b, kv head). Pure host function; returns 0 for invalid shapes.
 */
size_t libraspec_workspace_size(int B, int K, int V, int Hq, int Hkv, int head_dim, int S_cap);

/* Zero-fill `bytes` of workspace on `stream` (cudaMemsetAsync). */
int libraspec_workspace_init(void* workspace, size_t bytes, void* stream);

/*
 * Synchronise `stream`, copy the device status word of `workspace` into
 * *host_status (0 = no violation, else LIBRASPEC_ST_* bits) and clear it.
 * Returns LIBRASPEC_EDEVICE if the word was non-zero.
 */
int libraspec_get_status(void* workspace, void* stream, int32_t* host_status);

/*
 * Step 1 — drafter confidence (paper Sec. 3.4, Assumption 1: the drafter's
 * confidence q_k stands in for the target's acceptance probability p_k in
 * Algorithm 1).
 *
 * For every sequence b and draft position k:
 *   T      = temperature[b] > 0 ? temperature[b] : 1   (greedy uses T = 1)
 *   m      = max_v draft_logits[b,k,v]
 *   Z      = sum_v exp((draft_logits[b,k,v] - m) / T)
 *   conf[b,k]    = exp((draft_logits[b,k,draft_tokens[b,k]] - m) / T) / Z
 *   dstat[b,k,:] = (m, Z)       (optional; libraspec_accept needs it for
 *                                sampling sequences)
 * draft_logits [B,K,V] f32, draft_tokens [B,K] i32 in [0,V),
 * temperature [B] f32 >= 0, conf [B,K] f32 out, dstat [B,K,2] f32 out or NULL.
 * One pass over the logits (B*K*V*4 bytes), split over CTAs per row.
 */
int libraspec_confidence(const float* draft_logits, const int32_t* draft_tokens, const float* temperature,
                         int B, int K, int V, float* conf, float* dstat, void* workspace, size_t ws_bytes,
                         void* stream);

/*
 * libraspec_confidence on bf16 logits (the 16-bit patterns, as an engine's
 * LM head emits them): each logit widens to fp32 exactly, then the same
 * fp32 / binary64 arithmetic runs on the widened values. Half the bytes:
 * B*K*V*2. draft_logits must be 2-byte aligned; rows whose start is 16-byte
 * aligned with V % 8 == 0 stream in 128-bit loads.
 */
int libraspec_confidence_bf16(const uint16_t* draft_logits, const int32_t* draft_tokens, const float* temperature,
                              int B, int K, int V, float* conf, float* dstat, void* workspace, size_t ws_bytes,
                              void* stream);

/*
 * libraspec_confidence without a workspace, for callers that cannot allocate
 * device memory. The paper has no counterpart: this is an integration
 * variant of Step 1 with the same results (the same kernels run).
 *
 * Scratch is one file-scope __device__ array of the library, sized for
 * B*K <= LIBRASPEC_NOALLOC_MAX_ROWS drafter rows (about 4.2 MB per device);
 * larger calls return LIBRASPEC_EUNSUPPORTED and launch nothing. The call
 * allocates nothing. The first call on a device looks the array's address up
 * (cudaGetSymbolAddress, with that device current, which may load the
 * module): make it before any stream capture. The address is kept per device
 * and CUDA context; a call in a new context on the device (after a
 * cudaDeviceReset, say) looks it up again, and is then a first call too.
 * Each call clears the status
 * word and its row tickets in the array (cudaMemsetAsync on `stream`).
 * Calls share the one array per device, so calls whose executions overlap
 * (other streams, other host threads) race and give undefined results: order
 * them on one stream or synchronise between them.
 *
 * Arguments as for libraspec_confidence. status: device int32 or NULL; when
 * given it receives, in stream order, this call's LIBRASPEC_ST_* bits
 * (0 = no violation; e.g. LIBRASPEC_ST_BAD_TOKEN).
 */
#define LIBRASPEC_NOALLOC_MAX_ROWS 4096
int libraspec_confidence_noalloc(const float* draft_logits, const int32_t* draft_tokens, const float* temperature,
                                 int B, int K, int V, float* conf, float* dstat, int32_t* status, void* stream);

/*
 * Steps 1 and 2 in one launch (Assumption 1's q_k feeding Thm. 4's
 * criterion, Sec. 3.3-3.4): libraspec_confidence, and as soon as the
 * last of a sequence's K rows is done, that CTA selects the sequence's
 * length exactly as libraspec_select_lengths does (same L, same status
 * bits). Arguments as the two calls; K = 0 only selects.
 */
int libraspec_confidence_select(const float* draft_logits, const int32_t* draft_tokens, const float* temperature,
                                const float* cost_table, int B, int K, int V, float* conf, float* dstat, int32_t* L,
                                void* workspace, size_t ws_bytes, void* stream);
int libraspec_confidence_select_bf16(const uint16_t* draft_logits, const int32_t* draft_tokens,
                                     const float* temperature, const float* cost_table, int B, int K, int V,
                                     float* conf, float* dstat, int32_t* L, void* workspace, size_t ws_bytes,
                                     void* stream);

/*
 * Step 2 — LibraSpec length selection (paper Thm. 4, from Thm. 1's
 * ratio comparison; Eq. 2 with negligible drafting cost).
 *
 * With P_j = prod_{k<=j} conf[b,k-1] (prefix acceptance) and
 * E_L = 1 + sum_{j<=L} P_j (expected tokens from verifying L drafts,
 * counting the token verification always emits), extend L -> L+1 while
 *     P_{L+1} * T(L) > (T(L+1) - T(L)) * E_L ,      T(L) = cost_table[L],
 * i.e. while the marginal gain per unit of added verification cost beats
 * the expected speedup E_L / T(L) already reached. L[b] is the first L
 * where the test fails, or K. Computed in binary64; the strict comparison
 * means a tie does not extend.
 * conf [B,K] f32 in [0,1], cost_table [K+1] f32 (each > 0 and finite,
 * else status LIBRASPEC_ST_BAD_COST and L = 0), L [B] i32 out.
 * One warp per sequence; K <= LIBRASPEC_MAX_K.
 */
int libraspec_select_lengths(const float* conf, const float* cost_table, int B, int K, int32_t* L,
                             void* workspace, size_t ws_bytes, void* stream);

/*
 * Step 2, alpha mode — the length search of the paper's Algorithm 1 (its
 * position-wise bounds are Thm. 2 and Thm. 3 with the trade-off weight
 * alpha; Sec. 4 uses alpha = 2.0 for FastdLLM and 2.2 for DFlash / DDTree,
 * block size 16 and d_max = 24 for the latter two).
 *
 * With q_k = conf[b, k-1] (k = 1 .. K, K = d_max) and the current length d,
 *     eps_i = floor(alpha * sum_{j=i}^{d} prod_{k=i}^{j} q_k + i),  i = 1..d,
 *     eps*  = min_i eps_i.
 * Starting from one drafted block, d = block_size and a budget of 0 drafted
 * but unused tokens, while d < K: if eps* <= d then d = eps* and the search
 * stops (the single rollback); otherwise the budget drops by eps* - d,
 * d = min(eps*, K), and when the budget is negative ceil(-budget /
 * block_size) more blocks are drafted (each adds block_size to it).
 * L[b] = d, the number of draft tokens to verify (1 .. K); n_blocks[b] (if
 * not NULL) = the blocks drafted. The search reads only q_1 .. q_d of the
 * current d, so giving all K confidences up front matches drafting blocks
 * on demand. Computed in binary64; eps* above K is clamped to K.
 * conf [B,K] f32 (finite, in [0,1]), L and n_blocks [B] i32, device
 * pointers; 1 <= block_size <= K <= LIBRASPEC_MAX_K, alpha > 0 and finite,
 * else LIBRASPEC_EINVAL. One warp per sequence; no workspace.
 */
int libraspec_select_alpha(const float* conf, int B, int K, int block_size, float alpha, int32_t* L,
                           int32_t* n_blocks, void* stream);

/*
 * Step 3 — block-causal GQA verify attention, one layer (paper Sec. 3.1:
 * the target scores all drafted positions in one forward pass).
 *
 * For sequence b, query head h (kv head h / g, g = Hq / Hkv) and block row
 * t in [0, L[b]]: the block's own keys are already in the cache at
 * positions kv_len[b] .. kv_len[b] + L[b]; row t attends to keys
 * 0 .. kv_len[b] + t:
 *   O[b,t,h,:]  = softmax_s(softmax_scale * Q[b,t,h,:] . Kc[b,h/g,s,:]) Vc[b,h/g,s,:]
 *   lse[b,t,h]  = log sum_s exp(softmax_scale * Q . K)     (natural log)
 * Rows t > L[b] of O and lse are not written.
 * Q, O [B,K+1,Hq,head_dim] bf16; Kc, Vc [B,Hkv,S_cap,head_dim] bf16
 * (16-byte aligned base); kv_len [B] i32 >= 0 with kv_len + L + 1 <= S_cap
 * (else status LIBRASPEC_ST_KV_OVERFLOW, sequence skipped);
 * L [B] i32 in [0,K]; lse [B,K+1,Hq] f32 out or NULL.
 * head_dim in {64, 128}; Hq % Hkv == 0; (K+1) * Hq / Hkv <= 512.
 * Split-KV over a persistent grid with a deterministic in-kernel merge (one
 * cooperative launch; the same kernel as libraspec_verify_attn_layers with
 * one layer).
 */
int libraspec_verify_attn(const uint16_t* Q, const uint16_t* Kc, const uint16_t* Vc, const int32_t* kv_len,
                          const int32_t* L, int B, int K, int Hq, int Hkv, int head_dim, int S_cap,
                          float softmax_scale, uint16_t* O, float* lse, void* workspace, size_t ws_bytes,
                          void* stream);

/*
 * Step 3 over n_layers layers that share kv_len and L (the verified block of
 * every layer of the target), with the same per-layer definition as
 * libraspec_verify_attn. Q, Kc, Vc, O are HOST arrays of n_layers DEVICE
 * pointers; lse is a host array of n_layers device pointers (entries may be
 * NULL) or NULL.
 *
 * Up to LIBRASPEC_ATTN_LAYERS_PER_LAUNCH layers run in one persistent,
 * cooperative kernel launch (more layers take further launches). Layer l+1
 * starts once every CTA has finished layer l (a grid-wide barrier), as it
 * would in a model whose layer l+1 input depends on layer l. Before that
 * barrier the kernel already streams layer l+1's tiles that lie wholly in the
 * cache prefix (keys < kv_len[b], written in earlier rounds); after it, it
 * reads Q, the block's own keys, and merges layer l's split-KV partials. The
 * caller must therefore not let one layer's Q, O or cache rows at or past
 * kv_len[b] be produced by an earlier layer of the same call (they are
 * inputs here), and must not modify the cache prefix during the call.
 * If a wait inside the kernel gives up (LIBRASPEC_ST_TIMEOUT in the status
 * word), re-initialise the workspace (libraspec_workspace_init) before its
 * next use: its barrier counters are then left mid-count.
 */
#define LIBRASPEC_ATTN_LAYERS_PER_LAUNCH 64
int libraspec_verify_attn_layers(const uint16_t* const* Q, const uint16_t* const* Kc, const uint16_t* const* Vc,
                                 int n_layers, const int32_t* kv_len, const int32_t* L, int B, int K, int Hq, int Hkv,
                                 int head_dim, int S_cap, float softmax_scale, uint16_t* const* O, float* const* lse,
                                 void* workspace, size_t ws_bytes, void* stream);

/*
 * libraspec_verify_attn_layers over a paged KV cache (block tables, as
 * serving engines keep it): the same per-layer result as the dense call on
 * the cache the pages describe.
 *   Kp[l], Vp[l]  [n_pages, Hkv, page_size, head_dim] bf16 page pools;
 *   block_table   [B, max_pages] i32: key s of sequence b (cache prefix and
 *                 the verified block alike) is row s % page_size of page
 *                 block_table[b * max_pages + s / page_size] (all layers
 *                 share the table);
 *   page_size     a multiple of 64 (a 64-key tile lies in one page), else
 *                 LIBRASPEC_EUNSUPPORTED; the logical capacity is
 *                 max_pages * page_size (kv_len[b] + L[b] + 1 beyond it:
 *                 LIBRASPEC_ST_KV_OVERFLOW, sequence skipped).
 * A block-table entry read outside [0, n_pages) sets LIBRASPEC_ST_BAD_PAGE
 * and page 0 is read instead (that sequence's rows are then meaningless).
 * The workspace is sized as for the dense call with S_cap = max_pages *
 * page_size. Each CTA reads the page ids of its tile range once per launch.
 */
int libraspec_verify_attn_paged_layers(const uint16_t* const* Q, const uint16_t* const* Kp,
                                       const uint16_t* const* Vp, int n_layers, const int32_t* block_table,
                                       int max_pages, int page_size, int n_pages, const int32_t* kv_len,
                                       const int32_t* L, int B, int K, int Hq, int Hkv, int head_dim,
                                       float softmax_scale, uint16_t* const* O, float* const* lse, void* workspace,
                                       size_t ws_bytes, void* stream);

/*
 * Verification of a draft tree (the tree drafters the paper builds on,
 * Sec. 2, e.g. DDTree, which the paper runs with node budgets of 64 to 512,
 * Appendix C): the block holds the nodes of a tree instead of a chain. N is
 * the node budget (0 <= N <= LIBRASPEC_MAX_TREE_NODES) and takes the place
 * of K in every shape: Q [B, N+1, Hq, d], O and lse likewise. Node 0 is the
 * root (the last accepted token, block position 0); node t in [1, L[b]]
 * (L[b] <= N) sits at block position t, i.e. its query is Q[b, t] and its
 * key / value at cache row kv_len[b] + t, and
 *   parent [B, N+1] i32  parent[b * (N+1) + t] in [0, t) for 1 <= t <= L[b]
 *                        (node numbers are a topological order; other
 *                        entries are not read).
 * Node t attends to the cache prefix (keys < kv_len[b]) and to the keys of
 * its ancestors and itself (the root included): the block-causal mask of
 * libraspec_verify_attn_layers with each row's earlier block positions
 * replaced by its root path. A chain (parent[t] = t - 1, N <= 64) gives
 * exactly the chain call's result. A parent outside [0, t) sets
 * LIBRASPEC_ST_BAD_TREE and is read as the root. Unlike the chain calls,
 * (N+1) * Hq / Hkv query rows per kv head are not capped beyond N's bound.
 * Layers per launch, the ordering rules between layers and the paged-cache
 * rules are those of the chain calls; the workspace is
 * libraspec_workspace_size(B, N, ...). Each call first runs a small kernel
 * that turns the parents into ancestor bit sets (ceil(N / 64) 64-bit words
 * per node, in the workspace).
 */
int libraspec_verify_attn_tree_layers(const uint16_t* const* Q, const uint16_t* const* Kc,
                                      const uint16_t* const* Vc, int n_layers, const int32_t* parent,
                                      const int32_t* kv_len, const int32_t* L, int B, int N, int Hq, int Hkv,
                                      int head_dim, int S_cap, float softmax_scale, uint16_t* const* O,
                                      float* const* lse, void* workspace, size_t ws_bytes, void* stream);
int libraspec_verify_attn_tree_paged_layers(const uint16_t* const* Q, const uint16_t* const* Kp,
                                            const uint16_t* const* Vp, int n_layers, const int32_t* parent,
                                            const int32_t* block_table, int max_pages, int page_size, int n_pages,
                                            const int32_t* kv_len, const int32_t* L, int B, int N, int Hq, int Hkv,
                                            int head_dim, float softmax_scale, uint16_t* const* O,
                                            float* const* lse, void* workspace, size_t ws_bytes, void* stream);

/*
 * Greedy acceptance of a draft tree (the longest root path the target
 * agrees with; the tree drafters of Sec. 2 and Appendix C, verified by the
 * prefix-match rule of Sec. 3.1 along each root path). Row t of target_logits [B, N+1, V] is the target's
 * distribution after node t (tree layout as above; node t >= 1 carries
 * draft_tokens[b * N + t - 1], draft_tokens [B, N]). From the root, the walk
 * moves to the lowest-numbered child of the current node whose token is the
 * argmax of the current node's row (lowest index wins ties), while there is
 * one.
 *   n_accepted [B] i32 out  nodes walked below the root;
 *   last_node  [B] i32 out  the node the walk ends on (may be NULL);
 *   bonus_token [B] i32 out the argmax of that node's row.
 * A chain gives libraspec_accept's greedy result (last_node = n_accepted).
 * Reads target rows 0..L[b] once. A parent outside [0, t) or a token outside
 * [0, V) never matches (LIBRASPEC_ST_BAD_TREE / LIBRASPEC_ST_BAD_TOKEN).
 * Workspace: libraspec_workspace_size(B, N, V, ...). libraspec_accept_tree
 * is the same walk with per-sequence temperatures.
 */
int libraspec_accept_tree_greedy(const float* target_logits, const int32_t* draft_tokens, const int32_t* parent,
                                 const int32_t* L, int B, int N, int V, int32_t* n_accepted, int32_t* last_node,
                                 int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream);
int libraspec_accept_tree_greedy_bf16(const uint16_t* target_logits, const int32_t* draft_tokens,
                                      const int32_t* parent, const int32_t* L, int B, int N, int V,
                                      int32_t* n_accepted, int32_t* last_node, int32_t* bonus_token, void* workspace,
                                      size_t ws_bytes, void* stream);

/*
 * Acceptance of a draft tree at temperature[b] (temperature [B] f32, >= 0;
 * 0 gives the greedy walk above; Sec. 3.1's lossless verification, applied
 * to the candidate children of each node). At the current node the walk draws the
 * target's token x from softmax(row / T) and moves to the lowest-numbered
 * child carrying x while there is one; bonus_token is the last draw. Every
 * emitted token is a draw from the target given the prefix it extends, so
 * the output follows the target's distribution (lossless), and a child is
 * accepted with the target's probability of its token; the drafter's own
 * probabilities are not used (a tree drafter's candidates are chosen, not
 * sampled). Draw at node t: x = argmin_v log2(-ln u_v) - y_v log2(e) / T,
 * u_v the Philox4x32-10 uniform of counter (v >> 2, t, seq_offset + b,
 * 2 + 4 * round_offset), word v & 3, key (seed lo, seed hi) (the generator
 * and uniform mapping of libraspec_accept, purpose 2). The GPU ranks keys
 * in binary32. Every node row 0..L[b] is read once and drawn from (the
 * walk's path is known only after the draws). Shapes, outputs and
 * workspace as for libraspec_accept_tree_greedy.
 */
int libraspec_accept_tree(const float* target_logits, const int32_t* draft_tokens, const int32_t* parent,
                          const int32_t* L, const float* temperature, int B, int N, int V, uint64_t seed,
                          uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted, int32_t* last_node,
                          int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream);
int libraspec_accept_tree_bf16(const uint16_t* target_logits, const int32_t* draft_tokens, const int32_t* parent,
                               const int32_t* L, const float* temperature, int B, int N, int V, uint64_t seed,
                               uint64_t round_offset, uint32_t seq_offset, int32_t* n_accepted, int32_t* last_node,
                               int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream);

/*
 * Row statistics straight from the LM head (steps 1 and 4 without stored
 * logits; the confidence of Assumption 1, the acceptance row statistics of
 * Sec. 3.1): the logits x[r, v] = sum_k H[r, k] W[v, k] are accumulated on
 * the tensor cores and reduced in the GEMM's epilogue.
 *   H [M, Dm] bf16 hidden states (row r = sequence r / rows_per_seq), W [V, Dm]
 *   bf16 head weights, Dm a multiple of 64 (else LIBRASPEC_EUNSUPPORTED),
 *   both 16-byte aligned; temperature [M / rows_per_seq] f32 or NULL (T = 1;
 *   a row at T = 0 takes T = 1, like libraspec_confidence); tokens [M] i32 or
 *   NULL (-1: no token).
 *   row_stat [M, 2] f32 out (m = max_v x, Z = sum_v exp((x_v - m) / T)) or
 *   NULL; row_argmax [M] i32 out (lowest index on ties) or NULL;
 *   token_prob [M] f32 out = exp((x_tok - m) / T) / Z (0 for token -1) or
 *   NULL (needs tokens).
 * With H the drafter rows (rows_per_seq = K) and tokens the drafted tokens,
 * token_prob and row_stat are libraspec_confidence's conf and dstat. Logits
 * are binary32 accumulations of exact bf16 products; partials merge in
 * binary64. A token outside [-1, V) sets LIBRASPEC_ST_BAD_TOKEN (its
 * probability NaN). Reads W once per 128-row tile of H.
 * Workspace: libraspec_lm_head_workspace_size(M, V) bytes (status word and
 * the per-tile partials).
 */
size_t libraspec_lm_head_workspace_size(int M, int V);
int libraspec_lm_head_stats(const uint16_t* H, const uint16_t* W, const float* temperature, int rows_per_seq,
                            const int32_t* tokens, int M, int V, int Dm, float* row_stat, int32_t* row_argmax,
                            float* token_prob, void* workspace, size_t ws_bytes, void* stream);

/*
 * Appending the verified block's keys and values to the caches (the target
 * computes them for the block positions, Sec. 3.1; the verify attention
 * reads them at rows kv_len[b] .. kv_len[b] + T - 1):
 *   kv_new [n_layers, 2, B, Hkv, T, head_dim] bf16 (device, 16-byte aligned):
 *          layer l's keys ([l, 0]) and values ([l, 1]) of block positions
 *          0 .. T-1 (T = K+1 for a chain block, N+1 for a tree);
 *   Kc[l], Vc[l]: HOST arrays of device pointers to the layer caches,
 *          [B, Hkv, S_cap, head_dim] (dense) or page pools [n_pages, Hkv,
 *          page_size, head_dim] with block_table [B, max_pages] (paged: row s
 *          of sequence b at page block_table[b * max_pages + s / page_size],
 *          row s % page_size).
 * Row kv_len[b] + r lands in the cache for r < T; a row past the capacity
 * sets LIBRASPEC_ST_KV_OVERFLOW and a block-table entry outside [0, n_pages)
 * LIBRASPEC_ST_BAD_PAGE (the row is skipped). The workspace holds the status
 * word only (>= 256 bytes). One launch per 64 layers, 16 bytes per thread.
 */
int libraspec_kv_append(const uint16_t* kv_new, uint16_t* const* Kc, uint16_t* const* Vc, int n_layers,
                        const int32_t* kv_len, int B, int T, int Hkv, int head_dim, int S_cap, void* workspace,
                        size_t ws_bytes, void* stream);
int libraspec_kv_append_paged(const uint16_t* kv_new, uint16_t* const* Kp, uint16_t* const* Vp, int n_layers,
                              const int32_t* block_table, int max_pages, int page_size, int n_pages,
                              const int32_t* kv_len, int B, int T, int Hkv, int head_dim, void* workspace,
                              size_t ws_bytes, void* stream);

/*
 * Failure-detection self-test (no counterpart in the paper: it checks the
 * library's own bounded waits). One CTA waits, with the bounded wait that
 * acceptance's draws use for their sequence's decision, until the device
 * word *flag is non-zero, giving up after limit_ns nanoseconds
 * (1 <= limit_ns <= 2e9; the kernels' own waits give up after 2 s). On
 * expiry it raises LIBRASPEC_ST_TIMEOUT in the workspace's status word and
 * returns: the CUDA context stays usable. *observed (device i32) receives 1
 * if the flag was seen, 0 if the wait gave up. flag and observed are
 * caller-owned device pointers (4-byte aligned); the workspace needs only
 * its status word (>= 256 bytes, 256-byte aligned). Enqueues one launch.
 */
int libraspec_selftest_wait(const uint32_t* flag, uint64_t limit_ns, int32_t* observed, void* workspace,
                            size_t ws_bytes, void* stream);

/*
 * Step 4 — acceptance (paper Sec. 3.1; the standard speculative-sampling
 * rule of Leviathan et al. that the paper cites, lossless with respect to
 * the target distribution).
 *
 * Row j of target_logits is the target distribution p_j for draft position
 * j; row L[b] is the bonus row. For each sequence b:
 * temperature[b] == 0 (greedy): accept draft j while argmax_v p_j = x_j
 *   (lowest index wins ties); n = first mismatch or L[b];
 *   bonus = argmax p_n.
 * temperature[b] > 0 (sampling at T): p, q = softmax at T;
 *   for j < L[b], u_j = Philox4x32-10 uniform (purpose 0) and accept iff
 *   u_j < min(1, p_j(x_j) / q_j(x_j)); at the first rejection r the bonus is
 *   drawn from norm(max(0, p_r - q_r)), else from p_{L[b]}, by an
 *   exponential race argmin_v E_v / w_v over purpose-1 uniforms.
 * Generator: key = (seed lo, seed hi); counter = (idx, position,
 *   seq_offset + b, purpose + 4 * round_offset); u = ((w >> 9) + 1/2) 2^-23.
 * target_logits [B,K+1,V] f32, draft_logits [B,K,V] f32, draft_tokens
 * [B,K] i32, conf [B,K] f32 and dstat [B,K,2] f32 from libraspec_confidence
 * (may be NULL when every temperature is 0), L [B] i32, temperature [B] f32;
 * n_accepted [B] i32 out, bonus_token [B] i32 out.
 * Reads target rows 0..L[b] of a greedy sequence once; a sampling sequence
 * reads rows 0..L[b]-1 once, then target row L[b] for its bonus draw or
 * target and drafter rows r for its residual draw. Three launches on the
 * stream: the plan of the row slices (one CTA), the row statistics with the
 * decisions, and the draws.
 */
int libraspec_accept(const float* target_logits, const float* draft_logits, const int32_t* draft_tokens,
                     const float* conf, const float* dstat, const int32_t* L, const float* temperature, int B,
                     int K, int V, uint64_t seed, uint64_t round_offset, uint32_t seq_offset,
                     int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes, void* stream);

/*
 * libraspec_accept on bf16 target and drafter logits (16-bit patterns,
 * widened to fp32 exactly; same arithmetic and generator). conf and dstat
 * come from libraspec_confidence_bf16 on the same drafter logits.
 */
int libraspec_accept_bf16(const uint16_t* target_logits, const uint16_t* draft_logits, const int32_t* draft_tokens,
                          const float* conf, const float* dstat, const int32_t* L, const float* temperature, int B,
                          int K, int V, uint64_t seed, uint64_t round_offset, uint32_t seq_offset,
                          int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                          void* stream);

/*
 * The whole round on one stream (one verification step of Sec. 3.1 with the
 * length chosen per Thm. 4): confidence -> selection -> n_layers verify
 * attention layers -> acceptance. Q, Kc, Vc, O point to HOST arrays of
 * n_layers DEVICE pointers (layer l uses Q[l], Kc[l], Vc[l], O[l]); lse is a
 * host array of n_layers device pointers or NULL. conf, dstat, L are device
 * outputs the round also returns. Same shapes and rules as the four calls.
 */
int libraspec_verify_round(const float* draft_logits, const int32_t* draft_tokens, const float* temperature,
                           const float* cost_table, const float* target_logits, const uint16_t* const* Q,
                           const uint16_t* const* Kc, const uint16_t* const* Vc, uint16_t* const* O,
                           float* const* lse, int n_layers, const int32_t* kv_len, int B, int K, int V, int Hq,
                           int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                           uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat, int32_t* L,
                           int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                           void* stream);

/* libraspec_verify_round on bf16 drafter and target logits (the _bf16 forms
 * of steps 1 and 4; selection and attention unchanged). */
int libraspec_verify_round_bf16(const uint16_t* draft_logits, const int32_t* draft_tokens, const float* temperature,
                                const float* cost_table, const uint16_t* target_logits, const uint16_t* const* Q,
                                const uint16_t* const* Kc, const uint16_t* const* Vc, uint16_t* const* O,
                                float* const* lse, int n_layers, const int32_t* kv_len, int B, int K, int V, int Hq,
                                int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                                uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat, int32_t* L,
                                int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                                void* stream);

/*
 * The round fed from pinned host memory with the copies overlapped: three
 * host parts (host_parts[i], part_bytes[i] bytes, pinned) are copied to
 * dev_parts[i] on copy_stream, in order: part 0 must hold the drafter block
 * (draft_logits, draft_tokens, temperature, cost_table), part 1 the layers'
 * Q and kv_new, part 2 target_logits (the typed pointers below point into
 * the device parts). On `stream`, confidence and selection wait for part 0;
 * libraspec_kv_append of kv_new ([n_layers, 2, B, Hkv, K+1, head_dim]) and
 * the attention layers wait for part 1; acceptance waits for part 2; then
 * n_accepted and bonus_token are copied to n_accepted_host / bonus_host
 * (pinned, B entries each). copy_stream first waits for the work already on
 * `stream`, so a round never overwrites buffers an earlier one still reads.
 * The generator arguments travel with part 2: the call writes seed,
 * round_offset and seq_offset to rng_host[0..2] (pinned, inside host part
 * 2, 8-byte aligned) and acceptance reads them at rng_dev (the same bytes in
 * device part 2). The first call with a given set of buffers and shapes
 * runs eagerly; the second captures the round on `stream` as one CUDA graph
 * (per thread) and later calls with the same set replay it, whatever the
 * seed and offsets. The call returns after enqueuing; synchronise `stream`
 * before reading the host results or rewriting the host parts. Other
 * arguments as libraspec_verify_round (lse is not produced).
 */
int libraspec_verify_round_staged(const void* const* host_parts, void* const* dev_parts, const size_t* part_bytes,
                                  void* copy_stream, const uint16_t* kv_new, uint64_t* rng_host,
                                  const uint64_t* rng_dev, int32_t* n_accepted_host, int32_t* bonus_host,
                                  const float* draft_logits, const int32_t* draft_tokens, const float* temperature,
                                  const float* cost_table, const float* target_logits,
                                  const uint16_t* const* Q, uint16_t* const* Kc, uint16_t* const* Vc,
                                  uint16_t* const* O, int n_layers, const int32_t* kv_len, int B, int K, int V,
                                  int Hq, int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                                  uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat, int32_t* L,
                                  int32_t* n_accepted, int32_t* bonus_token, void* workspace, size_t ws_bytes,
                                  void* stream);
int libraspec_verify_round_staged_bf16(const void* const* host_parts, void* const* dev_parts,
                                       const size_t* part_bytes, void* copy_stream, const uint16_t* kv_new,
                                       uint64_t* rng_host, const uint64_t* rng_dev, int32_t* n_accepted_host,
                                       int32_t* bonus_host, const uint16_t* draft_logits,
                                       const int32_t* draft_tokens, const float* temperature,
                                       const float* cost_table, const uint16_t* target_logits,
                                       const uint16_t* const* Q, uint16_t* const* Kc, uint16_t* const* Vc,
                                       uint16_t* const* O, int n_layers, const int32_t* kv_len, int B, int K, int V,
                                       int Hq, int Hkv, int head_dim, int S_cap, float softmax_scale, uint64_t seed,
                                       uint64_t round_offset, uint32_t seq_offset, float* conf, float* dstat,
                                       int32_t* L, int32_t* n_accepted, int32_t* bonus_token, void* workspace,
                                       size_t ws_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* LIBRASPEC_H */
