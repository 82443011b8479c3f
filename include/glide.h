/*
 * glide.h -- C ABI of libglide: the KV-cache attention hot path of
 * GliDe-with-CaPE speculative decoding (arXiv 2402.02082) on GB300 (sm_103a).
 *
 * Three calls make up one speculative round for one target layer:
 *
 *   glide_cross_attn   the GliDe draft model's cross-attention: a draft query
 *                      per (sequence, head) attends to every cached key/value
 *                      of the frozen target model (Section 3.1, the hd_j
 *                      equation; no mask at inference).
 *   tree_verify_attn   the target's parallel verification of the linearized
 *                      expanded proposal: n tree queries attend to the cached
 *                      prefix and to their own ancestors and themselves
 *                      (the CaPE mask of Section 3.2 is this mask on CaPE's
 *                      trees).
 *   tree_accept        greedy acceptance on the token tree (Section 2): the
 *                      deepest node whose whole root path the target's argmax
 *                      reproduces, and the free bonus token.
 *
 * Two more calls close the round around them:
 *
 *   cape_expand        CaPE's confidence-aware proposal expansion (Section
 *                      3.2): from the draft's distributions, the proposal
 *                      tokens, the expansion sets and the linearized tree that
 *                      tree_verify_attn and tree_accept take.
 *   glide_kv_compact   the cache update after acceptance (Section 3.1): the
 *                      accepted path's keys/values become contiguous rows.
 *   spec_sample_accept speculative-sampling acceptance of a chain proposal
 *                      (Section 2's other acceptance strategy, used for GliDe
 *                      alone in Section 4.1), with caller-supplied uniforms.
 *
 * Conventions shared by all calls
 * -------------------------------
 * - Every tensor pointer is a DEVICE pointer owned by the caller; the library
 *   allocates nothing and keeps no state between calls.  All work is enqueued
 *   on `stream` (a cudaStream_t; NULL means the legacy default stream) and is
 *   asynchronous: a returned GLIDE_OK means "launched", not "finished".
 * - Layouts are dense, row-major, no padding:
 *     queries   [B, nq, H, D]          (nq = 1 for cross-attention, n for the tree)
 *     K, V      [B, H_kv, S_cap, D]    one contiguous S_cap x D slab per (b, cached
 *                                      head); H_kv = H is multi-head attention, fewer
 *                                      cached heads is grouped-query attention: query
 *                                      head h reads cached head h / (H / H_kv)
 *     out       [B, nq, H, D] fp32
 *     kv_len    [B] int32              cached prefix length of each sequence
 *     parent    [B, n] int32           linearized tree: -1 for a root, else an
 *                                      earlier node (parent[i] < i)
 * - The tree's own keys/values must already be written at cache rows
 *   kv_len[b] .. kv_len[b]+n-1, in linearized order (node j at row kv_len[b]+j).
 *   Rows at and beyond kv_len[b]+n are never read and may hold anything.
 * - Rotary embedding (if any) is applied by the caller before the call.
 * - Host-side checks run before anything is launched; a bad argument returns
 *   GLIDE_ERR_INVALID and touches no memory.  Device-resident values
 *   (kv_len, parent, draft tokens) cannot be checked on the host: the kernels
 *   clamp them into range, so bad values give meaningless results but never an
 *   out-of-bounds access.
 * - Workspace: caller-allocated device memory of at least the size the
 *   matching *_workspace_bytes function returns, ZERO-FILLED before its first
 *   use.  It holds a status word, arrival counters (and, for tree_accept,
 *   argmax slots) that must start at zero, and scratch for split partial
 *   results.  Every successful call returns the words that must start at zero
 *   to zero, so one buffer can be reused across calls on the same stream.
 *   Calls that run concurrently on different streams need separate
 *   workspaces.
 * - Kernel waits are bounded.  A kernel that gives up waiting records
 *   GLIDE_ERR_DEVICE_TIMEOUT in its workspace; glide_read_device_status reads
 *   and clears it.
 */
#ifndef GLIDE_H
#define GLIDE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define GLIDE_ABI_VERSION 2

typedef struct CUstream_st* glide_stream_t;

typedef enum {
  GLIDE_OK = 0,
  GLIDE_ERR_INVALID = 1,        /* bad argument found on the host; nothing launched        */
  GLIDE_ERR_UNSUPPORTED = 2,    /* well-formed but outside the supported shapes            */
  GLIDE_ERR_CUDA = 3,           /* a CUDA runtime call or kernel launch failed             */
  GLIDE_ERR_DEVICE_TIMEOUT = 4  /* a kernel gave up a bounded wait (device status only)    */
} glide_status;

typedef enum { GLIDE_BF16 = 0, GLIDE_F32 = 1 } glide_dtype;

/* flags */
#define GLIDE_FLAG_FORCE_FMA 1u   /* tree_verify_attn: use the CUDA-core kernel even where the
                                     tensor-core kernel applies (testing and comparison)     */
#define GLIDE_FLAG_TILE64 2u      /* grouped-query slabs and slabs of more than 64 query rows:
                                     use the 64-row tensor-core kernel rather than the 128-row
                                     one (testing and comparison)                            */

typedef struct {
  int32_t B;          /* sequences in the batch, 1..1024                                   */
  int32_t H;          /* query heads (of the target layer), >= 1                            */
  int32_t D;          /* head dimension d_k: 64 or 128                                     */
  int32_t S_cap;      /* rows of each (b, h) slab of the K/V cache                          */
  glide_dtype dtype;  /* element type of queries, K and V                                   */
  float scale;        /* softmax scale; 0 means 1/sqrt(D) (Section 3.1)                     */
  uint32_t flags;     /* GLIDE_FLAG_* bits                                                  */
  int32_t max_ctas;   /* upper bound on the CTAs of one attention launch; 0 = automatic     */
  int32_t H_kv;       /* cached (key/value) heads; 0 means H.  H % H_kv == 0: each run of
                         H / H_kv consecutive query heads shares one cached head (grouped-
                         query attention, as in Mistral-7B: 32 query over 8 cached heads).
                         tree_verify_attn needs n * H / H_kv <= 256 (query rows per
                         cached head; with bf16 and H / H_kv dividing 128, grouped-query
                         slabs are served in row tiles of 128, else in tiles of 64).      */
} glide_attn_desc;

/* Version of this ABI (GLIDE_ABI_VERSION of the built library). */
int32_t glide_abi_version(void);

/* Static, human-readable name of a status code. */
const char* glide_status_str(glide_status status);

/* Bytes of workspace that glide_cross_attn (n_queries = 1) and
 * tree_verify_attn (n_queries = n) need for this descriptor; 0 if the
 * descriptor is invalid.  A buffer sized for the largest n serves both. */
size_t glide_attn_workspace_bytes(const glide_attn_desc* desc, int32_t n_queries);

/* Bytes of workspace that tree_accept needs for B trees of n nodes. */
size_t glide_accept_workspace_bytes(int32_t B, int32_t n);

/*
 * GliDe cross-attention (Section 3.1):
 *   out[b,0,h,:] = SoftMax(q[b,0,h,:] . K[b,h,k,:] * scale, k < kv_len[b]) V[b,h,k,:]
 * q_draft [B,1,H,D] (desc->dtype), K_cache/V_cache [B,H,S_cap,D] (desc->dtype),
 * kv_len [B] int32 on the device, clamped to [0, max_kv_len]; a sequence with
 * kv_len 0 has nothing to attend to and gets zeros.
 * max_kv_len: host-side upper bound of kv_len, 1 <= max_kv_len <= S_cap.
 * out [B,1,H,D] fp32.
 */
glide_status glide_cross_attn(const glide_attn_desc* desc, const void* q_draft,
                              const void* K_cache, const void* V_cache,
                              const int32_t* kv_len, int32_t max_kv_len, float* out,
                              void* workspace, size_t workspace_bytes, glide_stream_t stream);

/*
 * Tree verification attention (Section 3.2, CaPE verification mask; the
 * ancestor-or-self rule of the token-tree verifier it borrows):
 *   out[b,i,h,:] = SoftMax over k in A_i of (q[b,i,h,:] . K[b,h,k,:] * scale) V[b,h,k,:]
 *   A_i = {0 .. kv_len[b]-1} U {kv_len[b] + j : j = i or j an ancestor of i}
 * q_tree [B,n,H,D], 1 <= n <= 64; parent_idx [B,n] int32 on the device (a forest
 * in topological order; an entry outside [-1, i) is treated as -1).
 * kv_len [B] on the device, clamped to [0, max_kv_len]; 0 <= max_kv_len and
 * max_kv_len + n <= S_cap.  out [B,n,H,D] fp32.
 */
glide_status tree_verify_attn(const glide_attn_desc* desc, const void* q_tree, int32_t n,
                              const int32_t* parent_idx, const void* K_cache,
                              const void* V_cache, const int32_t* kv_len, int32_t max_kv_len,
                              float* out, void* workspace, size_t workspace_bytes,
                              glide_stream_t stream);

/*
 * Greedy tree acceptance (Section 2, greedy "speculative decoding" rule, on
 * the token tree of Section 3.2):
 *   a_i  = argmax_v target_logits[b,i,v] (lowest v among equal maxima; -0 == +0)
 *   node c >= 1 with parent p is accepted iff draft_tokens[b,c] == a_p and p is
 *   accepted; node 0 (x_t, the last accepted token) is always accepted.
 *   Result: the accepted node of greatest depth (lowest index among equals).
 * draft_tokens [B,n] int32, parent_idx [B,n] int32 (node 0 the root, every other
 * parent earlier; an entry outside [0, i) makes node i unreachable),
 * target_logits [B,n,V] fp32, finite.  1 <= n <= 64, 1 <= V.
 * Outputs: path [B,n] int32 = root..node node indices, -1 padded;
 * len [B] int32 = depth of that node (accepted proposal tokens);
 * bonus [B] int32 = a_node, the target's free next token.
 */
glide_status tree_accept(const int32_t* draft_tokens, const int32_t* parent_idx,
                         const float* target_logits, int32_t B, int32_t n, int32_t V,
                         int32_t* path, int32_t* len, int32_t* bonus,
                         void* workspace, size_t workspace_bytes, glide_stream_t stream);

/* Bytes of workspace that cape_expand needs for B proposals of gamma
 * positions over a vocabulary of V; 0 if the sizes are out of range. */
size_t glide_cape_workspace_bytes(int32_t B, int32_t gamma, int32_t V);

/*
 * CaPE confidence-aware proposal expansion (Section 3.2; the fixed-size
 * variant of Section 4's ablation with fixed_k >= 0):
 *   for each sequence b and position i = 1..gamma, from the draft's
 *   distribution probs[b,i-1,:]:
 *     x_{t+i} = the most probable token, p_i = its probability (conf[b,i-1]);
 *     K_i = S(p_i) = 7, 5, 3, 1 for p_i in (0,0.3], (0.3,0.6], (0.6,0.8], (0.8,1]
 *           (exact comparison of the fp32 value with the decimal thresholds;
 *           p_i <= 0 gives 7, p_i > 1 gives 1), or fixed_k; at most V-1;
 *     X_i  = the K_i most probable tokens other than x_{t+i}.
 *   Ranking: higher probability first, then the lower token id; -0 == +0.
 *   Cap: the proposal and the sets hold at most max_tokens tokens (x_t not
 *   counted); when the sets overflow, the expansion tokens of lowest
 *   probability are dropped first (equal probabilities: the later position,
 *   then the later rank), so every kept set is still the top of its position.
 * Output: the linearized tree of n_out = 1 + max_tokens node slots per sequence,
 *   draft_tokens [B, n_out], parent_idx [B, n_out] int32:
 *     node 0          = root_token[b] (x_t), parent -1;
 *     node i, 1..gamma = x_{t+i}, parent i-1;
 *     then each position's kept set in position order, best first, every
 *     token with parent i-1 (a sibling of x_{t+i});
 *     unused slots n_nodes[b] .. n_out-1: token -1, parent 0 (a leaf that
 *     acceptance never takes, since no argmax equals -1).
 *   n_nodes [B] int32 = 1 + gamma + kept expansion tokens.
 *   conf [B, gamma] fp32 = p_i (a zero is reported as +0), or NULL.
 *   The ancestor-or-self mask of this tree is the CaPE mask of Section 3.2, so
 *   the arrays go to tree_verify_attn and tree_accept as they are (n = n_out).
 * probs [B, gamma, V] fp32 on the device, finite, 16-byte aligned;
 * root_token [B] int32 on the device.  1 <= gamma <= max_tokens <= 63;
 * fixed_k = -1 for S(p), or 0 .. 7 (larger: GLIDE_ERR_UNSUPPORTED).
 */
glide_status cape_expand(const float* probs, const int32_t* root_token, int32_t B, int32_t gamma,
                         int32_t V, int32_t max_tokens, int32_t fixed_k, int32_t* draft_tokens,
                         int32_t* parent_idx, int32_t* n_nodes, float* conf, void* workspace,
                         size_t workspace_bytes, glide_stream_t stream);

/*
 * Cache update after acceptance (Section 3.1: the target keeps the cache
 * entries of the accepted tokens and discards the rejected ones), in place,
 * for n_layers layers at once:
 *   for every layer, sequence b and head h, and k = 0 .. len[b]:
 *     K[b,h,kv_len[b]+k,:] <- K[b,h,kv_len[b]+path[b,k],:]   (same for V)
 *   new_kv_len[b] = kv_len[b] + len[b] + 1.
 * This keeps x_t (node 0) and the accepted proposal tokens, in path order;
 * the new bonus token has no entry yet (it is node 0 of the next tree).
 * Every other row keeps its contents.
 * desc: B, H, D, S_cap and dtype of one layer's cache (scale, flags and
 * max_ctas are ignored).  K_cache/V_cache: layer 0 of [n_layers][B,H,S_cap,D];
 * layer l starts layer_stride ELEMENTS after layer l-1 (layer_stride >=
 * B*H*S_cap*D and a multiple of 16 bytes when n_layers > 1; ignored when 1).
 * kv_len [B] (clamped to [0, S_cap-n]), path [B,n] (root-first node indices
 * as tree_accept writes them, clamped to [0, n)), len [B] (clamped to
 * [0, n-1]) are int32 on the device; 1 <= n <= 64, n <= S_cap.
 * new_kv_len [B] int32 on the device and not the kv_len buffer (the kernel
 * reads kv_len while it writes new_kv_len).  No workspace.
 * Correct for every path that tree_accept produces (node indices along a root
 * path are increasing); other paths stay in bounds but give unspecified rows.
 */
glide_status glide_kv_compact(const glide_attn_desc* desc, int32_t n_layers, int64_t layer_stride,
                              void* K_cache, void* V_cache, const int32_t* kv_len, int32_t n,
                              const int32_t* path, const int32_t* len, int32_t* new_kv_len,
                              glide_stream_t stream);

/* Bytes of workspace that spec_sample_accept needs for B proposals of gamma tokens. */
size_t glide_sample_workspace_bytes(int32_t B, int32_t gamma);

/*
 * Speculative-sampling acceptance of a chain proposal (the speculative
 * sampling named in Section 2 and used for GliDe alone in Section 4.1; its
 * outputs are distributed as the target model's own samples):
 *   p_T,i = SoftMax(target_logits[b,i,:]) for i = 0..gamma (temperature 1);
 *   position i (0-based) accepts draft_tokens[b,i] = x when
 *     uniforms[b,i] * draft_probs[b,i,x] < p_T,i(x);
 *   n_accepted[b] = the number of positions before the first rejection (gamma
 *   if none);
 *   next_token[b] = a draw from max(0, p_T,n - draft_probs[b,n,:]) if n < gamma,
 *   else from p_T,gamma: the first token whose running weight exceeds
 *   uniforms[b,gamma] * (total weight).  (If the residual weight sums to 0 in
 *   fp32 the draw is from p_T,n.)
 * The accepted tokens are draft_tokens[b,0..n-1], followed by next_token[b].
 * The kernel computes in fp32; a result can differ from exact arithmetic only
 * where a product u * p_D(x) or v * total lies within rounding of its threshold.
 * draft_tokens [B,gamma] int32 (clamped to [0,V)), draft_probs [B,gamma,V] fp32,
 * target_logits [B,gamma+1,V] fp32 finite and 16-byte aligned, uniforms
 * [B,gamma+1] fp32 in [0,1), all on the device.  1 <= gamma <= 63, 1 <= V.
 * Outputs n_accepted [B], next_token [B] int32.
 */
glide_status spec_sample_accept(const int32_t* draft_tokens, const float* draft_probs,
                                const float* target_logits, const float* uniforms, int32_t B,
                                int32_t gamma, int32_t V, int32_t* n_accepted, int32_t* next_token,
                                void* workspace, size_t workspace_bytes, glide_stream_t stream);

/* Bytes of workspace that glide_block_cross_attn needs for sequences of T
 * positions; 0 if the descriptor or T is out of range. */
size_t glide_block_attn_workspace_bytes(const glide_attn_desc* desc, int32_t T);

/*
 * The draft's cross-attention at training time under the block-wise mask
 * (Section 3.1, "Block-wise Attention Mask"): the query of every position j of
 * a training sequence attends to the target's cached keys/values of the
 * positions k with block(j) > block(k), block(x) = x / L -- the blocks before
 * j's own, i.e. keys 0 .. L*(j/L)-1 -- so that training sees the delayed cache
 * that speculation sees:
 *   out[b,j,h,:] = SoftMax over k < L*(j/L) of (q[b,j,h,:] . K[b,hk,k,:] * scale) V[b,hk,k,:]
 * with hk = h / (H / H_kv).  Positions of the first block (nothing to attend
 * to) and positions at or past seq_len[b] get zeros.
 * q [B,T,H,D] bf16; K_cache/V_cache [B,H_kv,S_cap,D] bf16 holding the target's
 * keys/values of positions 0..T-1; seq_len [B] int32 on the device (clamped to
 * [0,T]); out [B,T,H,D] fp32, every element written (no pre-zeroing needed).
 * 1 <= T <= S_cap, L >= 1.  fp32 inputs, B*T or B*H_kv*S_cap beyond 2^31 - 128
 * rows (32-bit TMA coordinates), or B*H*ceil(T/256) position-tile pairs plus the
 * CTA count beyond 2^31 - 1: GLIDE_ERR_UNSUPPORTED.  The workspace holds only the
 * device status word (glide_block_attn_workspace_bytes).
 */
glide_status glide_block_cross_attn(const glide_attn_desc* desc, const void* q, int32_t T, int32_t L,
                                    const void* K_cache, const void* V_cache, const int32_t* seq_len,
                                    float* out, void* workspace, size_t workspace_bytes,
                                    glide_stream_t stream);

/*
 * glide_cross_attn for callers that cannot allocate device memory when they
 * call (the paper has no counterpart; this is a deployment entry point).
 * Examples: an engine plugin whose enqueue path must not allocate because the
 * host engine owns and budgets all device memory, or a serving loop that has
 * given nearly all of HBM to its KV cache and bans allocator calls on its
 * per-token path.  Same arguments and result as glide_cross_attn, minus the
 * workspace: the scratch lives in one fixed 32 MiB array inside the library,
 * held on every GPU that loads the library until the process exits.
 * - Shapes whose workspace (glide_attn_workspace_bytes(desc, 1)) exceeds
 *   32 MiB are rejected with GLIDE_ERR_UNSUPPORTED (B*H up to 7035 for D = 128,
 *   14835 for D = 64).
 * - Every call looks up the array's device address in the current device's
 *   context (so a context created again after cudaDeviceReset is served
 *   correctly); the first call on a device also loads the library's device
 *   code there, so make that first call before any stream capture.  `stream`
 *   must belong to the current device.
 * - Every call first clears the counters that must start at zero, then reuses
 *   the array, so calls that overlap on the GPU (other streams, other host
 *   threads without ordering) race on it: serialize them.
 * - A bounded wait that ran out (GLIDE_ERR_DEVICE_TIMEOUT) is recorded in the
 *   array's status word, which calls do not clear: read it with
 *   glide_noalloc_read_device_status.
 * - Allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 */
glide_status glide_cross_attn_noalloc(const glide_attn_desc* desc, const void* q_draft,
                                      const void* K_cache, const void* V_cache,
                                      const int32_t* kv_len, int32_t max_kv_len, float* out,
                                      glide_stream_t stream);

/*
 * The device status of glide_cross_attn_noalloc (no counterpart in the paper):
 * waits for `stream`, then returns the status recorded in the fixed array of
 * the current device since it was last read (GLIDE_OK or
 * GLIDE_ERR_DEVICE_TIMEOUT) and clears it, as glide_read_device_status does for
 * a caller's workspace.  Allocates nothing.
 */
glide_status glide_noalloc_read_device_status(glide_stream_t stream);

/*
 * Device address of the fixed array of glide_cross_attn_noalloc on the current
 * device (no counterpart in the paper), for diagnostics: e.g. to point
 * glide_selftest_wait_timeout at it.  The contents belong to the library.
 * Returns GLIDE_ERR_INVALID for a null pointer, GLIDE_ERR_CUDA if the lookup
 * fails.  Allocates nothing.
 */
glide_status glide_noalloc_scratch(void** device_ptr);

/*
 * Host-side check of a parent array (HOST memory, [B,n]): every entry is -1 or
 * in [0, i).  With require_root0 != 0 (the tree_accept convention) node 0 must
 * be the only root.  Returns GLIDE_OK or GLIDE_ERR_INVALID.
 */
glide_status glide_validate_tree(const int32_t* parent_idx_host, int32_t B, int32_t n,
                                 int32_t require_root0);

/*
 * Self-test of the failure path (no counterpart in the paper): launches one
 * small kernel whose bounded waits on a barrier that nothing completes give up
 * after limit_us microseconds (1 .. 2,000,000), record GLIDE_ERR_DEVICE_TIMEOUT
 * in `workspace` (any attention or acceptance workspace) and release the
 * kernel's other waiter, as every kernel of the library does when a wait runs
 * out.  glide_read_device_status then returns that code and clears it.  The
 * GPU neither faults nor hangs, and the context stays usable.
 */
glide_status glide_selftest_wait_timeout(void* workspace, uint32_t limit_us, glide_stream_t stream);

/*
 * Waits for `stream`, then returns the status the kernels recorded in
 * `workspace` (GLIDE_OK or GLIDE_ERR_DEVICE_TIMEOUT) and clears it.  Works on
 * attention and acceptance workspaces alike.
 */
glide_status glide_read_device_status(void* workspace, glide_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* GLIDE_H */
