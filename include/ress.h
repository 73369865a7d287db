/*
 * ress.h -- C ABI of the ReSS (Residual-Restoring Sparse Attention) hot path on GB300.
 *
 * One sparsified global-attention layer of a 3D vision transformer:
 *   ress_score       block pooling, pooled attention map, block drift scores and the
 *                    initial selection (Sec. 4.1-4.2, Eq. 1, 5-9)
 *   ress_restore     R budget-neutral restoration rounds with track-best and the kept-block
 *                    lists (Sec. 4.3, Eq. 10-17)
 *   ress_sparse_attn exact attention over the kept 64x64 blocks (Sec. 3 step (3))
 *   ress_forward     the three in order on one stream (ress_forward_host: from and to
 *                    host buffers, the output copied back while the attention runs)
 * Also: the ablation variants of the selection (ress_score_variant, ress_restore_variant),
 * the residual update and token-level drift (ress_out_proj, ress_token_drift), an
 * allocation-free attention entry point, and a bounded-wait self-test of the error path.
 *
 * Conventions shared by every call
 *   - Pointers named "device" point to GPU memory owned by the caller; the library never
 *     allocates, frees or retains memory.  Host pointers are read before the call returns.
 *   - bf16 tensors are passed as uint16_t bit patterns.  Q, K, V and O are [N, H, 64]
 *     row-major (token, head, channel): one token is H*128 contiguous bytes.  Their base
 *     addresses must be 16-byte aligned.
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and validates all host-visible arguments before it launches anything.  On a
 *     validation error nothing is launched.
 *   - Return value: RESS_OK (0) or a negative ress_status code; ress_last_error() gives a
 *     message for the calling thread.  No C++ exception crosses the ABI.
 *   - Device-side failures (a bounded wait that gave up, an out-of-range index in a
 *     caller-built CSR) are recorded in a status word inside the workspace; read it with
 *     ress_status() after the stream work completes.  Kernels never trap.
 *   - Fixed constants: head_dim = 64, block = 64 (64x64 block grid), eps = 1e-4 (Eq. 7).
 *   - Results are deterministic: the same inputs give the same bits (Appendix B.4).
 */
#ifndef RESS_H
#define RESS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RESS_ABI_VERSION 6
#define RESS_HEAD_DIM 64
#define RESS_BLOCK 64
#define RESS_MAX_HEADS 32
#define RESS_MAX_BLOCKS 4096 /* key blocks per sequence: 262144 tokens */

typedef enum {
  RESS_OK = 0,
  RESS_EINVAL = -1,       /* null/misaligned pointer, inconsistent sizes or budgets      */
  RESS_EWORKSPACE = -2,   /* workspace or output buffer smaller than required            */
  RESS_EUNSUPPORTED = -3, /* head_dim != 64, block != 64, too many heads or blocks        */
  RESS_ECUDA = -4,        /* a CUDA runtime call or kernel launch failed                  */
  RESS_ETIMEOUT = -5,     /* a bounded device-side wait gave up (status word)             */
  RESS_EDEVICE = -6       /* a device-side argument check failed (status word)            */
} ress_status_code;

/* Shape of one global-attention layer.  Special tokens (camera/register) are the last
 * n_special tokens of the sequence (Sec. 3, "excluded from sparsification"): key blocks
 * that contain any of them are always kept, query blocks that contain any of them attend
 * densely.  The remaining key blocks form the candidate set P of Sec. 4.1, of size
 * (n_tokens - n_special) / 64 (rounded down). */
typedef struct {
  int32_t n_tokens;  /* N >= 1                                                    */
  int32_t n_heads;   /* H, 1..RESS_MAX_HEADS                                      */
  int32_t head_dim;  /* d_h, must be 64                                           */
  int32_t block;     /* block size, must be 64                                    */
  int32_t n_special; /* trailing special tokens, 0..N-1                           */
  int32_t d_model;   /* d: rows of the output projection W_o ([d, H*64])          */
  int32_t q_block;   /* query block size: 64 (0 means 64) or 128, the paper's own grid
                        of 128-token query blocks over 64-token key blocks (Appendix F).
                        Selection rows, CSR rows, J_best and drop masks are per (head,
                        query block): H * nq rows, nq = ceil(N / q_block); query blocks
                        that contain special tokens attend densely.                  */
} ress_dims;

/* Byte offsets of the arrays inside the workspace (for inspection and tests).  All
 * arrays are float32 unless noted; row strides are in elements. */
typedef struct {
  int64_t status;      /* uint32 status word (first device-side error, sticky)          */
  int64_t counter;     /* uint32 tile-scheduler counters of the attention kernel        */
  /* Rows i are the nq query blocks, columns j the nb key blocks (nq = nb on the 64 grid). */
  int64_t qbar, kbar, vbar, ztil; /* [H, nq, 64] q_bar; [H, nb, 64] k_bar, V_bar, z~_j = F_h V_j */
  int64_t ytil, gtil;  /* [H, nq, 64] y~_i = F_h v_bar_i (Eq. 1); g~ = F_h g (Eq. 10)    */
  int64_t P, q, t;     /* [H, nq, ld] pooled P_ij, q_ij = ||F_h e_ij||^2 (Eq. 9), gains;
                          t doubles as the attention kernel's pair-list scratch            */
  int64_t K, G, J, Jbest, J0; /* [H, nq] remaining mass, G, J of Eq. 12                  */
  int64_t dmask, bmask; /* uint32 [H, nq, words] current and best drop sets (bit j)      */
  int64_t plen;        /* int32 [H, ceil(nb/2)] lengths of the attention items' lists       */
  int64_t asplit;      /* bf16 [3, H, nq, 64]: row operand as three bf16 terms (hi, mid, lo):
                          q_bar, then y~, then g~ (tensor-core products)                   */
  int64_t ksplit, zsplit; /* bf16 [3, H, nb, 64]: k_bar and z~ as three bf16 terms          */
  int64_t cdot, ny, nz;   /* float [H, nq]: y~_i . g~_i, ||y~_i||^2; [H, nb]: ||z~_j||^2    */
  int64_t lstat;       /* float2 [H, nq, ceil(nb/128)]: per 128-block slice of a row of
                          pooled logits, its max and sum of exp(logit - max)               */
  int64_t kcount;      /* int32 [H, nq]: key blocks kept by each candidate query row       */
  int64_t prow;        /* int32 [H, ceil(nb/2)]: query blocks a | b << 16 of each attention
                          item that ress_forward pairs by the overlap of their kept lists   */
  int64_t ld;          /* row stride of P, q, t                                          */
  int64_t words;       /* uint32 words per drop-set bitmask = ceil(nb / 32)              */
  int64_t total;       /* bytes                                                          */
} ress_ws_layout;

/* Message describing the last error returned on the calling thread ("" if none). */
const char* ress_last_error(void);
int32_t ress_abi_version(void);

/* Number of kernels this library has enqueued since it was loaded, over all calls, streams
 * and threads of the process (host-side count, incremented at each launch).  For telemetry
 * and benchmarks: the difference around a sequence of calls is the number of kernels they
 * put on the GPU.  No paper counterpart. */
uint64_t ress_kernel_launches(void);

/* Number of key blocks nb = ceil(N / 64) and candidate blocks |P|; -1 on bad dims. */
int32_t ress_num_blocks(const ress_dims* dims);
int32_t ress_num_candidates(const ress_dims* dims);
/* Query blocks nq = ceil(N / q_block) (the rows of the selection and of the CSR), and the
 * candidate query blocks, floor((N - n_special) / q_block), that are sparsified. */
int32_t ress_num_query_blocks(const ress_dims* dims);
int32_t ress_num_query_candidates(const ress_dims* dims);

/* Workspace needed by ress_score / ress_restore / ress_sparse_attn / ress_forward
 * (0 on invalid dims).  The same workspace serves every call on that layer shape; it
 * must be 256-byte aligned and must not be shared by calls that may overlap on the GPU. */
size_t ress_workspace_bytes(const ress_dims* dims);
int ress_workspace_layout(const ress_dims* dims, ress_ws_layout* out);

/* Entries of col_idx that ress_restore writes for the budgets c_h (host array [H]):
 * every candidate query block keeps c_h + (nb - |P|) key blocks, every other query block
 * keeps all nb.  -1 on invalid arguments. */
int64_t ress_csr_capacity(const ress_dims* dims, const int32_t* c_h_host);

/* Eq. 8 at model-load time.  W_o: device bf16 [d_model, H*64] (Linear.weight layout,
 * out x in; head h owns columns 64h..64h+63, i.e. W_O^h).  F: device float32 [H, 64, 64]
 * receives an upper-triangular F_h with F_h^T F_h = M_h = W_O^h^T W_O^h (Cholesky factor,
 * computed in float64; a zero pivot of a rank-deficient M_h yields a zero row).  The
 * scoring kernels use ||F_h e||^2 = e^T M_h e, the Gram form of Eq. 9. */
int ress_prepare_wo(const ress_dims* dims, const uint16_t* W_o, float* F, void* stream);

/* Sec. 4.1-4.2: pooled attention map P (softmax over all key blocks of the block-mean
 * logits q_bar . k_bar / 8), the dense pooled output (Eq. 1), q_ij = ||F_h (v_bar_i - V_j)||^2
 * (Eq. 9), drift scores s = P sqrt(q) (Eq. 6) and the initial selection: per candidate
 * query row the c_h candidate blocks with the largest s / max(1 - P, 1e-4) (Eq. 7), ties to
 * the lower block index.  Writes P, q, the initial drop sets and their objective J_0
 * (Eq. 10-12) into the workspace.  c_h_host: host int32 [H], 1 <= c_h <= |P|. */
int ress_score(const ress_dims* dims, const uint16_t* Q, const uint16_t* K, const uint16_t* V,
               const float* F, const int32_t* c_h_host, void* ws, size_t ws_bytes,
               void* stream);

/* Selection variants of the paper's ablations (Sec. 6: the sign flip of Fig. 8 and the
 * probability selection of Table 3; the random baseline of Fig. 8).  `key` picks what the
 * initial selection ranks: the Eq. 7 drift key (ReSS), the pooled probability P_ij alone
 * (top-k by attention mass) or random keys (the top 24 bits of SplitMix64 at the counter
 * seed + (h * 4096 + i) * 4096 + j for row (h, i) and block j; ties to the lower index).
 * `direction` flips the objective: RESS_MAXIMIZE_SWAP makes the restoration rounds maximise
 * J (track-best keeps the largest J), RESS_MAXIMIZE_FULL also makes the initial selection
 * keep the c_h smallest keys.  A NULL variant is ReSS: {RESS_KEY_DRIFT, RESS_MINIMIZE, 0}. */
typedef enum { RESS_KEY_DRIFT = 0, RESS_KEY_PROBABILITY = 1, RESS_KEY_RANDOM = 2 } ress_key_kind;
typedef enum { RESS_MINIMIZE = 0, RESS_MAXIMIZE_SWAP = 1, RESS_MAXIMIZE_FULL = 2 } ress_direction;
typedef struct {
  int32_t key;       /* ress_key_kind  */
  int32_t direction; /* ress_direction */
  uint64_t seed;     /* RESS_KEY_RANDOM */
  float cdf;         /* 0: off.  tau in (0, 1]: the CDF threshold of Table 3 (the top-p rule
                        of probability-based selection on the pooled map).  After its c_h
                        largest keys a candidate row keeps further candidates in key order
                        (ties to the lower index) until the pooled mass P of its kept blocks,
                        the always-kept ones included, reaches tau.  Row lengths then depend
                        on the data; needs rounds = 0 and direction RESS_MINIMIZE.        */
  int32_t reserved;  /* must be 0 */
} ress_variant;

/* col_idx entries that ress_restore_variant may write for this variant: ress_csr_capacity
 * for a fixed budget; with a CDF threshold every query row may keep all nb key blocks, so
 * H * nq * nb.  The entries actually written are row_ptr[H * nq] after the call.  -1 on
 * invalid arguments. */
int64_t ress_csr_capacity_variant(const ress_dims* dims, const int32_t* c_h_host,
                                  const ress_variant* variant);

/* ress_score with a selection variant (NULL: ReSS).  RESS_EINVAL on an unknown key or
 * direction, a CDF threshold outside [0, 1] or combined with a maximising direction, or a
 * nonzero reserved field. */
int ress_score_variant(const ress_dims* dims, const uint16_t* Q, const uint16_t* K,
                       const uint16_t* V, const float* F, const int32_t* c_h_host,
                       const ress_variant* variant, void* ws, size_t ws_bytes, void* stream);

/* Sec. 4.3: `rounds` budget-neutral swap rounds on the drop sets left by ress_score.
 * Round r exchanges m_r = floor(rho c_h / 2^(r+1)) blocks (Eq. 17), capped by the sizes of
 * the two sides: the m_r restores and the m_r drops with the largest exact decrease of
 * J (Eq. 13-16), both taken from the round-start state.  The set with the smallest J seen
 * (track-best, strict <) is returned as kept-block lists in CSR form over the H*nq query
 * rows (h-major; nq query blocks, see ress_dims.q_block): row_ptr device int32 [H*nq + 1],
 * col_idx device int32 [col_capacity] with
 * ascending block indices; col_capacity >= ress_csr_capacity().  Optional device outputs
 * (NULL to skip): J_best float [H*nq] (0 for special query rows), drop_mask uint32
 * [H*nq, ceil(nb/32)] (bit j of row (h, i) set when key block j is dropped).
 * rounds in [0, 32]; rho in [0, 1]. */
int ress_restore(const ress_dims* dims, const int32_t* c_h_host, int32_t rounds, float rho,
                 void* ws, size_t ws_bytes, int32_t* row_ptr, int32_t* col_idx,
                 int64_t col_capacity, float* J_best, uint32_t* drop_mask, void* stream);

/* ress_restore with a selection variant (NULL: ReSS); pass the same variant as to
 * ress_score_variant.  RESS_EINVAL as ress_score_variant, or rounds > 0 with a CDF
 * threshold.  With a CDF threshold the row lengths come from the device (row_ptr is a
 * scan of the per-row kept counts) and col_capacity >= ress_csr_capacity_variant(). */
int ress_restore_variant(const ress_dims* dims, const int32_t* c_h_host, int32_t rounds,
                         float rho, const ress_variant* variant, void* ws, size_t ws_bytes,
                         int32_t* row_ptr, int32_t* col_idx, int64_t col_capacity,
                         float* J_best, uint32_t* drop_mask, void* stream);

/* Sec. 3 step (3): for every head h, query block i and query token of that block,
 * O = softmax(q K^T / 8) V over the tokens of the key blocks listed in row h*nq + i of the
 * CSR (renormalised among them); keys past N are excluded.  Q, K, V: device bf16 [N, H, 64];
 * O: device bf16 [N, H, 64].  Lists must hold ascending, distinct block indices < nb and be
 * non-empty; entries past col_capacity or >= nb are skipped and flagged as RESS_EDEVICE in
 * the status word.  Uses tcgen05 tensor cores with TMA-fed K/V tiles. */
int ress_sparse_attn(const ress_dims* dims, const uint16_t* Q, const uint16_t* K,
                     const uint16_t* V, const int32_t* row_ptr, const int32_t* col_idx,
                     int64_t col_capacity, uint16_t* O, void* ws, size_t ws_bytes,
                     void* stream);

/* ress_sparse_attn with a float32 output O [N, H, 64] (16-byte aligned): the same kernel
 * and the same arithmetic; the bf16 output of ress_sparse_attn is this result rounded to
 * nearest-even.  For callers that keep the attention output in float32 and for checking
 * the kernel against a float32 reference without the bf16 output rounding. */
int ress_sparse_attn_f32(const ress_dims* dims, const uint16_t* Q, const uint16_t* K,
                         const uint16_t* V, const int32_t* row_ptr, const int32_t* col_idx,
                         int64_t col_capacity, float* O, void* ws, size_t ws_bytes, void* stream);

/* ress_score, ress_restore and ress_sparse_attn in order on one stream.  Inside the forward
 * the CSR kernel also writes the attention items' union lists into the workspace, so the
 * attention starts without the union pass of ress_sparse_attn.  The CSR and J_best are bit
 * for bit those of the three separate calls.  O is too on the 128-token query grid; on the
 * 64-token grid the forward pairs the candidate query blocks by the overlap of their kept
 * lists (ress_sparse_attn pairs adjacent blocks), which changes only the order in which a
 * row takes its own kept blocks, so O agrees with the separate calls' to rounding (and is
 * deterministic). */
int ress_forward(const ress_dims* dims, const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                 const float* F, const int32_t* c_h_host, int32_t rounds, float rho, void* ws,
                 size_t ws_bytes, int32_t* row_ptr, int32_t* col_idx, int64_t col_capacity,
                 uint16_t* O, float* J_best, void* stream);

/* ress_forward from host memory to host memory, for callers that keep a layer's Q, K, V
 * and O on the host (the paper has no counterpart: an interface, not part of the method).
 * Enqueued on `stream`, in order: host -> device copies of Q, K, V into the caller's device
 * buffers Q_dev, K_dev, V_dev, then ress_forward on them, with the output brought back while
 * the attention still runs: the attention is split into up to 8 chunks of 128-token query
 * rows, and as each chunk completes its rows of O_dev are copied into O_host on a copy
 * stream the library owns (one per device, with a second compute stream for alternate
 * chunks; both are joined back into `stream` before the call's work ends, so `stream`
 * passing the call means O_host is complete).  Nothing waits for completion on the host.
 * Host buffers should be page-locked (for
 * example cudaHostAlloc) for the copies to overlap other work; every buffer belongs to the
 * caller and must stay untouched until the stream has passed the call.  Two calls on two
 * streams with separate device buffers, workspaces and CSR arrays overlap one layer's copies
 * with another's compute (their attention chunks and output copies share the library's two
 * streams of the device, so those parts of the two calls run one after the other).  Q_host, K_host, V_host, O_host: bf16 [N, H, 64]; the other
 * arguments as ress_forward.  Returns as ress_forward, or RESS_ECUDA if a copy could not be
 * enqueued; arguments are checked before anything is enqueued. */
int ress_forward_host(const ress_dims* dims, const uint16_t* Q_host, const uint16_t* K_host,
                      const uint16_t* V_host, uint16_t* O_host, uint16_t* Q_dev, uint16_t* K_dev,
                      uint16_t* V_dev, uint16_t* O_dev, const float* F, const int32_t* c_h_host,
                      int32_t rounds, float rho, void* ws, size_t ws_bytes, int32_t* row_ptr,
                      int32_t* col_idx, int64_t col_capacity, float* J_best, void* stream);

/* Sec. 3: the attention sublayer's residual update, y = x + O W_o^T (pre-LN structure
 * x_{l+1} = x_l + f_l(x_l); O W_o^T is what the sublayer adds to the residual stream).
 * O: device bf16 [N, H*64] (the attention output, [N, H, 64]); W_o: device bf16 [d_model,
 * H*64] (Linear weight, out x in); x, y: device bf16 [N, d_model] (x may equal y for an in-
 * place update; x NULL gives y = O W_o^T).  fp32 accumulation on the tensor cores (tcgen05),
 * one rounding to bf16.  d_model must be a multiple of 64.  Uses the workspace's status word
 * only. */
int ress_out_proj(const ress_dims* dims, const uint16_t* O, const uint16_t* W_o,
                  const uint16_t* x, uint16_t* y, void* ws, size_t ws_bytes, void* stream);

/* Sec. 3's token-level reference for the drift: for every query block b,
 *   drift[b] = sum over the query tokens t of block b of || W_o (O_a[t] - O_b[t]) ||^2,
 * the squared change one attention output leaves in the residual stream relative to another
 * (O_a sparse, O_b dense in the paper's use).  O_a, O_b: device bf16 [N, H*64]; W_o as in
 * ress_out_proj; drift: device float [ceil(N/64)].  Both products are accumulated in fp32
 * TMEM and subtracted there; each block's sum is formed in a fixed order (deterministic).
 * d_model must be a multiple of 64.  Uses the workspace's status word only. */
int ress_token_drift(const ress_dims* dims, const uint16_t* O_a, const uint16_t* O_b,
                     const uint16_t* W_o, float* drift, void* ws, size_t ws_bytes, void* stream);

/* Allocation-free variant of ress_sparse_attn (the paper has no counterpart: this is an
 * interface for callers, not part of the method).  It is for callers that cannot allocate
 * device memory when they call in: a host framework that owns all device memory through
 * its own pool and forbids allocations inside plugins, a real-time runtime that reserves
 * everything at start-up because a later cudaMalloc can stall the device or fail under a
 * tight budget, or a caller that cannot spare the full workspace for the attention step.
 * Same arguments and results as ress_sparse_attn (bf16 O), without `ws`: the scratch is a
 * file-scope device array of RESS_NOALLOC_SCRATCH_BYTES (4 MiB) that every GPU loading the
 * library holds until the process exits.  No cudaMalloc, cudaFree or allocating routine is
 * called.
 *   - Limit: col_capacity must not exceed (4 MiB - 256 - 4*H*ceil(nb/2) rounded up to 256) / 4
 *     entries (about one million: enough for 16 heads x 32 views at 90% sparsity);
 *     larger requests return RESS_EWORKSPACE with the limit in the message.  The check is on
 *     col_capacity as passed, not on the entries the CSR uses (row_ptr's last value): pass
 *     the used length when the buffer is larger.
 *   - Set-up: the first call on each device looks up the array's device address (with that
 *     device current) and caches it for the life of the process; make that first call
 *     before any stream capture.  A cudaDeviceReset (or anything else that reloads this
 *     library's module in a new primary context) leaves that cached address stale: do not
 *     call this entry point after resetting a device it was already called on.
 *   - Every call shares the one array, and it keeps the last call's contents: calls that
 *     may overlap on the GPU (other streams, other host threads) race and must be ordered
 *     by the caller.  The tile counter is cleared by each call.
 *   - wait != 0: the call synchronises `stream` and returns RESS_ETIMEOUT / RESS_EDEVICE
 *     for device-side failures (then clears them).  wait == 0: asynchronous; a device-side
 *     failure stays recorded until a later call with wait != 0 reports it. */
#define RESS_NOALLOC_SCRATCH_BYTES (4u << 20)
int ress_sparse_attn_noalloc(const ress_dims* dims, const uint16_t* Q, const uint16_t* K,
                             const uint16_t* V, const int32_t* row_ptr, const int32_t* col_idx,
                             int64_t col_capacity, uint16_t* O, int32_t wait, void* stream);

/* Failure detection without a fault, for tests of the error path: one thread waits on a
 * shared-memory barrier that nothing arrives at, with the bounded wait the kernels use
 * (limit_us microseconds, 1..100000), gives up and records RESS_ETIMEOUT in the workspace
 * status word exactly as a kernel's timed-out wait does; ress_status then reports it and
 * clears it, and the context stays usable.  ws: a workspace of any layer (only its status
 * word is used).  RESS_EINVAL on a bad pointer or limit.  No paper counterpart. */
int ress_wait_selftest(void* ws, size_t ws_bytes, uint32_t limit_us, void* stream);

/* Synchronises `stream`, returns the workspace status word as a ress_status_code
 * (RESS_OK, RESS_ETIMEOUT or RESS_EDEVICE) and clears it. */
int ress_status(void* ws, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* RESS_H */
