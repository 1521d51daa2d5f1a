/*
 * cola.h -- C ABI of the GB300 (sm_103a) CoLA auto-encoder layer library.
 *
 * CoLA (arXiv 2502.10940) replaces every full-size projection h = W x of a
 * LLaMA-style block by the low-rank auto-encoder
 *
 *     h = B sigma(A x),   A in R^{r x d_in},  B in R^{d_out x r},  r < min(d_in, d_out)
 *
 * (Sec. 3.2, Eq. (main-fwd)).  This library runs its forward pass and its full
 * backward pass (Sec. 3.4: the "2x rule" grad_x = W^T grad_h,
 * grad_W = grad_h x^T applied to both products, chain rule through sigma) on
 * the tensor cores, in the two modes of the paper: CoLA, which saves both
 * rank-r activations A x and sigma(A x), and CoLA-M (Sec. 4.2, App. C), which
 * saves only A x and recomputes sigma(A x) in the backward.
 *
 * Storage (row-major, token-major; row t = token t, n tokens):
 *   X  [n x d_in]    layer input,              row pitch ld_x  (also dX)
 *   A  [r x d_in]    down-projection factor,    row pitch ld_a  (also dA)
 *   B  [d_out x r]   up-projection factor,      row pitch r     (also dB)
 *   Z  [n x r]       Z = X A^T  (the rank-r activation A x), pitch r
 *   H  [n x r]       H = sigma(Z), pitch r
 *   Y  [n x d_out]   Y = H B^T,   row pitch ld_y (also dY)
 * The paper writes X column-wise (X in R^{d_in x n}, Sec. 3.3); token-major
 * storage is its transpose, and A, B keep the nn.Linear weight layouts.
 *
 * Numerics: every tensor is bf16 (IEEE bfloat16) in device memory; products
 * accumulate in fp32; Z is rounded to bf16 once and H = bf16(sigma(bf16 Z)),
 * so CoLA-M's recomputed H is bit-identical to CoLA's saved H; the gradient at
 * Z is dZ = bf16(fp32(dY B) * sigma'(Z)).  Weight gradients reduce their token
 * split in a fixed order: every result is deterministic.
 *
 * Conventions shared by every entry point:
 *   - All pointers are DEVICE pointers of the current device, owned by the
 *     caller and at least 16-byte aligned.  The library never allocates,
 *     frees or synchronises (cola_check_status excepted).
 *   - Calls are asynchronous on `stream` (0 = legacy default stream).
 *     Argument errors are detected before any launch and return without
 *     touching memory.  A launch failure returns COLA_ERR_LAUNCH.
 *   - Sizes: n, d_in, d_out >= 1; r >= 64 and r % 64 == 0 (else
 *     COLA_ERR_UNSUPPORTED); row pitches (ld_*) are in elements, >= the
 *     logical width and a multiple of 8 (16 bytes); 0 selects the logical
 *     width.  Every extent must stay below 2^31 elements per row/column.
 *   - `ws` is a caller-owned device workspace of at least
 *     cola_workspace_size() bytes, 256-byte aligned; its first 256 bytes hold
 *     the device status word and must be zeroed once with
 *     cola_workspace_init() before first use.  One workspace must not be
 *     used by two calls that may run concurrently.
 *   - The entry points may be called from several host threads at once, each
 *     with its own workspace (and, typically, its own stream); the launch
 *     tracing below is the one exception.
 *   - Every wait inside the kernels is bounded (about 2 s).  A wait that runs
 *     out records a code in the workspace status word and the kernel returns
 *     early (its outputs are then undefined); cola_check_status() reports it.
 */
#ifndef COLA_H
#define COLA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    COLA_OK = 0,
    COLA_ERR_INVALID = 1,        /* null pointer, non-positive size, bad pitch or enum */
    COLA_ERR_ALIGN = 2,          /* a pointer not 16-byte aligned (ws: 256-byte) */
    COLA_ERR_UNSUPPORTED = 3,    /* r not a positive multiple of 64, extent too large, no sm_103 device */
    COLA_ERR_WORKSPACE = 4,      /* ws_bytes below cola_workspace_size() */
    COLA_ERR_LAUNCH = 5,         /* a CUDA launch or driver call failed */
    COLA_ERR_DEVICE_TIMEOUT = 6  /* a bounded device-side wait ran out (see cola_check_status) */
} cola_status_t;

typedef enum {
    COLA_SIGMA_IDENTITY = 0,     /* sigma(z) = z: the plain low-rank product B A x */
    COLA_SIGMA_SILU = 1,         /* Swish / SiLU, z / (1 + e^-z) (LLaMA, Sec. 5) */
    COLA_SIGMA_GELU = 2          /* GELU, erf form z * Phi(z) (BERT, Sec. 5.2) */
} cola_sigma_t;

typedef enum {
    COLA_MODE_COLA = 0,          /* forward stores Z and H; backward reads both */
    COLA_MODE_COLA_M = 1,        /* forward stores Z only; backward recomputes H = sigma(Z) */
    COLA_MODE_INFER = 2          /* forward only (inference, App. E.2): nothing is saved, H lives
                                    in the workspace; the backward entry points reject it */
} cola_mode_t;

/* The layer of Eq. (main-fwd) as the paper states it: (d_in, d_out, rank r,
 * sigma) applied to n tokens. */
typedef struct {
    int64_t n;          /* tokens (sequences x sequence length) */
    int64_t d_in;       /* input width */
    int64_t d_out;      /* output width */
    int64_t r;          /* rank, r % 64 == 0 */
    int64_t ld_x;       /* row pitch of X and dX in elements (0: d_in) */
    int64_t ld_y;       /* row pitch of Y and dY in elements (0: d_out) */
    int64_t ld_a;       /* row pitch of A and dA in elements (0: d_in) */
    int32_t sigma;      /* cola_sigma_t */
    int32_t mode;       /* cola_mode_t */
    int32_t wgrad_fp32; /* 0: dA, dB are bf16 and overwritten; 1: dA, dB are fp32 and
                           accumulated into (dA += ..., dB += ...), row pitches as above */
    int32_t reserved;   /* must be 0 */
} cola_desc_t;

/* Bytes of workspace the calls on `nproj` projections of shape `desc` that
 * share one input need on the current device: nproj = 1 for cola_fwd /
 * cola_bwd, 2 or 3 for cola_fwd_shared_x / cola_bwd_shared_x with that count
 * (3 for the q/k/v entry points).  The value depends on n, r, d_in, d_out,
 * the mode, wgrad_fp32 and the device's SM count (it sizes the
 * weight-gradient split over tokens). */
cola_status_t cola_workspace_size(const cola_desc_t* desc, int32_t nproj, size_t* bytes);

/* Zero the workspace status word (first 256 bytes of ws), asynchronously. */
cola_status_t cola_workspace_init(void* ws, void* stream);

/* Forward, Eq. (main-fwd):  Z = X A^T,  H = sigma(Z),  Y = H B^T.
 *   X [n x d_in] (ld_x), A [r x d_in] (ld_a), B [d_out x r]: inputs.
 *   Y [n x d_out] (ld_y): output.
 *   Z_save [n x r]: output, saved for the backward (COLA, COLA_M); must be
 *                   NULL under COLA_MODE_INFER (Z is then never stored).
 *   H_save [n x r]: output under COLA_MODE_COLA; must be NULL under COLA_M
 *                   and INFER (H is then formed in the workspace and not kept).
 * Two tensor-core GEMMs: Z/H (sigma fused in the epilogue), then Y.  For
 * r = 64 or 128 when both products are HBM-bound (neither compute-heavy nor
 * split over K) and n is at most 128 tokens per SM (19456 on GB300), one
 * kernel instead: each CTA keeps the H of its 128-row tile in shared memory
 * between the two products (H is an intermediate of Eq. (main-fwd), not an
 * output), storing Z and H only as the mode saves them; the results are the
 * same bit for bit (cola_set_fused_forward). */
cola_status_t cola_fwd(const cola_desc_t* desc, const void* X, const void* A, const void* B, void* Y,
                       void* Z_save, void* H_save, void* ws, size_t ws_bytes, void* stream);

/* Backward, Sec. 3.4 (two GEMMs per forward GEMM, chain rule through sigma):
 *   dZ = (dY B) * sigma'(Z)      [n x r]    (workspace)
 *   dB = dY^T H                  [d_out x r]
 *   dA = dZ^T X                  [r x d_in] (ld_a)
 *   dX = dZ A                    [n x d_in] (ld_x)
 * Inputs X, A, B, dY [n x d_out] (ld_y), Z_save; H_save under COLA (must be
 * NULL under COLA_M, where H = sigma(Z_save) is recomputed into the
 * workspace).  Outputs dX (bf16), dA and dB (bf16, or fp32 accumulated when
 * desc->wgrad_fp32).  The result does not depend on the mode, bit for bit.
 * Launches: the dZ GEMM (sigma' fused in its epilogue), the weight-gradient
 * GEMMs (and their token-split reduce), the dX GEMM.  For r = 64 or 128 when
 * neither the dZ nor the dX GEMM is compute-heavy and n is at most 128
 * tokens per SM, dZ and dX run as one kernel instead: each CTA keeps the dZ
 * of its 128-row tile in shared memory between the two products (loading the
 * tile's Z there and overwriting it with dZ), storing dZ (and, under COLA_M,
 * H) to the workspace for the weight gradients; the results are the same
 * bit for bit (cola_set_fused_backward). */
cola_status_t cola_bwd(const cola_desc_t* desc, const void* X, const void* A, const void* B, const void* dY,
                       const void* Z_save, const void* H_save, void* dX, void* dA, void* dB, void* ws,
                       size_t ws_bytes, void* stream);

/* Projections that read the same input (Fig. 4: q, k and v read the
 * attention input; gate and up read the MLP input): `count` = 2 or 3 CoLA
 * layers of one shape (desc: d_in, d_out, r per projection) on one X.
 *   A_cat [count r x d_in] (ld_a): the A_j stacked by rows.  One GEMM with
 *     N = count r reads X once and writes Z_cat [n x count r] = [Z_1 .. Z_c]
 *     and, under COLA, H_cat [n x count r] (NULL under COLA_M; under
 *     COLA_MODE_INFER both Z_cat and H_cat are NULL).
 *   B[j] [d_out x r], Y[j] [n x d_out] (ld_y): host arrays of `count` device
 *     pointers; the count output GEMMs Y_j = H_j B_j^T run as one launch. */
cola_status_t cola_fwd_shared_x(const cola_desc_t* desc, int32_t count, const void* X, const void* A_cat,
                                const void* const* B, void* const* Y, void* Z_cat, void* H_cat, void* ws,
                                size_t ws_bytes, void* stream);

/* Backward of cola_fwd_shared_x: dZ_j = (dY_j B_j) * sigma'(Z_j) for all j in
 * one launch; dB_j = dY_j^T H_j and dA_cat = dZ_cat^T X (M = count r) in one
 * launch; dX = dZ_cat A_cat (K = count r), i.e. the sum of the count input
 * gradients, as one GEMM.  dY[j], dB[j]: host arrays of device pointers;
 * dA_cat [count r x d_in] (ld_a); H_cat NULL under COLA_M. */
cola_status_t cola_bwd_shared_x(const cola_desc_t* desc, int32_t count, const void* X, const void* A_cat,
                                const void* const* B, const void* const* dY, const void* Z_cat, const void* H_cat,
                                void* dX, void* dA_cat, void* const* dB, void* ws, size_t ws_bytes, void* stream);

/* Fused q/k/v forward (Fig. 4: the q, k and v auto-encoders read the same x);
 * cola_fwd_shared_x with count = 3.
 * desc->d_out is the width of each projection; desc->r the rank of each.
 *   A_qkv [3r x d_in] (ld_a) = [A_q; A_k; A_v] stacked by rows: one GEMM with
 *   N = 3r reads X once and writes Z_qkv [n x 3r] = [Z_q Z_k Z_v] and (COLA)
 *   H_qkv [n x 3r]; then Y_j = H_j B_j^T for j in q, k, v (Y_j pitch ld_y).
 * H_qkv must be NULL under COLA_M. */
cola_status_t cola_fwd_qkv_fused(const cola_desc_t* desc, const void* X, const void* A_qkv, const void* B_q,
                                 const void* B_k, const void* B_v, void* Y_q, void* Y_k, void* Y_v,
                                 void* Z_qkv, void* H_qkv, void* ws, size_t ws_bytes, void* stream);

/* Fused q/k/v backward (cola_bwd_shared_x with count = 3): three
 * dZ_j = (dY_j B_j) * sigma'(Z_j) into one
 * [n x 3r] buffer, then one GEMM with M = 3r gives dA_qkv [3r x d_in] (ld_a),
 * one GEMM with K = 3r gives dX = sum_j dZ_j A_j (ld_x), and dB_j = dY_j^T H_j.
 * H_qkv must be NULL under COLA_M. */
cola_status_t cola_bwd_qkv_fused(const cola_desc_t* desc, const void* X, const void* A_qkv, const void* B_q,
                                 const void* B_k, const void* B_v, const void* dY_q, const void* dY_k,
                                 const void* dY_v, const void* Z_qkv, const void* H_qkv, void* dX, void* dA_qkv,
                                 void* dB_q, void* dB_k, void* dB_v, void* ws, size_t ws_bytes, void* stream);

/* ---- the gated MLP (Fig. 4; Sec. 3.2; App. E) ----
 * LLaMA's MLP multiplies its gate and up projections element-wise and feeds
 * the product to the down projection.  CoLA turns gate, up and down into
 * auto-encoder layers and keeps the element-wise product (Sec. 3.2), with no
 * full-rank activation on the gate branch (App. E, "Low-Rank sigma Only"):
 *     M = Y_gate (.) Y_up,   Y_gate = B_gate sigma(A_gate x),  Y_up = B_up sigma(A_up x).
 *
 * Forward of gate and up and their product.  desc describes ONE of the two
 * projections (d_in = model width, d_out = d_ff, r); both read X.
 *   A_cat [2r x d_in] (ld_a) = [A_gate; A_up] stacked by rows: one GEMM with
 *     N = 2r reads X once and writes Z_cat [n x 2r] = [Z_gate Z_up] and, under
 *     COLA, H_cat [n x 2r], exactly as cola_fwd_shared_x with count 2.
 *   B_gate, B_up [d_out x r]: one GEMM over both, each output tile's gate and
 *     up halves in two accumulators of one CTA (CTA pair), whose epilogue
 *     stores M [n x d_out] (ld_y) = bf16(Y_gate * Y_up), the product of the
 *     bf16-rounded outputs (exact in fp32, rounded once), and, in the
 *     training modes, Y_gate and Y_up [n x d_out] (ld_y) = bf16 outputs for
 *     the backward.  Under COLA_MODE_INFER Y_gate, Y_up, Z_cat and H_cat must
 *     be NULL (M alone is stored); otherwise Y_gate and Y_up are required.
 * ws: cola_workspace_size(desc, 2).  The gate/up backward is
 * cola_bwd_shared_x (count 2) with dY = {dY_gate, dY_up} from
 * cola_bwd_down_gated. */
cola_status_t cola_fwd_gate_up(const cola_desc_t* desc, const void* X, const void* A_cat, const void* B_gate,
                               const void* B_up, void* M, void* Y_gate, void* Y_up, void* Z_cat, void* H_cat,
                               void* ws, size_t ws_bytes, void* stream);

/* Backward of the down projection whose input is M = Y_gate (.) Y_up: as
 * cola_bwd with X = M (desc: the down layer, d_in = d_ff, ld_x = the pitch of
 * M, Y_gate, Y_up, dY_gate, dY_up), except that its input gradient
 * dM = dZ A is not stored: the epilogue of that GEMM reads Y_gate and Y_up
 * and stores the gradients at the product's factors,
 *     dY_gate = bf16(bf16(dM) * Y_up),   dY_up = bf16(bf16(dM) * Y_gate),
 * which the gate/up backward (cola_bwd_shared_x, count 2) takes as its dY.
 * dA, dB as in cola_bwd; H_save NULL under COLA_M; ws: cola_workspace_size(desc, 1). */
cola_status_t cola_bwd_down_gated(const cola_desc_t* desc, const void* M, const void* A, const void* B,
                                  const void* dY, const void* Z_save, const void* H_save, const void* Y_gate,
                                  const void* Y_up, void* dY_gate, void* dY_up, void* dA, void* dB, void* ws,
                                  size_t ws_bytes, void* stream);

/* Block-level CoLA-M recompute of the up-projections (Sec. 4.2, App. C:
 * in the backward, CoLA-M recomputes B sigma(.) from the saved low-rank
 * activation instead of keeping the layer output):
 *   Y_j = sigma(Z_j) B_j^T        for j < count (1..3 projections)
 * Z_cat [n x count r]: the Z saved by cola_fwd / cola_fwd_shared_x under
 * COLA_MODE_COLA_M (column block j = Z_j).  B[j] [d_out x r], Y[j]
 * [n x d_out] (ld_y): host arrays of `count` device pointers.  desc->mode
 * must be COLA_MODE_COLA_M; ws must be sized by cola_workspace_size(desc,
 * count), and H = sigma(Z) is formed in it (one elementwise launch) before
 * the count output GEMMs run as one launch.  Y_j is bit for bit the Y_j of
 * the forward call that saved Z_cat. */
cola_status_t cola_recompute_up(const cola_desc_t* desc, int32_t count, const void* Z_cat, const void* const* B,
                                void* const* Y, void* ws, size_t ws_bytes, void* stream);

/* Synchronise `stream`, read and clear the workspace status word.
 * Returns COLA_OK, or COLA_ERR_DEVICE_TIMEOUT if a kernel that used this
 * workspace gave up on a wait since the last check (*code_out, if not NULL,
 * receives the raw status bits below), or COLA_ERR_LAUNCH on a CUDA error.
 * Every wait in the kernels is bounded (2 s of GPU global time); a wait that
 * runs out raises an abort flag that ends its CTA's other waits, and the
 * kernel drains its own copies and MMAs (bounded), frees its TMEM and exits,
 * leaving the results of that launch undefined and the context usable. */
#define COLA_STATUS_PRODUCER_TIMEOUT 0x1u   /* a TMA producer gave up waiting for a free stage */
#define COLA_STATUS_MMA_TIMEOUT 0x2u        /* an MMA issuer gave up waiting for operands or TMEM */
#define COLA_STATUS_EPILOGUE_TIMEOUT 0x4u   /* an epilogue gave up waiting for an accumulator or saved Z */
#define COLA_STATUS_DRAIN_TIMEOUT 0x8u      /* a CTA gave up waiting for its own copies or MMAs to drain */
cola_status_t cola_check_status(void* ws, void* stream, uint32_t* code_out);

/* ---- failure detection self-test ----
 * The paper has no counterpart.  Launches one 128 x 128 x 64 GEMM (operands
 * and output in ws after its 256-byte status header; ws_bytes >= 256 + 96 KB)
 * whose TMA producer issues no loads, so that its MMA issuer's first wait
 * runs out after 2 s: the next cola_check_status on ws then returns
 * COLA_ERR_DEVICE_TIMEOUT with COLA_STATUS_MMA_TIMEOUT set (and, if the
 * epilogue's wait for that accumulator ran out first, also
 * COLA_STATUS_EPILOGUE_TIMEOUT; no other bit).  No copy or MMA
 * is ever in flight, nothing in ws beyond the status word is touched, and the
 * CUDA context stays usable.  Async on `stream`. */
cola_status_t cola_selftest_wait_timeout(void* ws, size_t ws_bytes, void* stream);

/* The same self-test on a CTA pair (tcgen05 cta_group::2, the tile of the
 * compute-heavy GEMMs): one 256 x 256 x 512 GEMM whose operands (zeros) and
 * output lie in ws after its status header (ws_bytes >= 256 + 640 KB).
 *   variant 1: neither CTA's TMA producer issues a load; the even CTA's MMA
 *              issuer and the odd CTA's epilogue give up after 2 s.
 *   variant 2: the odd CTA's producer issues its first k-block only, while
 *              the even CTA's producer fills its whole ring; the MMA
 *              issuer's second wait runs out with the even CTA's loads of
 *              six more stages landed or in flight.  Before the pair exits,
 *              the even CTA must see every load of both CTAs land (the abort
 *              drain of a pair), or it records COLA_STATUS_DRAIN_TIMEOUT.
 * The next cola_check_status on ws returns COLA_ERR_DEVICE_TIMEOUT with some
 * of COLA_STATUS_PRODUCER_TIMEOUT, COLA_STATUS_MMA_TIMEOUT and
 * COLA_STATUS_EPILOGUE_TIMEOUT set and, when the drain saw every load land,
 * not COLA_STATUS_DRAIN_TIMEOUT.  Nothing is stored (ws beyond the status
 * word is only read), and the CUDA context stays usable.  Async on `stream`;
 * variant outside {1, 2}: COLA_ERR_INVALID. */
cola_status_t cola_selftest_wait_timeout_pair(void* ws, size_t ws_bytes, int32_t variant, void* stream);

/* The same self-test on a cluster-reduced weight gradient (cola_set_cluster_splitk):
 * one 128 x 128 gradient tile over 512 tokens split over a cluster of two
 * CTAs, operands in ws after its status header (ws_bytes >= 256 + 256 KB).
 * CTA 1 issues no loads: its MMA issuer gives up after 2 s, and it still
 * sends its (zero) partial band so that CTA 0 completes; CTA 0 then stores its
 * band (64 rows of bf16) over the start of the first operand, CTA 1 stores
 * nothing.  The next cola_check_status on ws returns COLA_ERR_DEVICE_TIMEOUT
 * with some of COLA_STATUS_PRODUCER_TIMEOUT, COLA_STATUS_MMA_TIMEOUT and
 * COLA_STATUS_EPILOGUE_TIMEOUT set and not COLA_STATUS_DRAIN_TIMEOUT (the
 * exchange between the two CTAs completed), and the CUDA context stays
 * usable.  Async on `stream`. */
cola_status_t cola_selftest_wait_timeout_cluster(void* ws, size_t ws_bytes, void* stream);

/* ---- weight gradient without any workspace or allocation ----
 * The paper has no counterpart to this entry point.  It serves callers that
 * cannot allocate device memory: an operator or plugin interface that hands
 * the library its inputs and outputs but no workspace, or a process whose
 * device memory is fixed at start-up by another allocator, where any later
 * cudaMalloc would fail or break its budget.
 *
 *   D[M x N] = sum over t < n_tokens of P[t, m] * Q[t, n]
 *
 * i.e. dB = dY^T H (P = dY [n x d_out], Q = H [n x r]) or dA = dZ^T X
 * (P = dZ [n x r], Q = X [n x d_in]), the token-reduction GEMM of cola_bwd
 * on the same kernels.  P, Q: bf16, token-major, row pitches ld_p, ld_q
 * (elements, multiples of 8).  D: bf16 (overwritten) or, with
 * accumulate_f32 = 1, fp32 accumulated into (D += ...); row pitch ld_d.
 * All pointers are device pointers, 16-byte aligned; async on `stream`.
 *
 * The token-split partial sums live in one static device array of
 * COLA_STATIC_SCRATCH_BYTES inside libcola.so, which every GPU that loads
 * the array holds until the process exits.  The entry point calls no
 * cudaMalloc, cudaFree or other allocating routine.  A problem whose fp32
 * partial tile grid (M and N rounded up to the tile size) does not fit the
 * array even without a token split returns COLA_ERR_WORKSPACE before any
 * launch.  A problem the planner runs without a token split, with a bf16
 * D, stores D straight from the GEMM epilogue and does not touch the array.
 * The first call on each device that uses the array fetches its device
 * address (cudaGetSymbolAddress, which may load the library's device module;
 * a failed lookup returns COLA_ERR_LAUNCH and is retried by the next call):
 * make that first call before any stream capture begins on the device.  Every
 * call shares the one array, so calls that may overlap on the GPU (other
 * streams, other host threads) race and must be serialised by the caller.
 * Nothing in the array needs to start at zero: each call overwrites the
 * partials it reads.  A device-side wait that runs out leaves D undefined
 * and is not reported here (there is no workspace status word). */
#define COLA_STATIC_SCRATCH_BYTES (64u * 1024u * 1024u)

cola_status_t cola_wgrad_static_scratch(int64_t n_tokens, int64_t M, int64_t N, const void* P, int64_t ld_p,
                                        const void* Q, int64_t ld_q, void* D, int64_t ld_d, int32_t accumulate_f32,
                                        void* stream);

/* ---- launch tracing (optional; for measurement) ----
 * While a slot array is attached, every kernel the library launches is
 * bracketed by two CUDA events recorded on the launch stream: slot
 * (*count) receives the events' use, the kernel kind and the extents of the
 * GEMMs (one launch may run up to four of one kind: the q/k/v outputs, the
 * weight gradients of a layer), and *count is incremented (host side) until
 * it reaches `capacity`.
 * `start` / `stop` are cudaEvent_t handles the caller created with timing
 * enabled, one distinct pair per slot; the library only records them.
 * The attachment is process-wide and not thread-safe: attach, launch and
 * detach from one host thread. */
typedef enum {
    COLA_KERNEL_FWD_ZH = 0,      /* Z = X A^T, H = sigma(Z)               (M=n, N=r or 3r, K=d_in) */
    COLA_KERNEL_FWD_Y = 1,       /* Y = H B^T                             (M=n, N=d_out, K=r) */
    COLA_KERNEL_BWD_DZ = 2,      /* dZ = (dY B) * sigma'(Z)               (M=n, N=r, K=d_out) */
    COLA_KERNEL_WGRAD = 3,       /* dB = dY^T H and dA = dZ^T X, token split (M=d_out | r, N=r | d_in, K=n) */
    COLA_KERNEL_REDUCE = 4,      /* fixed-order sum of the partials       (M, N of the gradient, K=splits) */
    COLA_KERNEL_BWD_DX = 5,      /* dX = dZ A                             (M=n, N=d_in, K=r or 3r) */
    COLA_KERNEL_SIGMA = 6,       /* H = sigma(Z), elementwise             (M=n, N=count r, K=0) */
    COLA_KERNEL_FWD_GLU = 7,     /* M = (H_gate B_gate^T) * (H_up B_up^T) (M=n, N=d_ff, K=2r) */
    COLA_KERNEL_FWD_FUSED = 8,   /* Z, H = sigma(Z), Y = H B^T in one kernel, count 2:
                                    (n, r, d_in) and (n, d_out, r) */
    COLA_KERNEL_BWD_FUSED = 9    /* dZ = (dY B) * sigma'(Z), dX = dZ A in one kernel, count 2:
                                    (n, r, d_out) and (n, d_in, r) */
} cola_kernel_t;

typedef struct {
    void* start;        /* cudaEvent_t, recorded just before the launch */
    void* stop;         /* cudaEvent_t, recorded just after the launch */
    int32_t kernel;     /* cola_kernel_t */
    int32_t count;      /* GEMMs (or reductions) this one launch runs, 1..4 */
    int32_t mnk[4][3];  /* M, N, K of each (reductions: M, N, splits) */
    int32_t splits;     /* token splits (weight gradients), else 1 */
    int32_t flags;      /* bit 0: the epilogue also wrote H (CoLA forward or CoLA-M backward);
                           bit 1: a forward GEMM split over K into fp32 partials (the reduce
                                  launch after it applies the epilogue);
                           bit 2: the GEMM ran on CTA pairs (clusters of two CTAs, tcgen05
                                  cta_group::2, 256-row tiles);
                           bit 3: one CTA ran two 128-row sub-tiles sharing each B tile;
                           bit 4: weight gradients with a split tail (splits = pieces per
                                  tail tile; a reduce launch follows when they are > 1);
                           bit 5: the dX epilogue stored the gated-MLP gradients dY_gate,
                                  dY_up instead of dX (cola_bwd_down_gated);
                           bit 6: the fused forward stored Z (bit 0: it stored H; in the
                                  fused backward bit 0 means H recomputed under CoLA-M);
                           bit 7: the GEMM's K range split `splits` ways inside thread-block
                                  clusters of that size, the partial tiles reduced on chip and
                                  the epilogue applied in the same launch (no reduce launch) */
} cola_trace_slot_t;

cola_status_t cola_trace_attach(cola_trace_slot_t* slots, int32_t capacity, int32_t* count);
cola_status_t cola_trace_detach(void);

/* Process-wide choice of cola_fwd's forward where the single-kernel form
 * applies (see cola_fwd): 1 (default) runs it, 0 runs the two GEMMs instead,
 * for comparisons; both give the same results bit for bit.  enable outside
 * {0, 1}: COLA_ERR_INVALID.  Takes effect for calls made after it returns. */
cola_status_t cola_set_fused_forward(int32_t enable);

/* The same choice for cola_bwd's dZ and dX GEMMs (see cola_bwd): 1 (default)
 * runs them as one kernel where that form applies, 0 as two GEMMs; both give
 * the same results bit for bit.  enable outside {0, 1}: COLA_ERR_INVALID. */
cola_status_t cola_set_fused_backward(int32_t enable);

/* Weight-gradient launches with few output tiles and a short token walk (a
 * few thousand tokens) split their tokens to fill the SMs.  1 (default): the
 * splits of a 128 x 128 gradient tile run as one thread-block cluster of up
 * to 8 CTAs that adds the partial tiles on chip, in a fixed order, and
 * stores (or accumulates) in the same launch; 0: the planned split with fp32
 * partials in the workspace and a reduce launch.  The two add the same
 * partials in the same order only when they split alike, so results may
 * differ in the last bits between the settings (each is deterministic run
 * to run).  enable outside {0, 1}: COLA_ERR_INVALID. */
cola_status_t cola_set_cluster_splitk(int32_t enable);

/* Static description of a status code. */
const char* cola_status_string(cola_status_t status);

#ifdef __cplusplus
}
#endif

#endif /* COLA_H */
