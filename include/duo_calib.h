/*
 * duo_calib.h -- C ABI of libduo's calibration precompute: the part of
 * DuoGPT's activation-sparsity-aware pruning (§4.3, Algorithm 1) that is
 * computed once per layer before the column sweep, on one GPU.
 *
 * Notation (§3, §4.3): W (n x k) is the layer weight; the calibration input
 * X (k x m) has one column per token.  X_hat keeps in every token the
 * `keep` channels of largest |x| (§3; equal magnitudes: lower channel index
 * first); X_tilde = X is the dense input; dX = X_tilde - X_hat.
 *
 *   H = X_hat X_hat^T + damp * mean(diag) * I     (act_order, dampening: App. B.1)
 *   H^-1 = L L^T, L lower-triangular               ("Inverse_Cholesky")
 *   Q = dX X_hat^T L,  U = Q (.) M_u (strictly upper part of Q)
 *   a = diag(dX dX^T), b = diag(U U^T), c = diag(Q) / diag(L), D = U L^T
 *   S[:, p] = W[:, p]^2 (1 / L_pp^2 + a_p - b_p + 2 c_p)   (the efficient score)
 *
 * Readings where the paper is silent: a channel with H_ii = 0 (never kept)
 * gets H_ii = 1; with act_order the channels are reordered by the exact
 * Hessian diagonal, largest first, ties to the lower index, before the
 * dampening; every output is in that processing order (position p holds
 * original channel perm[p]).
 *
 * Precision: X is fp16; H and dX X_hat^T are fp16 products accumulated in
 * fp32; the factorisation and the products with L are fp32 (on the tensor
 * cores: each fp32 operand split into three bf16 pieces, six piece products
 * summed in fp32).  The act_order permutation is decided on exact integer
 * sums, so it is reproducible.
 *
 * All pointers named *_dev are device memory.  Calls are asynchronous on the
 * given stream (a cudaStream_t passed as void*) unless stated.
 */
#ifndef DUO_CALIB_H
#define DUO_CALIB_H

#include <stdint.h>

#include "duo.h"   /* status codes DUO_OK, DUO_EINVAL, ... */

#ifdef __cplusplus
extern "C" {
#endif

/* Opaque: library handles, workspace and the precomputed quantities of one
 * layer shape (k channels, m tokens).  Owned by the library from
 * duo_calib_create to duo_calib_free. */
typedef struct duo_calib duo_calib;

/*
 * duo_calib_create -- allocates a context for k channels and m tokens:
 * about 9 k^2 fp32 plus 2 k m fp16 of device memory, two buffers for
 * prepared tensor-core operands (k^2 fp32 split into three bf16 pieces,
 * 6 k^2 bytes each, at least), and a high-priority side stream with two
 * events, on which the factorisation runs its diagonal blocks (work
 * enqueued on the caller's stream forks to it and joins back, so a stream
 * capture takes it in).  Synchronous.
 *   k : 1..32768 channels.   m : 1..2^20 tokens.
 * Errors: DUO_EINVAL (sizes, NULL), DUO_ENOMEM, DUO_ECUDA.
 */
int duo_calib_create(int64_t k, int64_t m, void* stream, duo_calib** out);

/*
 * duo_calib_precompute -- the precompute of Algorithm 1 for one layer.
 *   X_fp16_dev : device fp16, token-major: m rows of k activations, token t's
 *                input at X[t*k .. t*k + k-1] (this is X^T in the paper's
 *                k x m notation).  Finite values.
 *   keep       : channels kept per token, 0..k.
 *   damp       : dampening ratio (0.1 in the paper's settings), >= 0.
 *   act_order  : 1 = reorder channels by the Hessian diagonal, 0 = keep order.
 * The results stay in the context (duo_calib_query / duo_calib_export).
 * A factorisation that fails (H not positive definite, e.g. damp = 0 with a
 * singular H) is reported by duo_calib_status, not here.
 * Errors: DUO_EINVAL (NULL, dead context, keep, damp), DUO_ECUDA.
 */
int duo_calib_precompute(duo_calib* h, const void* X_fp16_dev, int64_t keep, float damp,
                         int act_order, void* stream);

/* Synchronises `stream`, then reports the last precompute's factorisation:
 * DUO_OK, or DUO_ERANGE if the Cholesky factorisation of the dampened H
 * failed (not positive definite); DUO_ETIMEOUT if a bounded wait inside a
 * tensor-core product ran out since the last call (a process-wide word,
 * read and cleared here; that product's output tile was not written);
 * DUO_ECUDA on a CUDA error. */
int duo_calib_status(const duo_calib* h, void* stream);

/* Buffers of a context (device pointers owned by the context; valid until
 * the next precompute or duo_calib_free).  Matrices are k x k, ROW-major:
 * element (p, i) at [p*k + i]. */
typedef struct duo_calib_info {
    int64_t k, m;
    const int32_t* perm_dev;  /* [k] original channel at position p            */
    const float* H_dev;       /* dampened, reordered Hessian (symmetric)        */
    const float* L_dev;       /* lower factor, H^-1 = L L^T                     */
    const float* Q_dev;       /* Q = dX X_hat^T L                               */
    const float* U_dev;       /* U = Q with the diagonal and below set to 0     */
    const float* D_dev;       /* D = U L^T                                      */
    const float* a_dev;       /* [k] */
    const float* b_dev;       /* [k] */
    const float* c_dev;       /* [k] */
    const float* col_dev;     /* [k] 1 / L_pp^2 + a_p - b_p + 2 c_p             */
} duo_calib_info;

int duo_calib_query(const duo_calib* h, duo_calib_info* info);

/* Copies one buffer of the context into caller device memory (async).
 *   which : 0 perm (int32 [k]), 1 H, 2 L, 3 Q, 4 U, 5 D (fp32 [k*k] row-major),
 *           6 a, 7 b, 8 c, 9 col (fp32 [k]).
 *   bytes : must equal the buffer's size.
 * Errors: DUO_EINVAL (dead context, which, NULL, size), DUO_ECUDA. */
int duo_calib_export(const duo_calib* h, int which, void* dst_dev, int64_t bytes, void* stream);

/*
 * duo_calib_score -- S = W^2 (1 / L_pp^2 + a - b + 2 c) per column p (the
 * efficient score of §4.3) for the last precompute.
 *   W_fp16_dev : device fp16, n x k row-major with leading dimension ldw,
 *                columns in the ORIGINAL channel order.
 *   S_dev      : device fp32, n x k row-major (leading dimension k), columns
 *                in the processing order (column p = channel perm[p]).
 * Errors: DUO_EINVAL (NULL, n < 1, ldw < k, dead context), DUO_ECUDA.
 */
int duo_calib_score(const duo_calib* h, const void* W_fp16_dev, int64_t n, int64_t ldw,
                    float* S_dev, void* stream);

/*
 * duo_calib_prune -- Algorithm 1's column sweep for the last precompute: in
 * the processing order, blocks of `block` columns; at each block's start the
 * scores S = W^2 (1 / L_pp^2 + a - b + 2 c) of its current weights choose
 * the floor(n * B_j * pw_pct / 100) weights to prune (lowest scores; equal
 * scores: lower flat index r * B_j + c first); then column by column
 * P_j = W_j M_j, E_j = (W_j - P_j) / L_jj and later columns q get
 * W_q -= E_j L_qj - W_j D_jq (within the block at once, for the columns
 * after the block in one lazy product that uses each W_j as it was at its
 * step); finally W_j = P_j.  Asynchronous; the context keeps scratch of
 * about n k (4 + 1) + n 2 KiB bytes, grown when a call needs more rows
 * (growing waits for the stream), and 8 k^2 bytes for the lazy products'
 * operand (interleaved -L and D^T), rebuilt after each precompute.
 *   W_fp16_dev : device fp16, n x k row-major (leading dimension ldw), the
 *                dense weight in the ORIGINAL channel order.
 *   pw_pct     : weight sparsity in percent, 0..100.   block : 1..128 (the
 *                paper uses 128).
 *   Wout_dev   : device fp32, n x k row-major: the pruned and compensated
 *                weight in the original channel order, pruned entries 0.
 *   keep_dev   : device uint8 n x k (original order), 1 = kept; may be NULL.
 * Errors: DUO_EINVAL (NULL, sizes, pw_pct, block, dead context), DUO_ENOMEM,
 * DUO_ECUDA.
 */
int duo_calib_prune(duo_calib* h, const void* W_fp16_dev, int64_t n, int64_t ldw, int pw_pct,
                    int block, float* Wout_dev, uint8_t* keep_dev, void* stream);

/* Frees a context (NULL is a no-op; an unknown or freed handle: DUO_EINVAL). */
int duo_calib_free(duo_calib* h);

#ifdef __cplusplus
}
#endif

#endif /* DUO_CALIB_H */
