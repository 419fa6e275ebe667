/*
 * duo.h -- C ABI of the GB300 (sm_103a) dual-sparse batch-1 spMspV library.
 *
 * The library computes the decode-time product of DuoGPT (arXiv 2506.20194),
 * §3 "Activation Sparsity":
 *
 *     y = W (x ⊙ m^x) = sum_{i : m^x_i = 1} W[:, i] * x_i
 *
 * where W (O rows x I input channels, fp16) carries unstructured weight
 * sparsity (pruned entries are stored as zero, §3 mask m^w) and m^x keeps the
 * k input channels of largest |x_i|, chosen per input at decode time (§3).  §4.1
 * describes the execution: only the compressed weight columns of the
 * surviving channels are fetched from HBM.
 *
 * Conventions shared by every entry point:
 *   - Every call returns an int status (DUO_OK or a negative DUO_E* code) and
 *     never aborts the process.  Arguments are validated on the host before
 *     any CUDA call; an invalid call changes nothing.
 *   - Pointers named *_dev are device pointers of the current CUDA device;
 *     the caller owns them (typically PyTorch tensors) and keeps them alive
 *     until the work enqueued on `stream` has finished.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Calls documented "async" only enqueue work on it.
 *   - Channel ids are uint16, so I <= 65535.
 *   - Device-side waits are bounded; a wait that runs out sets a device
 *     status word (DUO_ETIMEOUT).  Every packed handle has its own word,
 *     written by the launches whose first handle it is and read by
 *     duo_packed_status(); duo_device_status() reads every word of the
 *     device at once.
 *   - There is no host fallback: without a usable CUDA device every compute
 *     entry point returns DUO_ECUDA.
 */
#ifndef DUO_H
#define DUO_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DUO_ABI_VERSION 1

/* Status codes. */
enum {
    DUO_OK = 0,
    DUO_EINVAL = -1,    /* bad argument: NULL, size, alignment, dead handle */
    DUO_ENOMEM = -2,    /* device allocation failed (nothing leaked) */
    DUO_ECUDA = -3,     /* a CUDA runtime call failed or no device */
    DUO_ERANGE = -4,    /* a size exceeds what the format can index */
    DUO_EFORMAT = -5,   /* handle format does not support the call */
    DUO_ETIMEOUT = -6   /* a bounded device-side wait ran out */
};

/* Packed weight formats (the paper fixes none: §4.1 only says each weight
 * column is stored compressed; both layouts below are this library's). */
enum {
    DUO_FMT_IDX16 = 0,      /* per channel: fp16 non-zeros + uint16 row ids */
    DUO_FMT_BITMASK = 1,    /* "CMB": per (channel, 1024-row segment) a 128-byte
                               row bitmask followed by the fp16 non-zeros */
    DUO_FMT_BITMASK_Q8 = 2, /* CMB with 8-bit RTN codes in place of the fp16
                               non-zeros, plus a table of grids (see duo_pack) */
    DUO_FMT_BITMASK_Q4 = 3  /* the same with 4-bit codes, two per byte */
};

/* Opaque packed weight, owned by the library from duo_pack to duo_free. */
typedef struct duo_packed duo_packed;

/*
 * duo_pack -- compress a pruned weight into channel-major storage
 * (§4.1: "only the compressed model parameters are loaded"; §3 footnote:
 * weights are stored column-major, i.e. one run per input channel).
 *
 *   W_fp16_dev : device, fp16, row-major O x I with leading dimension ldw
 *                (element (r, j) at W[r * ldw + j]); entries equal to +0 or
 *                -0 are pruned, every other entry is stored bit-exactly.
 *   out, in    : O >= 1 and 1 <= I <= 65535; IDX16 also needs O <= 65536.
 *   ldw        : >= in.
 *   fmt        : DUO_FMT_BITMASK, DUO_FMT_BITMASK_Q8, DUO_FMT_BITMASK_Q4 or
 *                DUO_FMT_IDX16.
 *   stream     : work is enqueued on it and the call synchronises it before
 *                returning (the packed size must be known to allocate).
 *   h_out      : receives the new handle; untouched on error.
 *
 * BITMASK layout (normative): S = ceil(O / 1024) row segments; for input
 * channel j (outer) and segment s (inner) a record at byte 16 * off[j*S + s]
 * of the data buffer: 32 little-endian uint32 mask words (bit b of word w set
 * iff W[s*1024 + 32*w + b, j] != 0; rows >= O give 0), then those entries'
 * fp16 bit patterns in increasing row order, zero padded to 16 bytes.
 * off is uint32[I*S + 1]; off[I*S] is the total size in 16-byte units.
 *
 * BITMASK_Q8 / _Q4 layout (§5, weight-only quantisation with channel-wise
 * RTN and group size 128, Table 4; the grid is this library's reading of it):
 * each (row i, group g of input channels 128g .. 128g+127) has the
 * asymmetric min-max grid lo = min(0, min W), hi = max(0, max W) over the
 * group's stored weights, s = fp16((hi - lo) / (2^b - 1)) from an fp64
 * quotient (1 if the group stores nothing, 2^-24 if the quotient rounds to
 * 0), z = rint(-lo / s) clamped to [0, 2^b - 1]; a stored weight w becomes
 * q = clamp(rint(w / s) + z, 0, 2^b - 1) (fp64 quotient, ties to even) and
 * stands for s (q - z).  Records are as for BITMASK with the codes in place
 * of the fp16 values: one byte each (Q8) or two per byte, the n-th code of
 * the record in byte n / 2, low nibble first (Q4).  The grids are the aux
 * buffer: uint32 entries s_bits | z << 16, entry ((s * G + g) * 32 + t) * 32
 * + l for row i = 1024 s + 32 l + t, G = ceil(I / 128); rows >= O hold 0.
 *
 * IDX16 layout: per channel j a block at byte colptr[j]: cnt[j] fp16
 * non-zeros (increasing row), zero padded to 16 bytes, then their uint16 row
 * ids, zero padded to 16 bytes.  colptr is uint64[I + 1], cnt is uint32[I].
 *
 * Errors: DUO_EINVAL (NULL, sizes, ldw, fmt), DUO_ERANGE (format limits),
 * DUO_ENOMEM, DUO_ECUDA.
 */
int duo_pack(const void* W_fp16_dev, int64_t out, int64_t in, int64_t ldw,
             int fmt, void* stream, duo_packed** h_out);

/*
 * duo_sparsify -- the activation mask of §3: keep the k channels of largest
 * |x_i| (equal magnitudes: the lower index is kept first; +0 and -0 have
 * magnitude 0; NaN orders above Inf by bit pattern).  Async.
 *
 *   x_fp16_dev        : device, fp16[in].
 *   in                : 1..65535.   k : 0..in.
 *   kept_idx_dev      : device, uint16[k]: the kept channel ids, ascending.
 *   kept_val_fp16_dev : device, fp16[k]: x at those ids, bit-exact.
 * Errors: DUO_EINVAL, DUO_ECUDA.
 */
int duo_sparsify(const void* x_fp16_dev, int64_t in, int64_t k,
                 uint16_t* kept_idx_dev, void* kept_val_fp16_dev, void* stream);

/*
 * duo_spmspv -- y = W (x ⊙ m^x) over the packed weight (§3, §4.1).  Async.
 *
 * Two modes:
 *   fused   : kept_idx_dev == kept_val_fp16_dev == NULL.  The kernel selects
 *             the k largest-|x| channels itself (same rule as duo_sparsify)
 *             from x_fp16_dev (device fp16[in]) and streams only their
 *             compressed columns.
 *   listed  : kept_idx_dev (uint16[k], distinct ids < in, any order) and
 *             kept_val_fp16_dev (fp16[k]) give the sparse input directly;
 *             x_fp16_dev is ignored and may be NULL.  For BITMASK_Q8 / _Q4
 *             handles the ids must not decrease in id / 128 (ascending ids
 *             do); a list out of that order is rejected on the device
 *             (duo_packed_status(h) then returns DUO_EFORMAT).
 *   coded   : BITMASK_Q8 / _Q4 handles need every (handle, 1024-row
 *             segment) pair of the call to have an SM of its own (at most
 *             one per SM of the device, e.g. 152 on a GB300): DUO_ERANGE
 *             otherwise.  y sums the dequantised weights s (q - z).
 *   k == 0  : y = 0; the input pointers are not read and may be NULL.
 *   y_dev   : device fp32[O], 16-byte aligned; fully overwritten.  Summation
 *             order is not fixed, so y is reproducible only to fp32 rounding.
 * Errors: DUO_EINVAL (NULL, alignment, k, dead handle), DUO_ERANGE,
 * DUO_ECUDA.
 */
/* Concurrency: calls whose first handle is the same must be ordered on the
 * GPU (same stream, or otherwise synchronised): the bitmask kernel keeps a
 * small grid-barrier state with that handle. */
int duo_spmspv(const duo_packed* h, const void* x_fp16_dev,
               const uint16_t* kept_idx_dev, const void* kept_val_fp16_dev,
               int64_t k, float* y_dev, void* stream);

/*
 * duo_spmspv_multi -- n (1..4) products that share one sparse input, in one
 * launch and with one selection: y_p = W_p (x ⊙ m^x) for p < n.  In a
 * decoder layer the q/k/v projections read the same input, as do gate/up
 * (the per-layer linear layers of §5's LLaMA models).  All handles must be
 * DUO_FMT_BITMASK with the same I; O may differ.  Arguments as in
 * duo_spmspv, with ys_dev[p] the output of handle hs[p].  Async.
 */
int duo_spmspv_multi(const duo_packed* const* hs, int n, const void* x_fp16_dev,
                     const uint16_t* kept_idx_dev, const void* kept_val_fp16_dev,
                     int64_t k, float* const* ys_dev, void* stream);

/*
 * Threshold mask (§5, "compatibility with threshold-based activation
 * sparsity", Table 3(b)): instead of the k largest magnitudes, keep every
 * channel whose magnitude is strictly above a threshold fixed beforehand for
 * the layer (calibrated offline for a target sparsity); the number kept then
 * depends on x.  tau_fp16 is the threshold as fp16 bits; its sign is ignored
 * (channel j is kept iff (x_j bits & 0x7FFF) > (tau bits & 0x7FFF), i.e.
 * |x_j| > |tau| for non-NaN values).
 *
 * duo_sparsify_threshold -- the kept channels, ascending.  Async.
 *   x_fp16_dev        : device, fp16[in], 1 <= in <= 65535.
 *   kept_idx_dev      : device, uint16[in]: room for every channel; the
 *                       first *count_dev entries are written.
 *   kept_val_fp16_dev : device, fp16[in]: x at those ids, bit-exact.
 *   count_dev         : device, int32: the number kept.
 * Errors: DUO_EINVAL (NULL, size, alignment), DUO_ECUDA.
 */
int duo_sparsify_threshold(const void* x_fp16_dev, int64_t in, uint16_t tau_fp16,
                           uint16_t* kept_idx_dev, void* kept_val_fp16_dev, int32_t* count_dev,
                           void* stream);

/*
 * duo_spmspv_threshold -- y_p = W_p (x ⊙ m^x) for n (1..4) DUO_FMT_BITMASK
 * handles with the same I, with the threshold mask above computed inside
 * the launch (each CTA takes a channel range of one (product, segment) run
 * and keeps the channels above the threshold in it: no ranking across the
 * vector).  ys_dev[p]: device fp32[O_p], 16-byte aligned, fully overwritten.
 * Async; same ordering rule as duo_spmspv for calls sharing a first handle.
 * Errors: DUO_EINVAL, DUO_EFORMAT (not BITMASK), DUO_ERANGE (more (product,
 * segment) runs than SMs), DUO_ECUDA.
 */
int duo_spmspv_threshold(const duo_packed* const* hs, int n, const void* x_fp16_dev,
                         uint16_t tau_fp16, float* const* ys_dev, void* stream);

/* duo_free -- release a handle and its device memory.  NULL is a no-op
 * (DUO_OK); a handle that is not live (already freed, never created)
 * returns DUO_EINVAL without touching memory.  Synchronises the device
 * memory release with cudaFree semantics. */
int duo_free(duo_packed* h);

/* Describes a live handle.  Pointers stay owned by the handle.
 *   BITMASK: index = uint32 off[I*S+1], aux = NULL.
 *   BITMASK_Q8 / _Q4: index = uint32 off[I*S+1], aux = uint32 grids
 *            [S][ceil(I/128)][1024] (layout under duo_pack).
 *   IDX16  : index = uint64 colptr[I+1], aux = uint32 cnt[I]. */
typedef struct duo_packed_info {
    int32_t fmt;
    int32_t version;
    uint32_t magic;          /* "CMB1" or "IDX0" little-endian */
    int32_t seg_rows;        /* 1024 for BITMASK, 0 for IDX16 */
    int64_t out, in, nseg, nnz;
    const void* index_dev; int64_t index_bytes;
    const void* aux_dev;   int64_t aux_bytes;
    const void* data_dev;  int64_t data_bytes;
} duo_packed_info;

int duo_packed_query(const duo_packed* h, duo_packed_info* info);

/* Copies one buffer of a live handle to host memory (synchronous), e.g. to
 * save a packed weight or to compare its bytes with a reference packer.
 *   which : 0 = index, 1 = aux, 2 = data (as described by duo_packed_info).
 *   dst_host, bytes : host destination; bytes must equal the buffer size
 *                     (dst_host may be NULL when that size is 0).
 * Errors: DUO_EINVAL (dead handle, which, NULL dst, size mismatch), DUO_ECUDA. */
int duo_packed_export(const duo_packed* h, int which, void* dst_host, int64_t bytes);

/*
 * duo_pack_cmb_noalloc -- the bitmask packing of duo_pack (same bytes)
 * without any device allocation.  The paper has no counterpart: this entry
 * point exists for callers that cannot call cudaMalloc themselves, such as
 * an engine that hands out all device memory from its own pool, or a
 * process whose device allocations someone else accounts for.  duo_pack
 * needs per-record scratch and allocates it (and the packed buffers); this
 * variant writes into buffers the caller provides and keeps its scratch in a
 * fixed file-scope device array of the library.
 *
 *   W_fp16_dev, out, in, ldw : as in duo_pack.
 *   off_dev       : device, uint32[in * ceil(out/1024) + 1], 4-byte aligned:
 *                   receives the record offsets (16-byte units).
 *   data_dev      : device, 16-byte aligned, data_capacity bytes: receives
 *                   the records.  NULL asks only for the size.
 *   data_bytes    : host out: the packed data size in bytes.
 *   stream        : work is enqueued on it; the call synchronises it.
 *
 * Limits and behaviour:
 *   - in * ceil(out/1024) must not exceed DUO_NOALLOC_MAX_RECORDS (the
 *     scratch holds one 32-bit count per record), else DUO_ERANGE; so must
 *     in > 65535 or ceil(out/1024) > 65535, as in duo_pack;
 *   - W_fp16_dev, off_dev and (when given) data_dev must be device or
 *     managed memory, else DUO_EINVAL (checked before any device work);
 *   - data_capacity smaller than the packed size: DUO_ERANGE, with
 *     *data_bytes set to the size needed;
 *   - calls no cudaMalloc, cudaFree or other allocating routine;
 *   - the scratch array (about 1 MiB) is held by every GPU that loads the
 *     library until the process exits; every call shares it and the previous
 *     call's contents are never read, but calls that overlap on the GPU
 *     (concurrent calls from several threads or streams) race on it;
 *   - the first call on a device looks up the array's device address with
 *     that device current; make that first call before any stream capture
 *     (the call synchronises its stream and cannot be captured anyway).
 * Errors: DUO_EINVAL, DUO_ERANGE, DUO_ECUDA.
 */
#define DUO_NOALLOC_MAX_RECORDS 262144
int duo_pack_cmb_noalloc(const void* W_fp16_dev, int64_t out, int64_t in, int64_t ldw,
                         uint32_t* off_dev, void* data_dev, int64_t data_capacity,
                         int64_t* data_bytes, void* stream);

/*
 * duo_copy -- copies `bytes` bytes from src to dst with a kernel on the SMs
 * (asynchronous on `stream`, a cudaStream_t passed as void*).  Each pointer
 * is device memory of the current device, managed memory, or page-locked host
 * memory mapped into the device's address space (cudaHostAlloc /
 * cudaHostRegister memory on a system with unified addressing); the caller
 * owns both, and both ranges must lie inside their allocations and not
 * overlap.  Any alignment; 16-byte aligned ends copy in 16-byte words.  Not a
 * step of the method: it moves a decode step's inputs in and outputs out
 * without a copy-engine node, the cheaper choice inside a captured step.
 * The kernel first waits for the stream's previous kernel to complete.
 * Errors: DUO_EINVAL (NULL, bytes < 0, a pointer the device cannot reach:
 * unregistered host memory, another device's memory), DUO_ECUDA (no device,
 * launch).  bytes = 0 returns DUO_OK at once (NULL pointers allowed).
 */
int duo_copy(void* dst, const void* src, int64_t bytes, void* stream);

/* Synchronises `stream`, returns and clears the device status words of the
 * current device (the process-wide word and the word of every live handle
 * on it): DUO_OK; DUO_ETIMEOUT if a bounded device wait ran out since the
 * words were last read; DUO_EFORMAT if a kernel met a record size or channel
 * id outside the format's bounds (the affected work was skipped); DUO_ECUDA
 * if the stream reports an error. */
int duo_device_status(void* stream);

/* duo_packed_status -- the same for one handle's word only: the status of
 * the launches whose first (or only) handle h is, since the word was last
 * read.  Synchronises `stream`.  Launches on other handles, or on other
 * streams, do not report here.  Errors: DUO_EINVAL (NULL or freed h),
 * DUO_ECUDA. */
int duo_packed_status(const duo_packed* h, void* stream);

/* Text of a status code (static storage). */
const char* duo_strerror(int code);

/* DUO_ABI_VERSION of the loaded library. */
int duo_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DUO_H */
