/*
 * bsr.h -- C ABI of the GB300 (sm_103a) block-sparse-row x dense product.
 *
 * Section 2.2 of "Algorithm to Compilation Co-design: An Integrated View of
 * Neural Network Sparsity" (Guo and Huang, 2021) stores a pruned weight
 * W[M, K] in Block Sparse Row form -- block values, block column indices and
 * block-row pointers, following SciPy -- and multiplies only the kept blocks
 * with the input tensor. Eq. 3 partitions W into blocks; here a block is
 * R x C: R consecutive rows of W (output features) by C consecutive columns
 * (input features). MB = M/R block rows, KB = K/C block columns.
 *
 *   indptr[MB+1]     int32, indptr[0] = 0, non-decreasing, indptr[MB] = nnzb
 *   indices[nnzb]    int32 block-column index, strictly ascending inside a row
 *   data[nnzb][R][C] block values, row-major inside each block
 *
 * The product (the paper's linear/attention projection, Y = X W^T + b):
 *   Y[n, i*R + r] = bias[i*R + r]
 *                 + sum_{p = indptr[i]}^{indptr[i+1]-1} sum_{c<C} X[n, indices[p]*C + c] * data[p][r][c]
 * with X[N, K] and Y[N, M] row-major. Element types: BSR_F32 (fp32 data, X
 * and Y, fp32 accumulation) or BSR_BF16 (bf16 data, X and Y, fp32
 * accumulation, Y rounded to nearest even). bias is always fp32 or NULL.
 * Plain TF32 is never used for BSR_F32. fp32 blocks of 32 or more rows with
 * 16 or 32 columns, and 16-row blocks of such width in weights of at least
 * 2^20 elements (M K), run on the tensor cores as 3xTF32: each operand is split
 * into a tf32 high part and a tf32 low part (the remainder) and the product is
 * hi*hi + hi*lo + lo*hi, accumulated in fp32. The dropped lo*lo term and the
 * rounding of the low parts leave a relative error near 2^-20 per product,
 * inside the fp32 tolerance |dY| <= 1e-5 * (sum |x||w| + |b|). Calls of 512
 * or more tokens on fp32 blocks that only the generic kernel would take
 * otherwise (64 or 128 rows with 1 to 8 columns) run on the gathered-K
 * tensor-core kernel, 3xTF32 in the same way. Every other fp32 shape
 * multiplies in plain fp32 FMA.
 *
 * Conventions.
 *  - Every call returns a status; the library never aborts, prints or traps.
 *  - Pointers marked "device" are global-memory pointers of the device that
 *    was current when the handle was created (for bsr_from_dense: the
 *    current device).
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *    stream). Work is enqueued on it; calls say when they synchronise.
 *  - Supported shapes: 1 <= R, C and R*C <= 4096, M % R == 0, K % C == 0,
 *    MB + 1, KB and nnzb below 2^31.
 *  - One handle must not run bsr_spmm on two streams at once (the split-row
 *    workspace and staging buffers belong to the handle).
 */
#ifndef BSR_H
#define BSR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    BSR_OK = 0,
    BSR_ERR_INVALID_ARG = 1, /* NULL where a pointer is needed, negative size, aliasing, bad threshold */
    BSR_ERR_SHAPE = 2,       /* M % R or K % C non-zero, sizes beyond int32 indexing */
    BSR_ERR_UNSUPPORTED = 3, /* block shape or dtype not supported */
    BSR_ERR_CAPACITY = 4,    /* output arrays of bsr_from_dense too small */
    BSR_ERR_STRUCTURE = 5,   /* indptr/indices are not a canonical BSR structure */
    BSR_ERR_ALIGNMENT = 6,   /* X or Y not 16-byte aligned, bias not 4-byte aligned */
    BSR_ERR_CUDA = 7,        /* a CUDA runtime call or kernel launch failed */
    BSR_ERR_TIMEOUT = 8,     /* a bounded device-side wait gave up (reported by bsr_check_device_status) */
    BSR_ERR_ALLOC = 9        /* device or host allocation failed */
} bsr_status_t;

typedef enum { BSR_F32 = 0, BSR_BF16 = 1 } bsr_dtype_t;

typedef struct bsr_handle_s *bsr_handle_t;
typedef struct bsr_plan_s *bsr_plan_t;

/*
 * bsr_from_dense -- build the BSR arrays of a dense weight on the GPU
 * (Section 2.2: "data values, indices, and indptr").
 *
 * W        device, [M, K] row-major, element type dt.
 * R, C     block shape. threshold: a block is kept iff at least one element
 *          w has !(|w| <= threshold) in fp32 (so NaN keeps its block, -0.0
 *          never does). threshold must be >= 0 and not NaN.
 * indptr   device, MB+1 int32, always written on success and on CAPACITY.
 * indices  device, capacity_blocks int32; data: device, capacity_blocks*R*C
 *          elements. Kept blocks appear in ascending column order per row,
 *          their values copied bit for bit (sub-threshold values included).
 * Query:   indices == NULL, data == NULL, capacity_blocks == 0 -> BSR_OK,
 *          *nnzb_out = number of kept blocks, only indptr written.
 * If capacity_blocks < nnzb: BSR_ERR_CAPACITY, *nnzb_out set, indices/data
 *          untouched. nnzb_out (host) may be NULL.
 * Synchronises `stream` once (to read nnzb). Temporary device memory is
 * allocated and freed inside the call.
 */
bsr_status_t bsr_from_dense(const void *W, int64_t M, int64_t K, int R, int C, float threshold,
                            bsr_dtype_t dt, int32_t *indptr, int32_t *indices, void *data,
                            int64_t capacity_blocks, int64_t *nnzb_out, void *stream);

/*
 * bsr_create -- analyse a BSR structure and build its execution schedule
 * (the counterpart of the paper's task buffer and auto-scheduler, Section
 * 2.2: tasks with identical structure are reused).
 *
 * indptr, indices, data: device arrays as described above. They are
 * BORROWED: the caller keeps them alive and unmodified until bsr_destroy.
 * Validates the structure on the host (one device-to-host copy of indptr and
 * indices, synchronous): indptr[0] == 0, non-decreasing, indices strictly
 * ascending per row and < K/C; otherwise BSR_ERR_STRUCTURE.
 * Owns: the schedule (shared with other handles of identical structure),
 * the work list, a repacked copy of data in the kernels' layout, a device
 * status word and workspaces. *out receives the handle.
 */
bsr_status_t bsr_create(const int32_t *indptr, const int32_t *indices, const void *data, int R,
                        int C, int64_t M, int64_t K, bsr_dtype_t dt, bsr_handle_t *out);

/*
 * bsr_reserve -- size the handle's workspaces for up to N_max tokens so that
 * later bsr_spmm calls with N <= N_max allocate nothing (needed before
 * capturing bsr_spmm in a CUDA graph). Synchronous.
 */
bsr_status_t bsr_reserve(bsr_handle_t h, int64_t N_max);

/*
 * bsr_spmm -- Y[N, M] = X[N, K] W^T + bias[M] over the kept blocks.
 *
 * X, Y     row-major, element type of the handle, 16-byte aligned, not
 *          overlapping (else BSR_ERR_ALIGNMENT / BSR_ERR_INVALID_ARG).
 *          Both device pointers, or both host pointers: with host pointers
 *          the call copies X in and Y out on `stream` through device staging
 *          buffers owned by the handle; Y is valid once `stream` has
 *          synchronised.
 * bias     device, fp32 [M], or NULL for zero.
 * N        tokens; N == 0 is a no-op returning BSR_OK.
 * Asynchronous on `stream`; never synchronises unless a workspace must grow
 * beyond what bsr_reserve sized (then it allocates). Kernel launch failures
 * return BSR_ERR_CUDA.
 */
bsr_status_t bsr_spmm(bsr_handle_t h, const void *X, const float *bias, void *Y, int64_t N,
                      void *stream);

/*
 * bsr_check_device_status -- synchronise the device and return the first
 * error a kernel of this handle recorded (BSR_ERR_TIMEOUT when a bounded
 * wait gave up), then clear it. BSR_OK if none. Structure errors are not
 * reported here: bsr_create validates indptr/indices on the host and the
 * kernels read only the handle's own repacked copy, built from the
 * validated structure.
 */
bsr_status_t bsr_check_device_status(bsr_handle_t h);

/*
 * bsr_get_schedule -- a text description of the handle's schedule: kernel
 * variant, execution block height and width (exec_R x exec_C: max(R, 16) x 64
 * where small or narrow bf16 blocks run on the tensor cores as zero-filled
 * tiles), tile sizes, work items, split
 * rows, launches per call, the schedule-cache statistics and the task sizes
 * each kernel can run (items per CTA; the size a call uses is chosen per
 * call from its token count), as "key=value" lines. Writes at most len bytes
 * including the terminating NUL into buf (truncating). Returns
 * BSR_ERR_INVALID_ARG for a NULL handle or buffer.
 */
bsr_status_t bsr_get_schedule(bsr_handle_t h, char *buf, size_t len);

/*
 * bsr_spmm_noalloc -- bsr_spmm for callers that cannot allocate device memory.
 *
 * The paper has no counterpart: this is a deployment aid. Some callers may
 * not call cudaMalloc at the point where they run the product: code inside
 * a CUDA graph capture (allocation there is not allowed), code bound to a
 * fixed memory budget or to its own allocator, and latency-critical loops
 * where an allocation's implicit device synchronisation is unacceptable.
 * bsr_spmm allocates when a call needs more split-row workspace than the
 * handle holds; this entry point never does.
 *
 * Same product and arguments as bsr_spmm, except that X and Y must be device
 * pointers (host buffers would need staging memory: BSR_ERR_INVALID_ARG).
 * The fp32 partial tiles of block rows that the schedule splits across CTAs
 * go to one scratch array compiled into the library, of
 * BSR_NOALLOC_SCRATCH_BYTES bytes, which every GPU that loads the library
 * holds until the process exits. A call needs slots * N * exec_R * 4 bytes
 * of it ("slots" and "exec_R" as reported by bsr_get_schedule; exec_R is the
 * block height the kernels run, 16 for small or narrow bf16 blocks re-blocked
 * for the tensor cores, else R); a larger call returns BSR_ERR_CAPACITY and
 * launches nothing.
 * The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress, with that device current) and keeps it: make that
 * first call before any stream capture. All calls share the one array, so
 * calls whose kernels may run at the same time on the GPU (on streams with
 * no ordering between them) race and produce wrong results. The array keeps
 * the last call's contents; every element a call reads is written earlier
 * in the same call, so nothing is cleared.
 * Calls no cudaMalloc, cudaFree or allocating library routine.
 */
#define BSR_NOALLOC_SCRATCH_BYTES (32u << 20)
bsr_status_t bsr_spmm_noalloc(bsr_handle_t h, const void *X, const float *bias, void *Y, int64_t N,
                              void *stream);

/*
 * bsr_spmm_batch -- n products that share one input: Y_i = X · W_iᵀ + b_i.
 *
 * The paper prunes BERT (Section 2.3), whose self-attention applies several
 * weights (query, key, value) to the same activations; this entry point takes
 * such products together. Products whose weights run on the same kernel
 * configuration -- the SIMT kernel with the same dtype, block shape and task
 * layout for the call's N, or the tensor-core kernel with the same dtype and
 * block height -- are fused into one grid, up to 64 per launch, so one
 * product's last, partly filled wave overlaps the others' work; products on
 * the generic kernel run one after another on the same stream. Each output
 * is bit-identical to what bsr_spmm gives for the same arguments.
 *
 *   handles[n]  distinct handles, all on one device, one dtype and one K;
 *               BSR_ERR_INVALID_ARG for a NULL or repeated handle or a device
 *               or dtype mismatch, BSR_ERR_SHAPE for a K mismatch.
 *   X           device, [N, K] row-major, 16-byte aligned; read by all.
 *   biases      NULL (no bias anywhere) or n entries, each NULL or a device
 *               fp32 [M_i] array (4-byte aligned).
 *   Ys[n]       device, [N, M_i] row-major, 16-byte aligned; no output may
 *               overlap X, a bias or another output (BSR_ERR_INVALID_ARG).
 *   N           tokens; n == 0 or N == 0 is a no-op returning BSR_OK.
 *   stream      as in bsr_spmm. Host buffers are not accepted (BSR_ERR_INVALID_ARG).
 *
 * Asynchronous; like bsr_spmm it may grow a handle's split-row workspace (with
 * one stream synchronisation) unless bsr_reserve sized it for N beforehand.
 */
bsr_status_t bsr_spmm_batch(const bsr_handle_t *handles, int n, const void *X, const float *const *biases,
                            void *const *Ys, int64_t N, void *stream);

/*
 * bsr_plan_create -- a fixed sequence of n products, Y_i = X_i · W_iᵀ + b_i,
 * captured once into a CUDA graph that bsr_plan_launch replays.
 *
 * Section 2.2: the task scheduler keeps BSR tasks in a buffer, reuses
 * identical tasks and schedules similar ones next to each other. Identical
 * structures already share one schedule (bsr_create's cache); a plan adds the
 * adjacency for a whole sequence, such as every projection of a BERT model
 * (Section 2.3), and removes the per-call host work: validation, workspace
 * sizing and launch set-up happen here, once.
 *
 *   handles[n]   the weights (a handle may appear more than once); all on the
 *                current device, which must be the one they were created on.
 *                Each must outlive the plan (the plan uses its block values
 *                and status word); the plan owns its split-row workspaces, so
 *                later bsr_spmm calls on the same handles do not disturb it.
 *   X[n]         device, [N_i, K_i] row-major, 16-byte aligned.
 *   biases       NULL (no bias) or n entries, each NULL or device fp32 [M_i].
 *   Y[n]         device, [N_i, M_i] row-major, 16-byte aligned; Y_i must not
 *                overlap X_i or b_i.
 *   N[n]         tokens per product (>= 0; 0 is a no-op product).
 *   independent  0: the products run in the given order, one call each, so a
 *                later X may be an earlier Y (a chain of layers).
 *                1: the caller states that no product reads what another
 *                writes -- checked: no Y_i may overlap any X_j, b_j or other
 *                Y_j (BSR_ERR_INVALID_ARG otherwise) -- and the plan may
 *                reorder: products that share X and N are grouped in first-
 *                appearance order of their X, inside a group products whose
 *                kernels share a template come next to each other (handles
 *                that share a schedule adjacent) and run as fused grids as in
 *                bsr_spmm_batch (a handle repeated inside a group starts a new
 *                fused call). Outputs are bit-identical to bsr_spmm calls.
 *   out          receives the plan.
 *
 * The buffers are bound at capture: a replay reads the current contents of
 * X_i and b_i and writes Y_i. Synchronous (allocates the workspaces, captures
 * on a private stream); enqueues no device work. Errors: BSR_ERR_INVALID_ARG
 * (NULL, negative N, aliasing, host or foreign-device pointers),
 * BSR_ERR_ALIGNMENT, BSR_ERR_ALLOC, BSR_ERR_CUDA (capture or instantiation).
 */
bsr_status_t bsr_plan_create(const bsr_handle_t *handles, const void *const *X, const float *const *biases,
                             void *const *Y, const int64_t *N, int n, int independent, bsr_plan_t *out);

/* bsr_plan_launch -- replay the plan's graph on `stream` (asynchronous; the
 * products' device-side errors are reported per handle by
 * bsr_check_device_status). Two replays of one plan must not overlap in time
 * (they share the plan's workspaces). */
bsr_status_t bsr_plan_launch(bsr_plan_t plan, void *stream);

/* bsr_plan_get_order -- what the plan runs: order[k] = the product executed
 * k-th and call[k] = the index of the library call (one bsr_spmm, or one
 * fused bsr_spmm_batch group) that runs it, for k < n; products with N = 0
 * run nothing and are not listed, entries past the executed products are -1
 * (either array may be NULL); *n_kernels (if not NULL) = the kernel launches
 * in the graph. */
bsr_status_t bsr_plan_get_order(bsr_plan_t plan, int *order, int *call, int n, int *n_kernels);

/* bsr_plan_destroy -- release the graph and the workspaces. NULL is a no-op. */
void bsr_plan_destroy(bsr_plan_t plan);

/* bsr_destroy -- release what the handle owns (not the borrowed arrays). NULL is a no-op. */
void bsr_destroy(bsr_handle_t h);

/* bsr_status_str -- a static, human-readable name for a status code. */
const char *bsr_status_str(bsr_status_t s);

#ifdef __cplusplus
}
#endif
#endif /* BSR_H */
