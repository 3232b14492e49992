/*
 * sfc_gemm.h -- C ABI of the space-filling-curve (SFC) bf16 GEMM for GB300.
 *
 * The library computes C = A * B (A: M x K, B: K x N, C: M x N, all row-major)
 * the way Sec. II-D and Listing 1 of "Space Filling Curves is All You Need:
 * Communication-Avoiding Matrix Multiplication Made Simple" describe it:
 *
 *   - the output is blocked into bm x bn tiles, an Mt x Nt grid (Sec. II-A);
 *   - the tiles are ordered along a generalized Hilbert curve that works for
 *     any grid shape (Sec. II-B, Fig. 2);
 *   - the task space of Mt*Nt*ca_c items is handed to the workers in contiguous
 *     blocks; item i belongs to K layer i / (Mt*Nt) and curve position
 *     i % (Mt*Nt) (Listing 1, the parallel loop and its index arithmetic);
 *   - with ca_c > 1 ("K_layers", the replication factor c of the 2.5D/3D
 *     communication-avoiding scheme, Sec. II-C/II-D) each layer contracts its
 *     own share of K into an fp32 copy of C, and the copies are summed at the
 *     end in layer order 0..c-1 (Listing 1, the final reduction).
 *
 * Here a worker is a CUDA thread block resident on one SM of a persistent
 * kernel; the tile contraction (the paper's batch-reduce GEMM, Sec. II-A) runs
 * on the tcgen05 tensor cores with fp32 accumulation in tensor memory.
 *
 * Conventions for every entry point:
 *   - sizes and leading dimensions are in ELEMENTS; lda >= K, ldb >= N, ldc >= N;
 *   - A, B, C and workspace are DEVICE pointers owned by the caller (HOST
 *     pointers for sfc_gemm_host); the library never frees them and keeps no
 *     reference after the call's work has completed;
 *   - calls that take a stream are asynchronous on that stream (NULL = the
 *     legacy default stream); arguments are validated on the host first and a
 *     validation error launches nothing;
 *   - every function returns an sfc_status_t (0 = success) unless noted.
 *
 * Thread safety: entry points may be called from several host threads; after
 * a one-time per-device set-up the state calls share is either immutable or
 * guarded (the table of tuned shapes, the staging slots of sfc_gemm_host).
 * Kernels in flight at the same time -- on several streams, or replays of
 * captured graphs -- share no device state but the error word that
 * sfc_get_device_status reads: the counter from which a call's workers take
 * their items (SFC_ASSIGN_WAVE / AUTO) is memory of that call, taken from a
 * stream-ordered pool of the library and freed after the call's kernels
 * (sfc_gemm_noalloc: its scratch area).
 */
#ifndef SFC_GEMM_H
#define SFC_GEMM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    SFC_OK = 0,
    SFC_ERR_INVALID_ARG = -1,  /* bad size, null pointer, bad enum, ca_c out of range  */
    SFC_ERR_UNALIGNED = -2,    /* an element, bias or workspace misaligned (see each call)    */
    SFC_ERR_WORKSPACE = -3,    /* workspace smaller than sfc_gemm_workspace_size(...)  */
    SFC_ERR_CUDA = -4,         /* a CUDA runtime call failed (see sfc_last_cuda_error) */
    SFC_ERR_TIMEOUT = -5,      /* a device-side wait gave up (reported by sfc_get_device_status) */
    SFC_ERR_UNSUPPORTED = -6   /* no usable sm_103 device, or an option this build lacks */
} sfc_status_t;

typedef enum { SFC_F32 = 0, SFC_BF16 = 1 } sfc_dtype_t;

/* Storage of B (sfc_gemm_ex2).  KN: B is K x N row-major, the paper's
 * statement of the problem (Sec. II-A).  NK: the caller holds B transposed,
 * N x K row-major (a linear layer's weight matrix); the kernels then load B
 * K-major like A.  Not part of the paper, which fixes the KN layout. */
typedef enum { SFC_B_KN = 0, SFC_B_NK = 1 } sfc_b_layout_t;

/* Element type of A and B (sfc_gemm_ex2): bf16, or one of the two 8-bit float
 * formats (e4m3: 4 exponent bits, bias 7, no infinities; e5m2: 5 exponent
 * bits, bias 15).  The paper notes the method is independent of the data type
 * and evaluates bf16 (Sec. III, Sec. IV-A); the 8-bit kinds use the tensor
 * cores' 8-bit path (32 values of k per instruction) with fp32 accumulation. */
typedef enum { SFC_AB_BF16 = 0, SFC_AB_E4M3 = 1, SFC_AB_E5M2 = 2 } sfc_ab_t;

/* Order of the output tiles along which workers take their items.
 * SFC:    generalized Hilbert curve (Sec. II-B) -- the method.
 * RASTER: row-major tile order s -> (s / Nt, s % Nt), a comparison baseline. */
typedef enum { SFC_ORDER_SFC = 0, SFC_ORDER_RASTER = 1 } sfc_order_t;

/* How items are dealt to the P persistent workers.
 * SEGMENT:     worker p takes the contiguous block [p*W/P, (p+1)*W/P) of the W
 *              items, the static block partition of Listing 1's parallel loop.
 * WAVE:        each worker, when free, takes the next curve position from a
 *              counter shared by the launch, so the tiles running at any time
 *              are consecutive curve positions -- a compact patch of the grid
 *              whose A/B panels are shared through L2 -- however the workers'
 *              speeds drift.
 * WAVE_STATIC: worker p takes items p, p+P, p+2P, ... (the same deal decided
 *              up front; kept for comparison).
 * AUTO:        the library picks (currently WAVE). */
typedef enum {
    SFC_ASSIGN_SEGMENT = 0,
    SFC_ASSIGN_WAVE = 1,
    SFC_ASSIGN_AUTO = 2,
    SFC_ASSIGN_WAVE_STATIC = 3
} sfc_assign_t;

/* Output tile shape and the hardware that computes it.
 * N128 / N256:           128 x 128 / 128 x 256 tiles, one SM each.
 * PAIR_N128 / PAIR_N256: 256 x 128 / 256 x 256 tiles computed by a pair of SMs
 *                        (a 2-CTA cluster; each SM loads half of A and half of B).
 * AUTO: the tile sfc_gemm_tune measured fastest for the shape (and layer
 * count), else the time model's pick from the tile count and the number of
 * workers.  Every tile shape gives the same bits. */
typedef enum {
    SFC_TILE_AUTO = 0,
    SFC_TILE_N128 = 128,
    SFC_TILE_N256 = 256,
    SFC_TILE_PAIR_N128 = 1128,
    SFC_TILE_PAIR_N256 = 1256
} sfc_tile_t;

/*
 * sfc_tile_order -- the curve permutation over an Mt x Nt tile grid
 * (Sec. II-B; create_sfc_map / map_sfc_index of Listing 1).
 *   out_idx: HOST array of Mt*Nt int32, filled with out_idx[s] = tm*Nt + tn for
 *            curve position s.  The curve starts at tile (0,0), consecutive
 *            positions are edge-adjacent tiles.  Host-only, no GPU needed.
 * Errors: SFC_ERR_INVALID_ARG if Mt < 1, Nt < 1, Mt*Nt > 2^31-1 or out_idx NULL.
 */
int sfc_tile_order(int Mt, int Nt, int32_t *out_idx);

/*
 * sfc_tile_order_device -- the same permutation computed by the GPU decoder
 * that the GEMM kernel itself uses (one thread per curve position).
 *   out_idx_dev: DEVICE array of Mt*Nt int32.  Asynchronous on `stream`.
 * Errors: as sfc_tile_order, plus SFC_ERR_CUDA.
 */
int sfc_tile_order_device(int Mt, int Nt, int32_t *out_idx_dev, void *stream);

/*
 * sfc_gemm_workspace_size -- bytes of fp32 workspace sfc_gemm_ex needs for the
 * ca_c partial copies of C (Listing 1's C[K_layers][...], Sec. II-D):
 * 0 when ca_c == 1, else ca_c * M * round_up(N, 4) * 4.  For ca_c == 0 (layer
 * count chosen by the library) the size for the most layers it may choose,
 * min(64, ceil(K/64), ceil(320 / (ceil(M/128) * ceil(N/128)))).  Returns 0 for
 * invalid arguments.  Needs no GPU.
 */
size_t sfc_gemm_workspace_size(int64_t M, int64_t N, int64_t K, int ca_c);

/*
 * sfc_gemm -- C = A * B with bf16 A, B, fp32 accumulation and fp32 output,
 * curve order, automatic assignment and tile width.
 *   A: bf16, M x K, row stride lda.   B: bf16, K x N, row stride ldb.
 *   C: fp32, M x N, row stride ldc.   Written, never read (beta = 0).
 *   ca_c: number of K layers, 1 <= ca_c <= min(ceil(K/64), 4096).  Layer l contracts K
 *         tiles [floor(l*Kt/ca_c), floor((l+1)*Kt/ca_c)) of the Kt = ceil(K/64)
 *         64-wide K tiles.  For ca_c > 1 the library takes its fp32 workspace
 *         from its own stream-ordered pool (allocated and freed in order on
 *         `stream`; freed memory stays in the pool for the next call until
 *         sfc_release).  ca_c = 0 lets the library choose the count (and the
 *         tile) from a model of the call's time on this device: waves of
 *         items times the length of a layer, plus the reduction's cost for
 *         more than one layer (the replication factor choice of Sec. II-D,
 *         made per call), or the count sfc_gemm_tune measured fastest for the
 *         shape; sfc_gemm_plan reports the choice.
 *   stream: a cudaStream_t passed as void*.
 * Alignment: the tile loads (Tensor Memory Accelerator) read 16-byte-aligned
 * rows.  When A or B is not 16-byte aligned, or lda / ldb is not a multiple of
 * 8, the call first copies that operand into a padded buffer taken from the
 * stream-ordered pool (one extra read and write of the operand; no counterpart
 * in the paper, whose blocked layouts are always aligned).  A and B must be
 * aligned to their element size (else SFC_ERR_UNALIGNED).  C may have any
 * alignment.
 * Accuracy: products are exact and summed in fp32; the tensor core's running
 * sum is restarted every 4096 values of k and the partial sums are added with
 * round-to-nearest fp32 adds, which bounds the error growth of very long K.
 * Memory: besides the layer workspace, a call whose items outnumber the
 * workers (dynamic dealing over more than one wave) takes a 256-byte counter
 * from the library's stream-ordered ticket pool and frees it after its kernels
 * (both kept by the pools for the next call).  The counter's words are tagged
 * with a per-call value, so nothing is written to clear it before the kernels.
 * Errors: SFC_ERR_INVALID_ARG, SFC_ERR_UNALIGNED, SFC_ERR_CUDA, SFC_ERR_UNSUPPORTED.
 */
int sfc_gemm(int64_t M, int64_t N, int64_t K,
             const void *A, const void *B, void *C,
             int64_t lda, int64_t ldb, int64_t ldc,
             int ca_c, void *stream);

/*
 * sfc_gemm_ex -- sfc_gemm with every knob exposed.
 *   c_dtype:   SFC_F32 or SFC_BF16 (bf16 output is the fp32 result rounded to
 *              nearest, ties to even).
 *   order, assign, tile: see the enums above.
 *   workspace / workspace_bytes: caller-owned DEVICE scratch of at least
 *              sfc_gemm_workspace_size(M, N, K, ca_c) bytes, 16-byte aligned;
 *              may be NULL when ca_c == 1, or NULL to use the stream-ordered
 *              pool as sfc_gemm does.  Its contents on return are unspecified.
 * Errors: as sfc_gemm, plus SFC_ERR_WORKSPACE.
 */
int sfc_gemm_ex(int64_t M, int64_t N, int64_t K,
                const void *A, const void *B, void *C,
                int64_t lda, int64_t ldb, int64_t ldc,
                int ca_c, sfc_dtype_t c_dtype,
                sfc_order_t order, sfc_assign_t assign, sfc_tile_t tile,
                void *workspace, size_t workspace_bytes, void *stream);

/*
 * sfc_gemm_ex2 -- sfc_gemm_ex extended with the input type, and with the
 * operand layout and epilogue of a BLAS-style GEMM (no counterpart in the
 * paper, which computes C = A B with C zeroed first, Listing 1):
 *     C = A B + beta * C + bias[j]     (fp32 arithmetic, then rounded to c_dtype)
 *   ab_dtype: sfc_ab_t of both A and B.  For the 8-bit kinds rows are repacked
 *             unless lda and ldb are multiples of 16, K layers split ceil(K/128) slabs of
 *             128 values of k, and the N-major (SFC_B_KN) layout is not served
 *             by SFC_TILE_PAIR_N128 (SFC_TILE_N128 is used instead).
 *   b_layout: SFC_B_KN (B is K x N, ldb >= N) or SFC_B_NK (B is stored as its
 *             transpose, N x K, ldb >= K).
 *   beta:     0 leaves C write-only (its contents may be anything, even NaN);
 *             otherwise C is read once, before it is written.
 *   bias:     NULL or N fp32 device values, 4-byte aligned, added per column.
 * With ca_c > 1 the beta and bias terms are applied by the layer reduction,
 * after the layer partials are summed; with ca_c == 1 by the GEMM epilogue.
 * Other arguments, requirements and errors as sfc_gemm_ex; ldb must be a
 * multiple of 8 in either layout, and an invalid b_layout is
 * SFC_ERR_INVALID_ARG, a misaligned bias SFC_ERR_UNALIGNED.
 */
int sfc_gemm_ex2(int64_t M, int64_t N, int64_t K,
                 const void *A, const void *B, void *C,
                 int64_t lda, int64_t ldb, int64_t ldc,
                 int ab_dtype, int b_layout, float beta, const float *bias,
                 int ca_c, sfc_dtype_t c_dtype,
                 sfc_order_t order, sfc_assign_t assign, sfc_tile_t tile,
                 void *workspace, size_t workspace_bytes, void *stream);

/*
 * sfc_gemm_ex3 -- sfc_gemm_ex2 with Listing 1's K-block loop: k_block_factor
 * passes over K (Sec. II-D; the loop over ik, whose blocks set the A and B
 * panel depth k' of Sec. II-E).  Pass ik contracts block ik of every layer's
 * K slabs -- layer l's slabs [L_l, L_(l+1)) split as
 * [L_l + floor(ik * n_l / kbf), L_l + floor((ik + 1) * n_l / kbf)), n_l =
 * L_(l+1) - L_l -- for every output tile (one launch per pass), and adds it
 * into that layer's copy of C, which stays where it is between passes: an fp32
 * C with one layer is accumulated in place (pass 0 also applies beta and
 * bias), otherwise the copies are fp32 workspace and the final reduction
 * applies beta, bias and the output rounding.  Sums are fp32, pass by pass in
 * order, so the rounding differs from k_block_factor = 1 but not between
 * orders, assignments or runs.
 *   k_block_factor: 1..64, and every layer must hold at least that many
 *     slabs (a slab is 64 values of k for bf16, 128 for the 8-bit kinds):
 *     ca_c * k_block_factor <= ceil(K / slab) for ca_c > 0; with ca_c = 0 the
 *     planner keeps to it.  1 is exactly sfc_gemm_ex2.
 *   workspace: at least sfc_gemm_workspace_size2(M, N, K, ca_c,
 *     k_block_factor, c_dtype) bytes, or NULL to use the library's pool.
 * Errors: as sfc_gemm_ex2.
 */
int sfc_gemm_ex3(int64_t M, int64_t N, int64_t K,
                 const void *A, const void *B, void *C,
                 int64_t lda, int64_t ldb, int64_t ldc,
                 int ab_dtype, int b_layout, float beta, const float *bias,
                 int ca_c, int k_block_factor, sfc_dtype_t c_dtype,
                 sfc_order_t order, sfc_assign_t assign, sfc_tile_t tile,
                 void *workspace, size_t workspace_bytes, void *stream);

/*
 * sfc_gemm_workspace_size2 -- bytes of fp32 workspace sfc_gemm_ex3 needs:
 * ca_c copies of C (M * round_up(N, 4) * 4 bytes each) when ca_c > 1; one copy
 * when ca_c == 1, k_block_factor > 1 and c_dtype is SFC_BF16; else 0.  For
 * ca_c == 0 the size for the most layers the planner may choose, at most
 * ceil(K/64) / k_block_factor.  0 for invalid arguments.  Needs no GPU.
 */
size_t sfc_gemm_workspace_size2(int64_t M, int64_t N, int64_t K, int ca_c, int k_block_factor,
                                sfc_dtype_t c_dtype);

/*
 * sfc_gemm_tune -- measures the configurations of one shape and remembers the
 * fastest (the paper's first way to configure a shape: benchmark the small
 * space of knobs exhaustively, Sec. III-C).  For each layer count in 1, 2, 4,
 * ... up to max_layers (and the time model's own choice) every tile shape is
 * timed (one warm-up call, then the mean of five, CUDA events on `stream`);
 * then K blocks 2, 4, ... up to max_kbf are timed on the chosen (tile,
 * layers).  A measured alternative replaces the time model's tile, layer
 * count or single K block only when it is at least 3 % faster, so that
 * candidates within timing noise keep the model's pick.  The results go into a per-device table for this (M, N, K,
 * ab_dtype, b_layout, c_dtype): afterwards calls with tile = SFC_TILE_AUTO and
 * k_block_factor = 1 use the fastest tile measured for their layer count, and
 * with ca_c = 0 also the fastest layer count (sfc_gemm_plan reports the
 * same).  The tile never changes the result's bits; the layer count does, so
 * callers that need the same bits on every machine pass ca_c explicitly.
 *   A, B, C, strides, ab_dtype, b_layout, c_dtype: as sfc_gemm_ex2; C is
 *     overwritten, and holds the chosen configuration's result on return.
 *   max_layers: 1..64 (1 tunes the tile only); max_kbf: 1..64.
 *   out_tile, out_ca_c, out_kbf: the fastest configuration (tile as sfc_tile_t).
 * Synchronizes `stream` (it times on the host), so it cannot be captured:
 * SFC_ERR_UNSUPPORTED while `stream` is capturing.  Errors: as sfc_gemm_ex2,
 * SFC_ERR_INVALID_ARG for a null output pointer or bounds out of range.
 * Thread safety: the table is guarded; tuning the same shape from two
 * threads at once times each candidate with the other's launches beside it.
 */
int sfc_gemm_tune(int64_t M, int64_t N, int64_t K,
                  const void *A, const void *B, void *C,
                  int64_t lda, int64_t ldb, int64_t ldc,
                  int ab_dtype, int b_layout, sfc_dtype_t c_dtype,
                  int max_layers, int max_kbf, void *stream,
                  int *out_tile, int *out_ca_c, int *out_kbf);

/* sfc_gemm_tune_forget -- empties the current device's table of tuned
 * shapes (calls go back to the time model).  SFC_OK or a CUDA error. */
int sfc_gemm_tune_forget(void);

/* sfc_gemm_tune_lookup -- how AUTO calls consult the table (process-wide):
 * 1 (default) only a shape tuned exactly; 2 otherwise the nearest tuned shape
 * with the same input type, B layout and output type, by distance in
 * (log M, log N, log K), that was measured at the call's layer count (for
 * ca_c = 0: whose layer count fits the call's K) -- the paper's
 * nearest-neighbour prediction of a shape's knobs (Sec. III-C).  With 2 the
 * layer count of a ca_c = 0 call can come from another shape.
 * SFC_ERR_INVALID_ARG for another mode. */
int sfc_gemm_tune_lookup(int mode);

/*
 * sfc_gemm_plan -- the tile and K-layer count sfc_gemm_ex2 would use for these
 * arguments on the current device (ca_c = 0: the library's choice; ca_c >= 1:
 * that count with the tile AUTO or `tile` picks).  No kernel runs.
 *   ab_dtype, b_layout: as sfc_gemm_ex2 (SFC_AB_BF16, SFC_B_KN for sfc_gemm_ex).
 *   out_tile: an sfc_tile_t other than SFC_TILE_AUTO.  out_ca_c: >= 1.
 * Errors: SFC_ERR_INVALID_ARG (as sfc_gemm_ex2, or a NULL output pointer),
 * SFC_ERR_CUDA, SFC_ERR_UNSUPPORTED.
 */
int sfc_gemm_plan(int64_t M, int64_t N, int64_t K, int ca_c, int c_dtype, int tile,
                  int ab_dtype, int b_layout, int *out_tile, int *out_ca_c);

/* A device as the time model sees it (sfc_gemm_plan_desc). */
typedef struct {
    int num_sms;       /* SMs: workers of the one-SM tiles (GB300: 152) */
    int pair_workers;  /* 2-SM pairs that can be resident at once (GB300: 76) */
    double hbm_gbs;    /* attainable DRAM bandwidth, GB/s (GB300: about 6700 for a copy) */
    double sm_ghz;     /* SM clock the tensor cores' rate is taken at */
} sfc_device_desc_t;

/*
 * sfc_gemm_plan_desc -- the library's time model alone, on a described device
 * (no GPU needed; tuned shapes are not consulted).  For C = A B of these sizes
 * and types it returns the tile and K-layer count the model picks (ca_c = 0:
 * any count up to the limit sfc_gemm_workspace_size assumes; ca_c >= 1: that
 * count) and the time it predicts, in ns.  The model follows Sec. III-B's
 * roofline per BRGEMM, T = max(G gamma, beta (S_A + S_B)) (Eqs. 1-4), at two
 * levels: per worker, a 64-deep slab of a tile costs the longer of its MMA time
 * and its operand intake (folded into each tile's measured efficiency), over
 * waves = ceil(tiles * layers / workers) waves of the longest layer's slabs;
 * per launch, at least the DRAM bytes (A and B once, C or the layers' fp32
 * partials) at hbm_gbs; for more than one layer the reduction adds its launch
 * and the partials read back.
 * Errors: SFC_ERR_INVALID_ARG (as sfc_gemm_plan, a NULL pointer, or a device
 * with num_sms < 1, pair_workers < 0 or > num_sms / 2, hbm_gbs or sm_ghz <= 0).
 */
int sfc_gemm_plan_desc(const sfc_device_desc_t *desc, int64_t M, int64_t N, int64_t K, int ca_c,
                       int c_dtype, int ab_dtype, int b_layout, int *out_tile, int *out_ca_c,
                       double *out_ns);

/*
 * sfc_release -- returns to the driver the device memory the library holds
 * between calls on the current device: the staging slots of sfc_gemm_host and
 * what its stream-ordered pools keep after K-layer workspaces, repacked
 * operands and ticket counters were freed (synchronizes the device first).
 * SFC_OK, SFC_ERR_CUDA or SFC_ERR_UNSUPPORTED.
 */
int sfc_release(void);

/*
 * sfc_get_device_status -- synchronizes `stream`, then returns and clears the
 * device error word that kernels set when a bounded wait gives up
 * (SFC_ERR_TIMEOUT), or SFC_ERR_CUDA if the synchronization itself failed.
 * SFC_OK if no kernel reported a problem since the last call.  The word is
 * one per device: a kernel on any stream may have set it, and the first
 * caller to read it after that gets the report.  Only the bits read are
 * cleared (atomically, by a kernel on `stream`), so a report that another
 * stream's kernel makes meanwhile is kept for the next call.
 */
int sfc_get_device_status(void *stream);

/* sfc_last_cuda_error -- the cudaError_t code behind the most recent
 * SFC_ERR_CUDA on the calling thread (0 if none). */
int sfc_last_cuda_error(void);

/* sfc_num_workers -- number of persistent workers (SMs) used on the current
 * device, or a negative sfc_status_t. */
int sfc_num_workers(void);

/*
 * sfc_gemm_noalloc -- sfc_gemm_ex for callers that must not allocate memory.
 *
 * The paper has no counterpart: this is a deployment convenience.  Some
 * callers cannot call cudaMalloc or use a stream-ordered pool at all -- code
 * running inside a framework that owns every device allocation, a real-time
 * path where an allocation may block or fail, or a process that has already
 * handed all device memory to its own arena.  For them this entry point takes
 * the fp32 partial copies of C (ca_c > 1) and the workers' item counter from a
 * fixed scratch area compiled into the library: SFC_NOALLOC_SCRATCH_BYTES
 * bytes for the partials plus 256 bytes for the counter, device memory that
 * every GPU which loads the library holds until the process exits.  It calls
 * no cudaMalloc, cudaFree or allocating library routine, and takes nothing
 * from the library's pools.
 *
 *   Arguments as sfc_gemm_ex with order = SFC, assign and tile = AUTO.
 *   ca_c:   >= 1: that many layers; their partials, ca_c * M * round_up(N, 4)
 *           * 4 bytes when ca_c > 1, must fit in SFC_NOALLOC_SCRATCH_BYTES.
 *           0: the library's layer count, limited to what fits.
 *   Errors: SFC_ERR_WORKSPACE (nothing launched) when ca_c >= 2 and the
 *           partials exceed SFC_NOALLOC_SCRATCH_BYTES;
 *           SFC_ERR_UNALIGNED when A or B would need repacking (a base not
 *           16-byte aligned or lda / ldb not a multiple of 8), since that
 *           takes memory; otherwise as sfc_gemm_ex.
 * The first call on each device looks up the scratch area's device address
 * (with that device current; a lookup that fails is retried by the next
 * call), so make a first call before any stream capture.  All calls share
 * the one scratch area and leave their partials in it: calls whose kernels
 * can overlap on the GPU (different streams without ordering between them)
 * race on it, so order them.
 */
#define SFC_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)
int sfc_gemm_noalloc(int64_t M, int64_t N, int64_t K,
                     const void *A, const void *B, void *C,
                     int64_t lda, int64_t ldb, int64_t ldc,
                     int ca_c, sfc_dtype_t c_dtype, void *stream);

/*
 * sfc_gemm_host -- C = A * B with A, B and C in HOST memory: the library
 * uploads the operands, runs the GEMM and downloads C, with the copies
 * overlapped against the tile contraction.  No counterpart in the paper,
 * whose operands already sit in the memory the cores compute from.
 *
 * A is cut into row panels and B into column panels.  After the first panel
 * of each, the uploads follow a staircase: the next panel is the one that
 * keeps the rows and columns of C covered so far closest to equal, and each
 * upload is followed by the GEMM of the strip of C it completes, so GEMMs
 * start after two panels have arrived and finished strips of C go back while
 * later strips compute.  Panel edges fall on multiples of 512 rows or 256
 * columns (multiples of every output tile), so the result is bit-identical to
 * sfc_gemm_ex2 over the whole problem with the tile and ca_c that
 * sfc_gemm_plan(M, N, K, ca_c, c_dtype, tile, ab_dtype, b_layout, ...)
 * reports, which every strip uses.
 *
 *   A, B, C: HOST pointers, row-major with row strides lda, ldb, ldc in
 *            elements (any stride; the device copies get 16-byte rows).  A and
 *            B are ab_dtype (sfc_ab_t), B laid out per b_layout
 *            (sfc_b_layout_t); C is c_dtype (written, never read).  Use
 *            page-locked memory (cudaHostAlloc / cudaHostRegister): with
 *            pageable memory the result is the same but the copies do not
 *            overlap the GEMM.
 *   ca_c, tile: as sfc_gemm_ex2 (0 / SFC_TILE_AUTO: chosen for the whole
 *            problem).  Order is the curve, assignment automatic, beta = 0,
 *            no bias.
 *   panels:  number of panels of each operand; 0 picks about one per 2048
 *            rows of A and per 2048 columns of B (per 8 KB of a row of an
 *            N-major B, whose column panels are pitched copies), at most 8
 *            each.  Clamped to 64 and to the number of 512-row (256-column)
 *            units.
 *   stream:  the uploads, GEMMs and downloads run on three library streams
 *            (one set per device, shared by all calls); `stream` is made to
 *            wait for the call's last download, so C is complete once
 *            `stream` has reached that point.  The GEMMs touch staging memory
 *            only and are not ordered after earlier work on `stream`, and a
 *            call's GEMMs do not wait for the previous call's downloads:
 *            calls issued back to back overlap in all three streams.
 * The call is asynchronous: it returns once everything is enqueued.  A and B
 * are read after it returns: they must hold their values when the call is
 * made (their uploads are NOT ordered after work already on `stream`) and
 * stay unchanged until `stream` is synchronized; C is complete then.
 * Device memory: staging slots owned by the library, each holding one call's
 * device copies of A, B and C; a slot is reused once the call that used it
 * has completed, so calls issued back to back overlap (the next call's
 * uploads run while this one computes).  New slots are allocated while the
 * slots held stay under half of the device memory that was free at the first
 * call; past that, the call waits for the slots in use and frees them first.
 * sfc_release frees every slot.  Calls from several host threads are
 * serialized per device.
 * Errors (nothing is enqueued): SFC_ERR_INVALID_ARG for sizes, strides
 * (lda < K, ldb < N or K, ldc < N), enums or panels < 0 as sfc_gemm_ex2;
 * SFC_ERR_UNALIGNED when a pointer is not aligned to its element size;
 * SFC_ERR_CUDA when staging memory cannot be allocated; SFC_ERR_UNSUPPORTED.
 * A CUDA error after enqueueing began returns SFC_ERR_CUDA; the call then
 * still orders the staging slot's reuse after whatever it enqueued.
 */
int sfc_gemm_host(int64_t M, int64_t N, int64_t K,
                  const void *A, const void *B, void *C,
                  int64_t lda, int64_t ldb, int64_t ldc,
                  int ab_dtype, int b_layout, int ca_c, sfc_dtype_t c_dtype,
                  sfc_tile_t tile, int panels, void *stream);

/*
 * sfc_mma_peak -- the tensor cores' attainable rate on the current device:
 * every co-schedulable 2-SM pair issues iters x 4 back-to-back 256 x 256 x 16
 * bf16 MMAs (the GEMM's pair instruction) from zero-filled, resident shared
 * memory into tensor memory, one CTA per SM.  The per-SM constant of the
 * roofline the paper's performance model uses (Sec. III-B), measured.
 *   flop_per_clk_per_sm: FLOP per SM clock cycle (clock64 around the issue
 *                        loop up to the commit, slowest pair);
 *   tflops:              the whole device's rate at the clock it ran at (CUDA
 *                        events around the second of two launches).
 * Synchronizes `stream`.  Errors: SFC_ERR_INVALID_ARG (iters outside
 * 1..2^20 or a null output), SFC_ERR_UNSUPPORTED (not sm_103), SFC_ERR_TIMEOUT
 * (the completion wait, bounded at 2 s, gave up), SFC_ERR_CUDA.
 */
int sfc_mma_peak(int iters, double *flop_per_clk_per_sm, double *tflops, void *stream);

/*
 * sfc_debug_pool_used_high -- the high-water mark, in bytes, of the memory in
 * use from the library's stream-ordered pools on the current device (layer
 * workspaces, repacked operands, ticket counters) since the last reset; with
 * reset = 1 the mark is read and then reset, so the next reading covers only
 * what is used after this call.  A
 * diagnostic with no counterpart in the paper (the tests use it to show that
 * sfc_gemm_noalloc takes nothing from the pools).  Does not synchronize: read
 * it after the calls of interest have completed.
 * Errors: SFC_ERR_INVALID_ARG (NULL output, reset not 0 or 1), SFC_ERR_CUDA,
 * SFC_ERR_UNSUPPORTED.
 */
int sfc_debug_pool_used_high(size_t *used_high_bytes, int reset);

/*
 * sfc_debug_force_timeout -- test hook for the failure path: launches one GEMM
 * worker on a tiny problem whose MMA stage waits on a barrier that nothing
 * arrives at, with a wait limit of `limit_ms` milliseconds (1..1000).  The
 * kernel gives up, records SFC_ERR_TIMEOUT in the device error word, drains
 * its in-flight copies, frees its tensor memory and returns; the context stays
 * usable.  Read the outcome with sfc_get_device_status.
 *   A, B: DEVICE bf16 buffers of at least 128*64 and 64*128 elements;
 *   C:    DEVICE fp32 buffer of at least 128*128 elements.
 */
int sfc_debug_force_timeout(const void *A, const void *B, void *C, int limit_ms, void *stream);


#ifdef __cplusplus
}
#endif

#endif /* SFC_GEMM_H */
