/*
 * aspis.h -- C ABI of libaspis, the GB300 (sm_103a) implementation of the
 * parameter-server detection-and-aggregation step of Aspis
 * (Konstantinidis & Ramamoorthy, "Aspis: Robust Detection for Distributed
 * Learning", MLSys 2022).
 *
 * One training round at the PS (Algorithm 1): the K workers return, for each
 * of the f = C(K,r) files, the r copies of that file's gradient (d floats).
 * The PS
 *   1. compares every pair of copies of every file          aspis_check
 *   2. builds the agreement graph G (edge iff two workers
 *      agree on all C(K-2,r-2) files they share)             aspis_check
 *   3. finds the maximum cliques of G (Algorithm 3)           aspis_detect
 *   4. picks one copy per file: an honest one when the
 *      maximum clique is unique (Case 1), else the majority
 *      copy (Case 2, Eq. 2)                                   aspis_select
 *   5. aggregates the picked copies coordinate-wise
 *      (lower median; mean optional)                          aspis_aggregate
 *
 * Conventions shared by every call:
 *   - Pointers marked "device" are CUDA device pointers owned by the caller;
 *     the library never allocates on the per-round path.  The only library
 *     allocations are the tables of an aspis_assignment (host) and its device
 *     mirror, released by aspis_assignment_free.
 *   - Device calls are asynchronous on the given stream (a cudaStream_t
 *     passed as void*; NULL = legacy default stream).  They return after the
 *     launch; argument errors are returned synchronously before anything is
 *     enqueued.  Outcomes decided on the device (clique-search budget, empty
 *     selection) are written into the device-resident aspis_detection and are
 *     visible after the stream is synchronized.
 *   - Gradient copies are one fp32 buffer laid out [f][r][ld]: row (i, s) is
 *     the vector returned by the worker in slot s of file i (slots are in
 *     ascending worker order); only the first d of the ld floats of a row are
 *     read.  ld >= d.  The 128-bit load path is used when the buffer is
 *     16-byte aligned and ld % 4 == 0; otherwise a 4-byte path is used (not
 *     an error).
 *   - Equality of copies is bitwise equality of their fp32 words (+0 != -0;
 *     NaNs equal iff their bit patterns are).
 *   - Workers are 0-based.  Bit k of a worker mask is worker k.  K <= 31.
 *   - Slot pairs (s,t), s<t, of one file are numbered (0,1),(0,2),...,
 *     (0,r-1),(1,2),...,(r-2,r-1); bit p of a per-file mismatch word is set
 *     iff the copies of the p-th pair differ.  r <= 8, so at most 28 bits.
 */
#ifndef ASPIS_H
#define ASPIS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ASPIS_MAX_K 31
#define ASPIS_MAX_R 8
/* Largest number of files aspis_aggregate can reduce per coordinate (the
 * per-coordinate working set is staged in shared memory). */
#define ASPIS_MAX_AGG_FILES 6144

typedef enum {
    ASPIS_OK = 0,
    ASPIS_E_INVAL = 1,           /* bad argument (NULL pointer, r<2, r>K, d<1, ld<d, mode) */
    ASPIS_E_RANGE = 2,           /* K > 31, r > 8, or f > ASPIS_MAX_AGG_FILES for aggregation */
    ASPIS_E_ALIGN = 3,           /* reserved: misalignment is handled, never reported */
    ASPIS_E_CUDA = 4,            /* a CUDA runtime call or launch failed */
    ASPIS_E_LIMIT = 5,           /* clique search ran out of its node budget (device status) */
    ASPIS_E_EMPTY = 6,           /* no file kept a copy, nothing to aggregate (device status) */
    ASPIS_E_NOT_IMPLEMENTED = 7
} aspis_status;

/* Subset-based file assignment (Algorithm 2; Example 1 fixes file 0 to the
 * first r workers).  File i is given to the i-th r-subset of the workers in
 * lexicographic order. */
typedef struct {
    int32_t K;                   /* workers */
    int32_t r;                   /* redundancy: copies per file */
    int64_t f;                   /* files, C(K,r) */
    int64_t l;                   /* files per worker (computation load), C(K-1,r-1) */
    int64_t pair_share;          /* files shared by any two workers, C(K-2,r-2) */
    uint8_t *file_workers;       /* host [f*r]: worker of slot s of file i, ascending in s */
    int32_t *worker_files;       /* host [K*l]: files of worker j, ascending */
    uint8_t *slot_of;            /* host [K*l]: slot of worker j in worker_files[j*l+k] */
    uint8_t *dev_file_workers;   /* device [f*r] mirror of file_workers, or NULL */
} aspis_assignment;

/* Outcome of detection and selection for one round; lives in device memory
 * (the caller allocates sizeof(aspis_detection) = 36 bytes).  Written by
 * aspis_detect (all but n_sel; n_sel and median_exact reset to 0),
 * aspis_select (n_sel) and aspis_aggregate (status = ASPIS_E_EMPTY when
 * n_sel == 0; median_exact added to). */
typedef struct {
    uint32_t clique_mask;        /* the maximum clique with the smallest mask value */
    int32_t  omega;              /* size of a maximum clique */
    uint32_t n_max_cliques;      /* number of maximum cliques */
    int32_t  success;            /* 1 iff n_max_cliques == 1: H = clique (Case 1) */
    int32_t  n_sel;              /* files whose copy enters aggregation */
    int32_t  status;             /* ASPIS_OK, ASPIS_E_LIMIT or ASPIS_E_EMPTY */
    uint32_t search_nodes;       /* Bron-Kerbosch nodes visited (diagnostic) */
    uint32_t node_budget;        /* in: node limit per search branch, 0 = default
                                    (2^20); read by aspis_detect, never written */
    uint32_t median_exact;       /* coordinates that the lower median resolved by
                                    its exact key-space path (a NaN, a crowded or
                                    overflowed bin) since aspis_detect reset it;
                                    added to by aspis_aggregate (diagnostic) */
} aspis_detection;

/* Short text for a status code. */
const char *aspis_status_str(int status);

/* ABI version of this header (incremented on any signature change). */
int aspis_abi_version(void);

/* Algorithm 2.  Fills *out with host tables (allocated by the library).
 * Requires 2 <= r <= K, K <= ASPIS_MAX_K, r <= ASPIS_MAX_R.  Host only: needs
 * no GPU.  On error *out is zeroed. */
aspis_status aspis_assign(int K, int r, aspis_assignment *out);

/* Uploads file_workers to a device mirror (cudaMalloc + copy, synchronous),
 * once; later calls are no-ops.  Needed by every device call below. */
aspis_status aspis_assignment_to_device(aspis_assignment *a);

/* Frees the host tables and the device mirror and zeroes *a. */
void aspis_assignment_free(aspis_assignment *a);

/* Bytes of device workspace the calls below need for assignment a: always 0.
 * Every per-round intermediate is a named caller buffer (file_neq, adj, det,
 * sel, out) and each kernel keeps its working set in shared memory, so no
 * call takes a workspace argument.  Kept so that a caller written against a
 * workspace-passing interface can size it (to nothing).  Host only; a NULL a
 * also gives 0. */
size_t aspis_workspace_bytes(const aspis_assignment *a);

/* Steps 1-2: per-file agreement alpha_i and graph G (Section 4, the
 * definitions of alpha_i^{(j1,j2)} and alpha^{(j1,j2)} and the edge rule of
 * Algorithm 3).
 *   copies    device [f][r][ld] fp32
 *   file_neq  device [f] uint32, out: per-file slot-pair mismatch word
 *   adj       device [K] uint32, out: adj[j] bit k = edge (j,k), i.e. workers
 *             j and k returned bitwise-equal copies for every file they share;
 *             no self loops, bits >= K zero
 * Reads f*r*d*4 bytes.  Overwrites file_neq and adj entirely. */
aspis_status aspis_check(const float *copies, int64_t d, int64_t ld,
                         const aspis_assignment *a, uint32_t *file_neq,
                         uint32_t *adj, void *stream);

/* Step 2 alone: the graph G from per-file mismatch words (the edge rule of
 * Algorithm 3, as in aspis_check).  For a PS whose copies are split by
 * coordinate range over several devices: each device runs aspis_check on
 * its slice, the file_neq words of all slices are OR-combined (a copy pair
 * differs iff it differs in some slice), and every device then derives the
 * same G from the combined words.
 *   file_neq  device [f] uint32 (slot-pair mismatch words, all bits < r(r-1)/2)
 *   adj       device [K] uint32, out, as for aspis_check
 * Reads f*4 bytes.  Overwrites adj entirely. */
aspis_status aspis_graph(const uint32_t *file_neq, const aspis_assignment *a,
                         uint32_t *adj, void *stream);

/* Step 3: all maximum cliques of G (Algorithm 3: every maximum clique is
 * listed; exactly one of them means successful detection).  Bron-Kerbosch with pivoting over
 * 32-bit vertex masks in one thread block; each search branch has a node
 * budget (det->node_budget, 0 = 2^20 nodes) after which det->status =
 * ASPIS_E_LIMIT and det->success = 0 (the round then falls back to majority
 * voting, Case 2).
 *   adj  device [K] uint32 (as written by aspis_check)
 *   det  device aspis_detection, out (n_sel reset to 0) */
aspis_status aspis_detect(const uint32_t *adj, int K, aspis_detection *det,
                          void *stream);

/* Step 4: one copy per file (Algorithm 1).
 *   Case 1 (det->success): the copy of the lowest slot whose worker is in the
 *     clique; -1 (file dropped) if the file has no such worker.
 *   Case 2: the majority copy m_i of Eq. 2, read as the largest class of
 *     bitwise-equal copies (ties to the class holding the lower slot); sel is
 *     that class's lowest slot.  No file is dropped.
 *   file_neq  device [f] (from aspis_check)
 *   det       device, in: success/clique_mask; out: n_sel (added to)
 *   sel       device [f] int8, out: chosen slot or -1 */
aspis_status aspis_select(const uint32_t *file_neq, aspis_detection *det,
                          const aspis_assignment *a, int8_t *sel, void *stream);

/* Step 5: coordinate-wise aggregation of the chosen copies (Algorithm 1:
 * median of the majority gradients in Case 2, mean in Case 1).
 *   mode 0: lower median: for each coordinate c < d the element of rank
 *           floor((n_sel-1)/2) of {copies[i][sel[i]][c] : sel[i] >= 0} in
 *           IEEE-754 totalOrder; out[c] has that element's exact bits.
 *   mode 1: mean of the same values (compensated fp32 summation, one final
 *           rounding; within 1e-6 relative of the exactly-rounded mean).
 *   sel   device [f] (from aspis_select)
 *   det   device; n_sel is read, status set to ASPIS_E_EMPTY when 0 (then
 *         out is left untouched)
 *   out   device [d] fp32
 * Reads n_sel*d*4 bytes and writes d*4.  f must be <= ASPIS_MAX_AGG_FILES. */
aspis_status aspis_aggregate(const float *copies, int64_t d, int64_t ld,
                             const aspis_assignment *a, const int8_t *sel,
                             aspis_detection *det, int mode, float *out,
                             void *stream);

/* Steps 1-5 back to back on one stream (the whole PS step of one round). */
aspis_status aspis_round(const float *copies, int64_t d, int64_t ld,
                         const aspis_assignment *a, uint32_t *file_neq,
                         uint32_t *adj, aspis_detection *det, int8_t *sel,
                         int mode, float *out, void *stream);

/* Largest f accepted by aspis_round_static, and the size in bytes of the
 * fixed device array that holds its per-round intermediates. */
#define ASPIS_STATIC_MAX_FILES 6144
#define ASPIS_STATIC_SCRATCH_BYTES 81920

/* aspis_round for callers that cannot allocate device memory.  The paper has
 * no counterpart: this is a deployment variant of the same round.  Callers
 * such as runtimes that hand the library buffers from their own memory pool,
 * or processes whose allocator is locked or budgeted, may own the copies,
 * the output and the detection record but cannot let a library call
 * cudaMalloc (aspis_assignment_to_device does; aspis_round needs caller
 * buffers for file_neq, adj and sel).  This call allocates nothing: the
 * mismatch words, the graph, the selection and a device copy of the
 * assignment table live in one file-scope device array of
 * ASPIS_STATIC_SCRATCH_BYTES bytes, which every GPU that loads the library
 * holds until the process exits.
 *   copies  device [f][r][ld] fp32, as for aspis_round
 *   a       host tables from aspis_assign; the device mirror is not needed
 *           (file_workers is copied into the array on the stream every call)
 *   det     device aspis_detection, out, as for aspis_round
 *   out     device [d] fp32, out; mode as for aspis_aggregate
 * Results equal aspis_round's.  f > ASPIS_STATIC_MAX_FILES returns
 * ASPIS_E_RANGE before anything is enqueued.  The first call on a device
 * looks up the array's device address (cudaGetSymbolAddress, with that
 * device current); make that first call before any stream capture.  The
 * address is kept for the life of the process: after cudaDeviceReset of a
 * device (which unloads the library's device code there) the kept address
 * is stale, so do not call this function on that device again in the same
 * process.  Every call copies the assignment table (f*r bytes) from the
 * library's pageable host memory into the array on the stream, so the call
 * may return only after the work already queued on the stream has drained.
 * All calls share the array and its contents persist between calls (the
 * parts that must start at zero are cleared by each call): calls that may
 * overlap on the GPU, e.g. on unordered streams, race and must not be
 * issued. */
aspis_status aspis_round_static(const float *copies, int64_t d, int64_t ld,
                                const aspis_assignment *a, aspis_detection *det,
                                int mode, float *out, void *stream);

/* The whole round from host memory: copies the f*r*ld floats at
 * host_copies (pinned memory gives full bandwidth) into the device buffer
 * dev_copies, runs aspis_round, and copies the d aggregated floats into
 * host_out and the detection record into host_det.  All work and copies are
 * ordered on the stream.  Copies of 64 MiB or more from pinned host memory
 * that the device can address (16-byte aligned, ld % 4 == 0) are made by a
 * copy kernel whose SM loads stream over the host link, in eight file-aligned
 * chunks, and each chunk is compared on a library-owned stream (created on
 * first use) as soon as it has landed; other copies of 64 MiB or more are
 * split over four library-owned streams that the stream waits for.  The host
 * buffers must stay valid until the stream is synchronized.  Device
 * buffers are the caller's, as for aspis_round. */
aspis_status aspis_round_host(const float *host_copies, float *dev_copies,
                              int64_t d, int64_t ld, const aspis_assignment *a,
                              uint32_t *file_neq, uint32_t *adj,
                              aspis_detection *det, int8_t *sel, int mode,
                              float *dev_out, float *host_out,
                              aspis_detection *host_det, void *stream);

/* ---------------------------------------------------------------------
 * Detection beyond 32 workers (Algorithm 3 with vertex sets of up to 128
 * workers).  The round's other steps keep K <= 31; this call takes the
 * agreement graph directly, as in the clique-timing experiment of the
 * appendix (Table 5: K = 100, r = 5, whose C(100,5) = 75,287,520 files are
 * never materialised).  No counterpart of a separate call in the paper. */
#define ASPIS_WIDE_MAX_K 128
#define ASPIS_WIDE_ALL_MAXIMAL 1u     /* flags: enumerate every maximal clique */

/* Outcome of aspis_detect_wide; lives in device memory (64 bytes). */
typedef struct {
    uint32_t clique_mask[4];     /* the maximum clique with the smallest mask value;
                                    worker k is bit k % 32 of word k / 32, and word 3
                                    is the most significant in the comparison */
    uint64_t n_max_cliques;      /* number of maximum cliques */
    uint64_t n_maximal;          /* maximal cliques reported: all of them with
                                    ASPIS_WIDE_ALL_MAXIMAL, else those the size
                                    bound did not prune (diagnostic) */
    uint64_t search_nodes;       /* Bron-Kerbosch nodes visited (diagnostic) */
    int32_t  omega;              /* size of a maximum clique */
    int32_t  success;            /* 1 iff n_max_cliques == 1 and the search finished */
    int32_t  status;             /* ASPIS_OK or ASPIS_E_LIMIT */
    uint32_t node_budget;        /* in: node limit per warp, 0 = 2^20; never written */
    uint32_t flags;              /* in: ASPIS_WIDE_ALL_MAXIMAL or 0; never written */
    uint32_t reserved;
} aspis_detection_wide;

/* All maximum cliques of an agreement graph of K <= 128 workers
 * (Algorithm 3), by Bron-Kerbosch with Tomita pivoting over 128-bit vertex
 * sets, on one thread-block cluster (16 blocks of four warps where the device
 * allows that cluster size, else 8): every block tables the root's branches,
 * their children are dealt to the warps one at a time from a cluster-wide
 * counter, each warp walks its items cooperatively, and workers adjacent to
 * all other candidates join the clique without branching.  Without flags,
 * branches that cannot reach the largest clique found so far are pruned (what
 * detection needs); with ASPIS_WIDE_ALL_MAXIMAL every maximal clique is
 * enumerated and counted, as the NetworkX enumeration timed in Table 5 does.
 * Calls are independent: all search state lives in the launch's shared
 * memory, and det is written once at the end.
 *   adj  device [K][4] uint32: row j = the neighbours of worker j, worker k
 *        at bit k % 32 of word k / 32.  An edge counts only when both rows
 *        list it; self loops and bits >= K are ignored.
 *   det  device aspis_detection_wide, in/out (node_budget and flags in)
 * K < 1 or a NULL pointer returns ASPIS_E_INVAL, K > 128 ASPIS_E_RANGE,
 * before anything is enqueued.  A warp that exceeds its node budget stops
 * the search: status = ASPIS_E_LIMIT, success = 0. */
aspis_status aspis_detect_wide(const uint32_t *adj, int K, aspis_detection_wide *det,
                               void *stream);

/* The round for copies that are not bit-identical.  Section 5 (after
 * Algorithm 1) notes that honest copies differing by floating-point effects
 * can be handled: Case 1 averages the honest copies of each file, Case 2
 * clusters the copies and averages the largest cluster.  Readings:
 *   - copies a, b of a file are close iff |a[c] - b[c]| <= tau for every
 *     c < d (difference and magnitude in fp32; never close where either is
 *     NaN); the graph rule uses "close" for "equal";
 *   - Case 1 averages the slots whose worker is in the clique (a file with
 *     none is dropped); Case 2 the largest connected component of "close"
 *     among the r slots, ties to the component holding the lower slot;
 *   - the average of the chosen copies is their arithmetic mean, computed in
 *     fp32 as x0 + (sum of the deviations x_s - x0) / k with x0 the first
 *     copy (a deviation is 0 where x_s equals x0 bitwise): within
 *     1e-6 * max(|mean|, mean |x_s|) of the exact mean for close copies, and
 *     exactly the common value of identical copies.
 * The lower median (mode 0) or mean (mode 1) of the kept files' averages is
 * written to out.  With tau = 0 and copies without NaNs or signed-zero
 * differences the result equals aspis_round's.
 *   tau        >= 0 (NaN or negative: ASPIS_E_INVAL)
 *   file_neq, adj, det   as for aspis_round ("not close" bits)
 *   slot_mask  device [f] uint8, out: the slots averaged for file i (0 = dropped)
 *   sel        device [f] int8, out: 0 for kept files, -1 for dropped ones
 *   means      device [f][ldm] fp32, out: the averages (rows of dropped
 *              files untouched); ldm >= d; 16-byte aligned with ldm % 4 == 0
 *              for the 128-bit path
 * Reads f*r*d*4 bytes (compare) plus the chosen copies (averages), writes
 * n_kept*d*4 and reads them again (median).  f must be <= ASPIS_MAX_AGG_FILES. */
aspis_status aspis_round_tolerant(const float *copies, int64_t d, int64_t ld,
                                  const aspis_assignment *a, float tau, uint32_t *file_neq,
                                  uint32_t *adj, aspis_detection *det, uint8_t *slot_mask,
                                  int8_t *sel, float *means, int64_t ldm, int mode, float *out,
                                  void *stream);

/* The model update that follows the aggregation (Section 2, Eq. 1, with
 * the aggregate of Algorithm 1 in place of the batch gradient), with the
 * heavy-ball momentum of the experiments (Appendix A.3: momentum 0.9).  For
 * every coordinate c < d:
 *     mu != 0:  v[c] <- RN(mu * v[c] + g[c]);  w[c] <- RN(w[c] - eta * v[c])
 *     mu == 0:  w[c] <- RN(w[c] - eta * g[c])   (Eq. 1; v is not touched)
 * where RN rounds the exact value once to fp32 (round to nearest even), so
 * results are bitwise reproducible; NaN and infinity follow IEEE-754.
 *   g    device [d] fp32, in: the aggregated gradient (aspis_aggregate's out)
 *   w    device [d] fp32, in/out: the parameters
 *   v    device [d] fp32, in/out: the momentum buffer (zeros before the first
 *        update); may be NULL when mu == 0
 *   eta  the step eta_t of this iteration (the experiments' schedules are
 *        x * y^floor(t/z), computed by the caller)
 * g, w and v are each either the same array or disjoint; a partial overlap,
 * d < 0 or a missing pointer returns ASPIS_E_INVAL, d == 0 does nothing.
 * 16-byte aligned pointers take the 128-bit path (any d; the last d % 4
 * coordinates one by one), others a 4-byte path.  Reads 12 bytes per
 * coordinate and writes 8 (8 and 4 when mu == 0).  No counterpart of a
 * separate call in the paper, whose PS applies this update right after the
 * aggregation. */
aspis_status aspis_sgd(const float *g, float *w, float *v, int64_t d, float eta,
                       float mu, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* ASPIS_H */
