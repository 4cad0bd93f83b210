/* dirigo.h -- C ABI of the GB300 per-output-location equivalence checker.
 *
 * The problem (Sec. 3.4, "Flipping the quantifiers"): two programs A
 * (reference) and B (candidate) read the same input tensors x and write one
 * output y.  For a concrete output location l in dom(y), decide whether
 * forall x. A(x)[l] = B(x)[l].  Each program is an op graph whose ops have
 * per-element equations T_k[l] = f_k(l) (Sec. 3.4, "Per-element equations");
 * res() back-projects y[l] to an expression over the inputs only
 * (Sec. 3.4, "Back-projection").  For a batch of queried locations this
 * library computes, on one GPU:
 *
 *   dirigo_cone     the cone of influence of each location: the sorted unique
 *                   global input ids occurring in res(y[l]), as maximal runs;
 *   dirigo_terms    a key of the canonical form of res(y[l]) (normal form in
 *                   Q[atoms]; floats as reals, transcendentals as
 *                   uninterpreted functions, max as an unordered set, Sec. 3.3
 *                   "Setup"), evaluated in F_p0 x F_p1;
 *   dirigo_compare  per location: equal keys discharge the location; the
 *                   first `budget` others are exported as term lists for an
 *                   SMT solver (Sec. 3.4, "Solving");
 *   dirigo_eval     concrete fp32 evaluation of res(y[l]) (the semantics
 *                   [[R_y(i)]]_x of Sec. 3.3 "Setup").
 *
 * Conventions (all calls):
 *   - Device pointers are caller-owned and never freed by the library.  The
 *     library allocates no device memory: every call that needs scratch takes
 *     a caller workspace whose size dirigo_workspace_size() reports.
 *   - Calls are enqueued on `stream` (a cudaStream_t passed as void*; NULL is
 *     the legacy default stream).  dirigo_cone and dirigo_compare synchronise
 *     the stream once (to read their totals and status); the others do not.
 *     dirigo_cone_async is dirigo_cone without that wait: its errors are
 *     latched in a device word that dirigo_compare reads back with its
 *     statistics, so that a batch waits for the GPU once; with
 *     dirigo_compare_async, which leaves its statistics on the device, a batch
 *     makes no host wait at all (and can be recorded as one CUDA graph).
 *   - Errors: every call returns a dirigo_status; dirigo_last_error() returns
 *     a thread-local message for the last failing call of the thread.  Invalid
 *     arguments are rejected before anything is enqueued.
 *   - Global input ids: inputs are concatenated in declared order; id G (the
 *     total number of input elements) stands for the undefined value read by an
 *     out-of-range access (the paper's bottom, Sec. 3.3).  G + 1 < 2^32.
 *   - Locations are flat row-major indices into the output, 0 <= l < numel(y);
 *     duplicates are allowed (results are per query slot).  Out-of-range
 *     locations are rejected by a device check in dirigo_cone/dirigo_compare
 *     (DIRIGO_E_INVALID) and must not be passed to dirigo_terms/dirigo_eval.
 *   - Ranks are at most 4 for every tensor; reductions have at most 4 dims.
 */
#ifndef DIRIGO_H
#define DIRIGO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DIRIGO_OK = 0,
  DIRIGO_E_INVALID = 1,      /* bad argument, NULL pointer, out-of-range location */
  DIRIGO_E_SHAPE = 2,        /* shapes or broadcasting do not match the op */
  DIRIGO_E_UNSUPPORTED = 3,  /* a form outside the supported op/index-map subset */
  DIRIGO_E_CAPACITY = 4,     /* an output buffer is too small; the size is reported */
  DIRIGO_E_WORKSPACE = 5,    /* workspace smaller than dirigo_workspace_size() */
  DIRIGO_E_CUDA = 6,         /* a CUDA runtime call failed */
  DIRIGO_E_NOMEM = 7,        /* host allocation failed */
  DIRIGO_E_MISMATCH = 8      /* reference and candidate inputs or output differ */
} dirigo_status;

#define DIRIGO_MAX_RANK 4
#define DIRIGO_MAX_RED 4
#define DIRIGO_MAX_GUARDS 4

typedef enum {
  DIRIGO_OP_MATMUL = 1,   /* [M,K] x [K,N] */
  DIRIGO_OP_BMM,          /* [B,M,K] x [B,K,N] */
  DIRIGO_OP_LINEAR,       /* x[B,in], W[out,in], optional b[out] */
  DIRIGO_OP_CONV2D,       /* X[N,Ci,H,W], W[Co,Ci,kh,kw], optional b[Co]; stride, pad */
  DIRIGO_OP_MAXPOOL2D,    /* k x k window, stride */
  DIRIGO_OP_ADD, DIRIGO_OP_SUB, DIRIGO_OP_MUL, DIRIGO_OP_DIV,   /* broadcasting */
  DIRIGO_OP_SCALE,        /* c * x */
  DIRIGO_OP_ADD_SCALAR,   /* x + c */
  DIRIGO_OP_CLAMP_MIN,    /* max(x, c) */
  DIRIGO_OP_RELU,
  DIRIGO_OP_GELU,         /* exact (erf) form */
  DIRIGO_OP_GELU_TANH,
  DIRIGO_OP_TANH, DIRIGO_OP_EXP, DIRIGO_OP_RSQRT, DIRIGO_OP_RECIP,
  DIRIGO_OP_SIGMOID,      /* lowered to recip(1 + exp(-x)) (a sound identity, Sec. 4.2) */
  DIRIGO_OP_ERF, DIRIGO_OP_SQRT, DIRIGO_OP_LOG,
  DIRIGO_OP_SUM, DIRIGO_OP_MEAN, DIRIGO_OP_MAX,   /* over `dim`, `keepdim` */
  DIRIGO_OP_SOFTMAX,      /* over `dim` */
  DIRIGO_OP_LAYERNORM,    /* z, optional gamma, beta over the last dim; eps in `c` */
  DIRIGO_OP_CONTRACT,     /* explicit per-element equation: sum of products */
  DIRIGO_OP_MAXSET,       /* explicit per-element equation: max over terms */
  DIRIGO_OP_KERNEL_CONTRACT, /* a kernel's write set (dirigo_kernel_write), sums */
  DIRIGO_OP_KERNEL_MAXSET    /* a kernel's write set, maxima */
} dirigo_op_kind;

/* An exact constant: num/den when den != 0, else the exact binary value of
 * `value`. */
typedef struct {
  double value;
  int64_t num;
  int64_t den;
} dirigo_const;

/* A guard of a piece: the term is present only when
 *   lo <= oa * o[od] + r[rd] + c < hi     (od or rd = -1: that part absent). */
typedef struct {
  int32_t od, rd;
  int64_t oa, c, lo, hi;
} dirigo_guard;

/* Operand access of a piece: flat offset base + sum_d os[d]*o[d] + sum_e rs[e]*r[e]. */
typedef struct {
  int64_t base;
  int64_t os[DIRIGO_MAX_RANK];
  int64_t rs[DIRIGO_MAX_RED];
} dirigo_access;

/* One piece of an explicit per-element equation (Sec. 3.4 "Per-element
 * equations": the form a kernel's write set takes once inverted): for output
 * coordinates o in [lo, hi) and reduction coordinates r in the box
 * [red_lo, red_hi), each guard-satisfying r contributes a term
 * coef * prod_i operand_i[access_i(o, r)] (CONTRACT) or a member of the max
 * (MAXSET).  Terms are ordered pieces-first, then r row-major. */
typedef struct {
  int64_t lo[DIRIGO_MAX_RANK], hi[DIRIGO_MAX_RANK];
  int32_t n_red, n_guards;
  int64_t red_lo[DIRIGO_MAX_RED], red_hi[DIRIGO_MAX_RED];
  dirigo_const coef;                    /* CONTRACT only */
  dirigo_guard guards[DIRIGO_MAX_GUARDS];
  dirigo_access access[2];              /* one per operand */
} dirigo_piece;

/* Thread coordinates of a kernel launch, in this order:
 * (blockIdx.z, blockIdx.y, blockIdx.x, threadIdx.z, threadIdx.y, threadIdx.x). */
#define DIRIGO_THREAD_DIMS 6

/* A guard of a kernel write: the term is present only when
 *   lo <= sum_j tc[j] * theta[j] + r[rd] + c < hi     (rd = -1: no r part). */
typedef struct {
  int64_t tc[DIRIGO_THREAD_DIMS];
  int32_t rd;
  int64_t c, lo, hi;
} dirigo_kguard;

/* An operand read of a kernel write: flat offset
 *   base + sum_j tc[j] * theta[j] + sum_e rs[e] * r[e]. */
typedef struct {
  int64_t base;
  int64_t tc[DIRIGO_THREAD_DIMS];
  int64_t rs[DIRIGO_MAX_RED];
} dirigo_kaccess;

/* One symbolic write of a kernel (Sec. 3.4 "Per-element equations": under a
 * path condition a thread writes a value to an address).  The threads theta
 * in the box [when_lo, when_hi) (intersected with the launch) each write, at
 * flat output offset addr_base + sum_j addr[j] * theta[j], the value
 * sum over r in [red_lo, red_hi) with all guards true of
 * coef * prod_i operand_i[reads[i](theta, r)] (KERNEL_CONTRACT), or the max
 * of operand_0 over the same r (KERNEL_MAXSET). */
typedef struct {
  int64_t when_lo[DIRIGO_THREAD_DIMS], when_hi[DIRIGO_THREAD_DIMS];
  int64_t addr_base;
  int64_t addr[DIRIGO_THREAD_DIMS];
  int32_t n_red, n_guards;
  int64_t red_lo[DIRIGO_MAX_RED], red_hi[DIRIGO_MAX_RED];
  dirigo_const coef;                     /* KERNEL_CONTRACT only */
  dirigo_kguard guards[DIRIGO_MAX_GUARDS];
  dirigo_kaccess reads[2];               /* one per operand */
} dirigo_kernel_write;

typedef struct {
  int32_t kind;                          /* dirigo_op_kind */
  int32_t n_args;
  int32_t args[3];                       /* tensor ids (inputs 0..I-1, ops I..) */
  int32_t rank;                          /* CONTRACT/MAXSET: output rank */
  int64_t shape[DIRIGO_MAX_RANK];        /* CONTRACT/MAXSET: output shape */
  int32_t stride, pad, k;                /* CONV2D (stride, pad), MAXPOOL2D (k, stride) */
  int32_t dim, keepdim;                  /* SUM/MEAN/MAX/SOFTMAX */
  int32_t axes_rank[2];                  /* binary ops: -1 = numpy trailing alignment */
  int32_t axes[2][DIRIGO_MAX_RANK];      /*   operand dim -> output dim */
  dirigo_const c;                        /* SCALE/ADD_SCALAR/CLAMP_MIN; LAYERNORM eps */
  int32_t n_pieces;
  const dirigo_piece* pieces;            /* CONTRACT/MAXSET; copied at create */
  /* KERNEL_CONTRACT/KERNEL_MAXSET: launch geometry and write set (rank and
   * shape above give the output tensor).  dirigo_graph_create inverts the
   * writes (Sec. 3.4: the per-element equation at l is the value of the
   * thread whose write address is l) into pieces over output coordinates.
   * It needs each active thread coordinate of a write to be one mixed-radix
   * digit of one output coordinate (the digits of an output coordinate
   * forming 1, n1, n1*n2, ...), the written box inside the output, and every
   * read and guard to combine the digits of an output coordinate in the same
   * proportion (affine in the output coordinates); otherwise
   * DIRIGO_E_UNSUPPORTED.  A location two writes reach is rejected
   * (DIRIGO_E_UNSUPPORTED: the stored value would depend on which write
   * lands last); a location no write reaches holds the undefined value
   * (bottom): its equation is one term whose operands are all read out of
   * range. */
  int64_t grid[3], block[3];             /* (z, y, x) */
  int32_t n_writes;
  const dirigo_kernel_write* writes;     /* copied at create */
} dirigo_op_desc;

typedef struct {
  int32_t rank;
  int64_t shape[DIRIGO_MAX_RANK];
} dirigo_tensor_desc;

typedef struct {
  int32_t n_inputs;
  const dirigo_tensor_desc* inputs;      /* declared order = global id order */
  int32_t n_ops;
  const dirigo_op_desc* ops;             /* SSA order */
  int32_t output;                        /* tensor id of y */
} dirigo_graph_desc;

#define DIRIGO_AXIOM_GELU 1u   /* gelu_tanh == gelu_erf (approximation equivalence, Sec. 4.2) */

typedef struct {
  uint32_t flags;
} dirigo_options;

typedef struct dirigo_graph* dirigo_graph_t;

typedef struct {
  int64_t n_leaves;          /* G */
  int64_t out_numel;
  int32_t out_rank;
  int64_t out_shape[DIRIGO_MAX_RANK];
  int32_t n_tensors;         /* inputs + primitive tensors after lowering */
  int32_t n_inputs;
  /* cone cells: boxes of output coordinates on which a location's cone has
   * one run structure with starts affine in the coordinates, found when the
   * graph is compiled; dirigo_cone counts and writes the runs of a location
   * in a fast cell from the cell's plan, and plans the others one by one.
   * n_cells is 0 when the output space would need too many cells. */
  int64_t n_cells;
  int64_t n_fast_cells;
  /* work of the tensor-core key contractions per key lane and call of
   * dirigo_terms: multiply-adds x 2 of the limb products over each piece's
   * output box and reduction box (16 limb products per term), and bytes of
   * the limb matrices written */
  double key_tc_flops;
  double key_limb_bytes;
  int64_t n_tc_contractions; /* contractions on the tensor-core key path */
  /* the most runs any location's cone has when every cone cell has a fast
   * plan (n * this bounds a batch's runs, for sizing dirigo_cone_async's run
   * buffer without a counting call); 0 when unknown */
  int64_t max_runs_per_location;
  /* SplitMix64 finalisers the key definition needs per dirigo_terms call
   * (max-sets of m >= 2 members: m + 2 each, with m the piece's term bound;
   * uninterpreted functions: 3 each) */
  double key_mix_ops;
} dirigo_graph_info;

/* Validates the description, lowers every op to per-element equations
 * (Sec. 3.3 "Torch Operations": each op has a predefined equation) and keeps
 * the compiled program on the host.  Host only; copies `desc`.  On failure
 * *out is NULL and the status says why.  A softmax written out with its max
 * shift -- m = max(x, d, keepdim), z = x - m, e = exp(z),
 * s = sum(e, d, keepdim), y = e / s (or e * recip(s)) -- is lowered as
 * softmax(x) over d (a sound identity, Sec. 4.2), so its canonical term equals
 * the unshifted softmax's. */
dirigo_status dirigo_graph_create(const dirigo_graph_desc* desc, const dirigo_options* opt,
                                  dirigo_graph_t* out);
/* Frees the graph and the host memory it holds (its pinned copy of the cone
 * cell table included).  No call that uses g may still be in flight on a
 * stream: the cone call's upload of the cell table reads host memory that
 * this frees. */
void dirigo_graph_destroy(dirigo_graph_t g);
dirigo_status dirigo_graph_info_get(dirigo_graph_t g, dirigo_graph_info* info);

typedef struct {
  int32_t n_shared_ops;   /* ops of the common prefix cut from both programs */
  int32_t n_inputs;       /* inputs of the trimmed programs (entries of cut_ids) */
} dirigo_merge_info;

/* MERGE with prefix trimming (Sec. 3.2 "MERGE": a common prefix of the two
 * traces is trimmed).  Both descriptions must declare the same inputs
 * (DIRIGO_E_MISMATCH otherwise).  The longest common prefix of ops (same
 * kind, arguments and attributes, op by op; each program keeps the op that
 * computes its output) is cut off, and both programs are compiled as if the
 * tensors the rest of either program reads from before the cut were their
 * inputs.  Host only.
 *   ref_out, cand_out  out: the two trimmed graphs (destroy each with
 *                      dirigo_graph_destroy); with no common prefix they are
 *                      the programs as given
 *   cut_ids  int32[cut_capacity] host, out: for each input of the trimmed
 *            programs, in declared order, the tensor id it stands for in the
 *            original descriptions (an input id, or num_inputs + op index of
 *            a prefix op); ascending.  Global leaf ids, cones and the values
 *            dirigo_eval takes refer to these tensors.
 *   info     out: prefix length and number of trimmed inputs (always set)
 * Returns DIRIGO_E_CAPACITY (info set, no graphs) when cut_ids is too short.
 * Trimming never makes a location discharge wrongly: equal canonical terms
 * over the cut tensors stay equal when the prefix is substituted for them.
 * It can keep a location undischarged that the untrimmed pair discharges when
 * the prefix is not surjective. */
dirigo_status dirigo_graph_create_merged(const dirigo_graph_desc* ref,
                                         const dirigo_graph_desc* cand,
                                         const dirigo_options* opt, dirigo_graph_t* ref_out,
                                         dirigo_graph_t* cand_out, int32_t* cut_ids,
                                         int32_t cut_capacity, dirigo_merge_info* info);

typedef enum { DIRIGO_CALL_CONE = 1, DIRIGO_CALL_TERMS = 2, DIRIGO_CALL_EVAL = 3 } dirigo_call;

/* Bytes of workspace the call needs for a batch of n locations. */
dirigo_status dirigo_workspace_size(dirigo_graph_t g, int32_t call, int64_t n, size_t* bytes);
dirigo_status dirigo_compare_workspace_size(dirigo_graph_t ref, dirigo_graph_t cand, int64_t n,
                                            size_t* bytes);

/* Cone of influence of each queried location (Sec. 3.4: the leaves reached by
 * res(y[l]); syntactic, before simplification; bottom included).
 *   d_locs      int64[n] device, flat output locations
 *   d_offsets   int64[n+1] device, out: CSR offsets in runs
 *   d_runs      uint32[2*run_capacity] device, out: maximal runs (start, len)
 *               sorted, pairwise non-adjacent, over global ids
 *   d_fp        uint64[n] device or NULL, out: fingerprint of each run list:
 *               the sum mod 2^64 over its runs k = 0, 1, ... (in list order) of
 *               (A * start_k + B * len_k + C) * R^k, with
 *               A = 0x9E3779B97F4A7C15, B = 0xBF58476D1CE4E5B9,
 *               C = 0x94D049BB133111EB, R = 0x2545F4914F6CDD1D (it is affine in
 *               the starts, so a cone cell gives it without visiting the runs)
 *   h_total     host, out: total number of runs (always written)
 * Enqueues count, prefix sum and write, then synchronises `stream` once, at
 * the end, to read the total and the status (errors of every pass).  If the
 * runs do not fit, the write pass stores nothing and the call returns
 * DIRIGO_E_CAPACITY with *h_total set and d_runs and d_fp untouched. */
dirigo_status dirigo_cone(dirigo_graph_t g, const int64_t* d_locs, int64_t n, int64_t* d_offsets,
                          uint32_t* d_runs, int64_t run_capacity, uint64_t* d_fp,
                          int64_t* h_total, void* d_ws, size_t ws_bytes, void* stream);

/* Error bits a cone call latches on the device (dirigo_cone_async's d_status,
 * dirigo_compare_stats.cone_error). */
enum {
  DIRIGO_CONE_ERR_UNSUPPORTED = 1,  /* an index map outside the supported cone forms */
  DIRIGO_CONE_ERR_BOXES = 2,        /* a cone needs more boxes or run streams than supported */
  DIRIGO_CONE_ERR_LOCATION = 4,     /* a location outside the output */
  DIRIGO_CONE_ERR_NONMONOTONE = 8,  /* an index map outside the supported cone forms */
  DIRIGO_CONE_ERR_WAIT = 16,        /* a bounded wait of the prefix sum expired */
  DIRIGO_CONE_ERR_RUNS = 32         /* the runs exceed run_capacity (nothing written) */
};

/* dirigo_cone without the wait: count, prefix sum and write are enqueued on
 * `stream` and the call returns at once (Sec. 3.4 "Back-projection", as
 * dirigo_cone).  Arguments as dirigo_cone, except:
 *   d_status  int32 device, in/out: the call ORs its error bits into it
 *             (nonzero = the batch failed; clear it before the batch; the two
 *             programs' cone calls of one batch may share it).  Pass it to
 *             dirigo_compare, which reads it back with its statistics and
 *             returns the cone error (DIRIGO_E_INVALID for a location out of
 *             range, DIRIGO_E_CAPACITY when the runs do not fit run_capacity,
 *             DIRIGO_E_UNSUPPORTED, DIRIGO_E_CUDA for an expired bounded wait).
 * No h_total: d_offsets[n] receives the total number of runs on the device.
 * When any error bit is set before the write pass, or the total exceeds
 * run_capacity, nothing is written to d_runs or d_fp; the offsets are still
 * written.  dirigo_graph_info.max_runs_per_location sizes run_capacity
 * without a counting call.  The workspace is dirigo_cone's. */
dirigo_status dirigo_cone_async(dirigo_graph_t g, const int64_t* d_locs, int64_t n,
                                int64_t* d_offsets, uint32_t* d_runs, int64_t run_capacity,
                                uint64_t* d_fp, int32_t* d_status, void* d_ws, size_t ws_bytes,
                                void* stream);

/* dirigo_cone without a workspace, for callers that cannot allocate device
 * memory (a process whose device memory belongs to a memory manager that must
 * not be bypassed, or code that may not allocate after start-up).  The paper
 * has no counterpart: this is an interface convenience.  Arguments and results
 * are those of dirigo_cone; the scratch it needs (a status word and the
 * prefix-sum buffer, 17 KB) is a fixed array inside the library that every GPU
 * using the library holds until exit.  At most 8,388,608 locations per call
 * (larger batches: DIRIGO_E_WORKSPACE).  The first call on a device looks up
 * the array's device address with that device current; make it before any
 * stream capture.  Like dirigo_cone, every call waits for its stream once, at
 * the end, to read the run total and the status (errors of the write pass
 * included).  All calls share the array, so calls that overlap on the GPU
 * race; issue them one at a time.  Allocates no device memory. */
dirigo_status dirigo_cone_noalloc(dirigo_graph_t g, const int64_t* d_locs, int64_t n,
                                  int64_t* d_offsets, uint32_t* d_runs, int64_t run_capacity,
                                  uint64_t* d_fp, int64_t* h_total, void* stream);

/* Keys of the canonical terms (Sec. 3.4 "Solving": equal canonical terms
 * discharge a location): d_keys uint32[2n] device, out: (lane0, lane1) per
 * slot.  Two locations whose canonical forms are equal get equal keys; two
 * different forms collide with probability below 2^-50 (Schwartz-Zippel over
 * two primes near 2^29).  Asynchronous. */
dirigo_status dirigo_terms(dirigo_graph_t g, const int64_t* d_locs, int64_t n, uint32_t* d_keys,
                           void* d_ws, size_t ws_bytes, void* stream);

enum { DIRIGO_DISCHARGED = 0, DIRIGO_EXPORTED = 1, DIRIGO_DIFFERS_UNEXPORTED = 2 };
enum { DIRIGO_FLAG_CONE_DIFFERS = 1, DIRIGO_FLAG_BOT_REF = 2, DIRIGO_FLAG_BOT_CAND = 4,
       DIRIGO_FLAG_NO_CONES = 8 };

typedef struct {
  int64_t n_discharged, n_exported, n_unexported;
  int64_t n_cone_differs, n_bot_ref, n_bot_cand;
  int64_t export_bytes;      /* bytes written to d_export (0 if none) */
  int64_t export_required;   /* bytes the selected export needs */
  int64_t cone_error;        /* the error bits the cone calls latched in d_cone_status */
} dirigo_compare_stats;

/* Per-location compare and export (Sec. 3.4 "Solving").
 *   verdict  DISCHARGED iff both key lanes agree; else EXPORTED for the first
 *            `budget` undischarged slots (slot order) when the whole export fits
 *            in export_capacity bytes, DIFFERS_UNEXPORTED otherwise.
 *   flags    CONE_DIFFERS (run lists differ), BOT_REF/BOT_CAND (bottom in the
 *            cone); NO_CONES when the cone arguments are NULL.
 *   d_export the term lists of the exported slots in the documented "DXP1"
 *            byte format (may be NULL with budget 0); 8-byte aligned
 *            (DIRIGO_E_INVALID otherwise).
 * Cone arguments (offsets, runs, fingerprints from dirigo_cone) may be NULL
 * together (with n = 0 the run buffers may be NULL on their own).
 * d_cone_status: the status word of dirigo_cone_async calls that made the
 * cones (NULL for cones from dirigo_cone).  When it is nonzero the cones are
 * not read (flags are NO_CONES), verdicts and the export are still computed,
 * stats.cone_error holds the bits, and the call returns the cone error (see
 * dirigo_cone_async) instead of its own status.
 * cones_ready: a cudaEvent_t (as void*) recorded after the cone calls on
 * another stream, or NULL when the cones are already ordered before the call
 * on `stream`.  The verdicts and the export need only the keys; the flag
 * passes (which read the cones) run on a stream the library keeps per
 * device, after this event, so that with the compare enqueued on the keys'
 * stream the export overlaps the cones' writing.  Everything is joined back
 * into `stream` before the statistics are read.
 * Synchronises `stream` once at the end to fill *h_stats.
 * The export's per-program passes for the candidate run on a stream the
 * library keeps per device, forked from and joined back into `stream` with
 * events: everything the call does stays ordered after earlier work on
 * `stream` and before later work on it.
 * Returns DIRIGO_E_CAPACITY (with stats filled) when the export did not fit. */
dirigo_status dirigo_compare(dirigo_graph_t ref, dirigo_graph_t cand, const int64_t* d_locs,
                             int64_t n, const uint32_t* d_kref, const uint32_t* d_kcand,
                             const int64_t* d_off_ref, const uint32_t* d_runs_ref,
                             const uint64_t* d_fp_ref, const int64_t* d_off_cand,
                             const uint32_t* d_runs_cand, const uint64_t* d_fp_cand,
                             const int32_t* d_cone_status, void* cones_ready,
                             uint8_t* d_verdict, uint8_t* d_flags, int64_t budget,
                             uint8_t* d_export, int64_t export_capacity,
                             dirigo_compare_stats* h_stats, void* d_ws, size_t ws_bytes,
                             void* stream);

/* dirigo_compare without the host wait (Sec. 3.4 "Solving", as
 * dirigo_compare): every size and decision stays on the device, and the last
 * kernel of the call writes the statistics to d_stats (a dirigo_compare_stats
 * in device memory, 8-byte aligned) and the status dirigo_compare would have
 * returned to d_status (int32 device, may be NULL).  Argument errors are
 * still returned at once.  A whole batch -- asynchronous cones, term keys,
 * this compare -- then enqueues without any host wait; the caller reads the
 * statistics when it needs them (for example once per replay of a CUDA graph
 * of the batch).  The internal streams and events it uses are forked from and
 * joined back into `stream`. */
dirigo_status dirigo_compare_async(dirigo_graph_t ref, dirigo_graph_t cand,
                                   const int64_t* d_locs, int64_t n, const uint32_t* d_kref,
                                   const uint32_t* d_kcand, const int64_t* d_off_ref,
                                   const uint32_t* d_runs_ref, const uint64_t* d_fp_ref,
                                   const int64_t* d_off_cand, const uint32_t* d_runs_cand,
                                   const uint64_t* d_fp_cand, const int32_t* d_cone_status,
                                   void* cones_ready, uint8_t* d_verdict, uint8_t* d_flags,
                                   int64_t budget, uint8_t* d_export, int64_t export_capacity,
                                   dirigo_compare_stats* d_stats, int32_t* d_status, void* d_ws,
                                   size_t ws_bytes, void* stream);

/* Concrete fp32 evaluation of res(y[l]) on the inputs (Sec. 3.3 "Setup"):
 * d_inputs is a HOST array of n_inputs device pointers to contiguous fp32
 * tensors in declared order; d_out float[n] device.  A reached bottom
 * evaluates to NaN.  Asynchronous. */
dirigo_status dirigo_eval(dirigo_graph_t g, const float* const* d_inputs, const int64_t* d_locs,
                          int64_t n, float* d_out, void* d_ws, size_t ws_bytes, void* stream);

/* Kernel timing: when enabled, each call records CUDA events around its
 * kernels on its stream; dirigo_profile_read returns per-kernel-class totals
 * (milliseconds) and launch counts accumulated since the last reset. */
typedef enum {
  DIRIGO_K_CONE_COUNT = 0, DIRIGO_K_CONE_WRITE, DIRIGO_K_KEY_LEAF, DIRIGO_K_KEY_GEMM,
  DIRIGO_K_KEY_ELEM, DIRIGO_K_COMPARE, DIRIGO_K_EXPORT, DIRIGO_K_EVAL, DIRIGO_K_SCAN,
  DIRIGO_K_KEY_LIMBS, /* limb matrices of the tensor-core key contraction */
  DIRIGO_K_COUNT_
} dirigo_kernel_class;
dirigo_status dirigo_profile_enable(int32_t on);
dirigo_status dirigo_profile_read(double* ms, int64_t* launches, int32_t n_classes, int32_t reset);

/* Order in which to query the output locations of a reference/candidate pair
 * (Sec. 4, "Search Heuristic": a ranked prefix, then a random permutation of
 * the rest).  Host only; no device call.  The ranked prefix, deduplicated in
 * this order:
 *   1. corners: for every kernel op whose output reaches the graph output
 *      through same-shape elementwise ops (later kernels first, candidate
 *      first), the locations its launch's corner threads write -- the first
 *      and last thread of the first and last block, then threads 31 and 32
 *      of block 0 (blocks and threads numbered x fastest); then every corner
 *      of the output box and flat indices 31 and 32;
 *   2. region coverage: one location (the lowest corner) of every cone cell
 *      of the candidate, then of the reference (cells are output boxes of
 *      one piecewise cone structure; the paper's analogue is one satisfying
 *      location per path condition);
 *   3. tensor boundaries: the first and the last output element.
 * The remaining locations follow in a permutation drawn from `seed`
 * (Fisher-Yates with the SplitMix64 sequence seed, seed + gamma, ...).
 *   h_order   int64[out_numel] host, out: every output location exactly once
 *   h_prefix  out (optional): length of the ranked prefix
 * Returns DIRIGO_E_MISMATCH when the two outputs differ in shape. */
dirigo_status dirigo_query_order(dirigo_graph_t ref, dirigo_graph_t cand, uint64_t seed,
                                 int64_t* h_order, int64_t* h_prefix);

/* Integer-ALU peaks of the key arithmetic on the current device (the paper
 * has no counterpart: these are roofline denominators for the key kernels
 * that run on the CUDA cores).  *mix64_per_s: SplitMix64 output finalisers per
 * second (eight independent chains per thread); *madwide_per_s: 32 x 32 ->
 * 64-bit multiply-adds per second (eight independent accumulators per
 * thread).  Each is the best of three launches of 1,216 blocks x 256 threads
 * timed with CUDA events on `stream`; waits for the stream.  Allocates no
 * device memory. */
dirigo_status dirigo_alu_peak(double* mix64_per_s, double* madwide_per_s, void* stream);

/* Total number of kernel launches the library issued since process start. */
int64_t dirigo_launch_count(void);

const char* dirigo_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* DIRIGO_H */
