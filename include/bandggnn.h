/*
 * bandggnn.h -- C ABI of the band-GGNN library (libbandggnn.so).
 *
 * GGNN message propagation on low-bandwidth graphs as dense block contractions, after
 * "Fast Training of Sparse Graph Neural Networks on Dense Hardware" (arXiv 1906.11786):
 *   - a host-side compile step: Reverse Cuthill-McKee per graph (Section 3.1), sparse batching of
 *     many graphs into one supergraph (Section 2 "Sparse batching"), and the per-edge-type
 *     block-tridiagonal band tiles of Eq. 3 / Algorithm 1;
 *   - device-side propagation Y = sum_p A_p (E W_p + b_p) over the kept edges (Eq. 1 with P types,
 *     Section 2; per-type bias, Appendix D), its backward, and T GGNN steps with a GRU update
 *     (Eq. 1), forward and backward.
 *
 * Conventions for every entry point:
 *   - Return value: BG_OK (0) or a negative BG_E* code; bg_last_error() then gives a message
 *     (thread-local).  No entry point aborts, and none frees memory the caller owns.
 *   - Node arrays on the device are in packed band order: row q of an [N_pad, H] array is
 *     supergraph position q (bg_pack_states / bg_unpack_states convert from and to the caller's
 *     per-graph order).  Rows >= n_real are padding and hold 0.
 *   - Device pointers are caller-owned, must be 16-byte aligned and must not overlap unless
 *     stated.  Every device operation is asynchronous on the CUDA stream passed as `stream`
 *     (a cudaStream_t; NULL = the legacy default stream).
 *   - Shapes: S (block size) in {32, 64, 128, 256, 512}; H (state size) a multiple of 32 in
 *     [32, 256]; P (edge types) in [1, 64].
 *   - dtype BG_BF16: states E, weights W, W_ih, W_hh are bf16 and accumulation is fp32.
 *     dtype BG_F32: all fp32.  Biases, messages Y and every gradient are fp32 for both dtypes.
 */
#ifndef BANDGGNN_H_
#define BANDGGNN_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------------------------- */
#define BG_OK 0
#define BG_EINVAL (-1)    /* bad argument: ids/types out of range, unsupported S/H/P, misalignment */
#define BG_ECAPACITY (-2) /* workspace / saved buffer too small, or no graph fits the capacity */
#define BG_ENOMEM (-3)    /* host or device allocation failed */
#define BG_ECUDA (-4)     /* a CUDA runtime/driver call failed */
#define BG_ETIMEOUT (-5)  /* a device-side wait hit its iteration cap (kernel gave up and returned) */
#define BG_EDEVICE (-6)   /* a kernel recorded an error in the device status word */
#define BG_ESTATE (-7)    /* plan not uploaded, or used on a different device */

/* ---- plan flags (bg_band_plan) ---------------------------------------------------------- */
#define BG_RCM 1u            /* reorder every graph by Reverse Cuthill-McKee (Section 3.1) */
#define BG_KEEP_IF_BETTER 2u /* keep a graph's input order when RCM does not lower its bandwidth */
#define BG_SUPERNODES 4u     /* supernodes (bg_band_plan_opts): see bg_plan_opts */

/* ---- backward flags --------------------------------------------------------------------- */
#define BG_ACCUM 1u /* add into dE/dW/db (and GRU gradients) instead of overwriting them */

typedef enum bg_dtype { BG_F32 = 0, BG_BF16 = 1 } bg_dtype;

/* One input graph: edge e goes src[e] -> dst[e] (graph-local ids in [0, n_nodes)) and has type
 * etype[e] in [0, P).  Host pointers, read during bg_band_plan only. */
typedef struct bg_graph {
  int32_t n_nodes;
  int64_t n_edges;
  const int32_t* src;
  const int32_t* dst;
  const int32_t* etype;
} bg_graph;

typedef struct bg_plan bg_plan; /* opaque, library-owned */

typedef struct bg_info {
  int32_t K;              /* number of S x S block-rows of the supergraph */
  int32_t S;              /* block size */
  int32_t P;              /* edge types */
  int32_t n_graphs;       /* graphs passed in */
  int32_t n_packed;       /* graphs packed (a prefix of the input list) */
  int32_t n_real;         /* supergraph positions holding a node: sum of packed n_nodes */
  int32_t n_pad;          /* K * S */
  int64_t n_edges_in;     /* edges passed in for the packed graphs */
  int64_t n_edges_unique; /* after removing duplicate (src, dst, type) */
  int64_t n_kept;         /* edges inside the block-tridiagonal cover (Eq. 3) */
  int64_t n_dropped;      /* edges whose block distance exceeds one (coverage rule, Section 3.2) */
  int64_t bw_before_max;  /* max over packed graphs of the input-order bandwidth (Section 2) */
  int64_t bw_after_max;   /* max over packed graphs of the bandwidth after reordering (edges
                             without a supernode end) */
  int32_t n_super;        /* supernodes of the packed graphs (BG_SUPERNODES) */
  int64_t n_super_edges;  /* kept edges with a supernode end (included in n_kept) */
} bg_info;

/* ---- compile step (host) ------------------------------------------------------------------
 * bg_band_plan: validate the graphs, reorder each by RCM (flags), pack them contiguously in input
 * order into K = capacity_blocks block-rows of S positions (capacity_blocks = 0 means
 * ceil(sum n_nodes / S)), stopping at the first graph that does not fit (Section 2, "until no more
 * graphs fit"), remove duplicate edges, and build for every block-row k, diagonal d in {-1,0,+1}
 * and type p the S x S 0/1 tile of edges from block k+d to block k (Eq. 3 / Algorithm 1's Cks,
 * Uks, Lks).  Edges between blocks further apart are dropped and counted.  Host only; the plan
 * is library-owned: free it with bg_plan_free.  Errors: BG_EINVAL (bad ids, types, S or P),
 * BG_ECAPACITY (not even the first graph fits), BG_ENOMEM. */
int bg_band_plan(const bg_graph* graphs, int32_t n_graphs, int32_t n_types, int32_t block_S,
                 int32_t capacity_blocks, uint32_t flags, bg_plan** out);
/* bg_band_plan with options.  Supernodes (flag BG_SUPERNODES; the "supernode" propagation
 * primitive of Section 6: some nodes exchange messages with every node, through dense first rows
 * and columns of the adjacency): a node with at least supernode_min_degree distinct neighbours
 * (edges of any type and direction; self-loops not counted) is a supernode, at most
 * max_supernodes per graph, highest degree first (ties: lower id).  A graph's supernodes take its
 * first positions in that order, and RCM orders the graph without them after them, so a hub no
 * longer widens the band.  Every edge with a supernode end is kept whatever the block distance
 * and is propagated by the supernode rows and columns (a per-node gather over those edges, on
 * the device), not by the band tiles; the other edges follow the band cover as before. */
typedef struct bg_plan_opts {
  uint32_t flags;               /* BG_RCM | BG_KEEP_IF_BETTER | BG_SUPERNODES */
  int32_t supernode_min_degree; /* >= 1 when BG_SUPERNODES is set */
  int32_t max_supernodes;       /* per graph, >= 0 */
} bg_plan_opts;
int bg_band_plan_opts(const bg_graph* graphs, int32_t n_graphs, int32_t n_types, int32_t block_S,
                      int32_t capacity_blocks, const bg_plan_opts* opts, bg_plan** out);
void bg_plan_free(bg_plan* plan); /* frees host and device memory of the plan; NULL is a no-op */
int bg_plan_info(const bg_plan* plan, bg_info* out);

/* Reachability preprocessing (Section 4 "Reachability preprocessing"), host only: with T
 * propagation steps, only nodes from which some candidate node is reachable along at most T edges
 * (any types, in edge direction) can change the candidates' final states; the others are dropped.
 * g: the input graph; cand [n_cand]: candidate node ids.  Writes node_map [g->n_nodes] (new id of
 * a kept node -- kept nodes keep their relative order -- or -1), *n_nodes_out (kept nodes),
 * *n_edges_out (kept edges: both ends kept) and, where the arrays are non-NULL (capacity
 * g->n_edges each), the kept edges renumbered, in input order.  Candidates are always kept; T = 0
 * keeps only them.  Errors: BG_EINVAL (ids out of range, NULL arrays, negative T). */
int bg_reach_filter(const bg_graph* g, const int32_t* cand, int32_t n_cand, int32_t T,
                    int32_t* node_map, int32_t* n_nodes_out, int64_t* n_edges_out,
                    int32_t* src_out, int32_t* dst_out, int32_t* etype_out);

/* FLOPs of one forward propagation pass at state size H (the backward pass has the same band
 * and twice the transform FLOPs).  which: */
#define BG_FLOPS_BAND 0  /* band-dense: 2 (3K-2) P S^2 H (all tiles of Eq. 3 as dense products) */
#define BG_FLOPS_XFORM 1 /* edge-type transforms: 2 n_pad P H^2 */
#define BG_FLOPS_GRU 2   /* GRU gate products: 12 n_pad H^2 */
#define BG_FLOPS_NNZ 3   /* useful: 2 H n_kept (one H-vector add per kept edge) */
double bg_plan_flops(const bg_plan* plan, int32_t H, int32_t which);

/* Export host copies of the plan for inspection and for bit-exact comparison.  which: */
#define BG_EXPORT_PERM 0    /* int32 [sum n_nodes of all graphs]: per graph perm[new] = old, concatenated */
#define BG_EXPORT_OFFSETS 1 /* int32 [n_graphs]: first supergraph position, -1 if not packed */
#define BG_EXPORT_MASKS 2   /* uint8 [K][3][P][S][S/8]: bit c%8 of byte (k,d+1,p,r,c/8) = edge
                               from position (k+d)S+c to position kS+r, LSB first */
#define BG_EXPORT_MASKS_T 3 /* uint8 [K][3][P][S][S/8]: bit i%8 of byte (j,e,p,c,i/8) = edge
                               from position jS+c to position (j+e-1)S+i (the transposed band) */
#define BG_EXPORT_BW 4      /* int64 [2][n_graphs]: bandwidth before / after reordering */
#define BG_EXPORT_GATHER 5  /* int32 [n_real]: row of the caller's concatenated state array held
                               by each supergraph position */
#define BG_EXPORT_SUPER_EDGES 6 /* int32 [n_super_edges][3]: (target position, source position,
                               type) of the kept edges with a supernode end, sorted */
#define BG_EXPORT_SUPER_COUNT 7 /* int32 [n_graphs]: supernodes of each graph (its first
                               positions) */
size_t bg_plan_export_bytes(const bg_plan* plan, int32_t which);
int bg_plan_export(const bg_plan* plan, int32_t which, void* out, size_t out_bytes);

/* Block-row partition for running one supergraph on several GPUs (Eq. 3: block-row k couples
 * only to block-rows k - 1 and k + 1).  The supergraph is cut into units of max(128, S) rows (a
 * 128-row tile of 128 / S block-rows when S <= 128, one block-row when S > 128).  Part `part` of
 * n_parts (1 <= n_parts <= the number of units, else BG_EINVAL) owns a contiguous range of whole
 * units (ranges as equal as the unit count allows) and gets a local plan (free it with
 * bg_plan_free; upload it like any plan) over that range plus one unit of halo on each side,
 * clipped at the supergraph's ends.  Local row i is supergraph
 * position row0 + i.  The local forward tiles keep only the rows the part owns as targets, the
 * transposed tiles only the rows it owns as sources.  Used with bg_band_propagate_fwd/bwd:
 *   forward:  fill the local E with rows [row0, row0 + n_local) of the full E -- the halo rows
 *             [0, own_begin) and [own_end, n_local) from the neighbouring parts -- and the own
 *             rows of Y are exact (the halo rows of Y come out 0);
 *   backward: likewise for dY; the own rows of dE are exact (halo rows 0), and dW, db are the
 *             sums over the part's own source rows, so their sum over all parts (an all-reduce)
 *             is the whole plan's.
 * One halo exchange per direction per step: halo_lo rows from part - 1, halo_hi rows from
 * part + 1 (0 at the ends).  The local plan has no graph table (no pack/unpack or readout) and
 * n_real = the real positions of its range.  Plans with supernodes are not partitioned
 * (BG_EINVAL).  Host only. */
typedef struct bg_part_info {
  int32_t row0;      /* supergraph position of local row 0 */
  int32_t n_local;   /* local rows (the local plan's n_pad) */
  int32_t own_begin; /* local rows [own_begin, own_end) are the part's own */
  int32_t own_end;
  int32_t halo_lo;   /* rows before own_begin (from part - 1), = own_begin */
  int32_t halo_hi;   /* rows from own_end on (from part + 1), = n_local - own_end */
} bg_part_info;
int bg_plan_partition(const bg_plan* full, int32_t n_parts, int32_t part, bg_plan** out,
                      bg_part_info* info);

/* Copy the plan's tiles and index tables to the current CUDA device (plan-owned memory, freed by
 * bg_plan_free).  Must precede every device call with this plan; a plan serves one device. */
int bg_plan_upload(bg_plan* plan, void* stream);

/* ---- layout conversion (device) ------------------------------------------------------------
 * E_orig: [sum n_nodes of all graphs, H], the graphs' states concatenated in input order, each
 * graph in its own node order.  E_band: [n_pad, H] in packed band order (Section 3.1: states and
 * labels are permuted with the nodes).  pack writes every row of E_band (padding rows = 0);
 * unpack writes the rows of packed graphs only. */
int bg_pack_states(const bg_plan* plan, bg_dtype dtype, int32_t H, const void* E_orig,
                   void* E_band, void* stream);
int bg_unpack_states(const bg_plan* plan, bg_dtype dtype, int32_t H, const void* E_band,
                     void* E_orig, void* stream);

/* ---- workspace ---------------------------------------------------------------------------
 * Device scratch the caller allocates (e.g. as a torch tensor) and passes as ws / ws_bytes,
 * 256-byte aligned.  op: */
#define BG_OP_PROPAGATE_FWD 0
#define BG_OP_PROPAGATE_BWD 1
#define BG_OP_GGNN_FWD 2
#define BG_OP_GGNN_BWD 3
#define BG_OP_READOUT 4
/* Scratch of the propagate and readout ops (0 for the GGNN ops, whose size depends on T). */
size_t bg_workspace_bytes(const bg_plan* plan, bg_dtype dtype, int32_t H, int32_t op);
/* Scratch of bg_ggnn_step (op BG_OP_GGNN_FWD) or bg_ggnn_step_bwd (BG_OP_GGNN_BWD) for T steps. */
size_t bg_ggnn_workspace_bytes(const bg_plan* plan, bg_dtype dtype, int32_t H, int32_t T,
                               int32_t op);

/* ---- propagation (device) -------------------------------------------------------------------
 * Forward (Eq. 1 / Eq. 3 with P types and per-type bias):
 *   Y[v] = sum over kept edges (u -> v, type p) of (E[u] W_p + b_p)
 * computed per block-row as Algorithm 1 does: the three diagonals' tiles aggregate the
 * neighbouring state blocks per type, then one contraction with the concatenated [P*H, H] edge
 * weights.  E [n_pad, H] (dtype), W [P, H, H] (dtype, W[p][h_in][h_out]), b [P, H] fp32 or NULL,
 * Y [n_pad, H] fp32 (overwritten).  The bf16 tensor-core path adds the bias as in-degree x bias
 * products on the tensor cores; on a plan where some node has more than 256 in-edges of one type
 * these run in fp16, which holds |b| <= 65504: a larger finite bias is reported by
 * bg_check_device as BG_EDEVICE (site 120). */
int bg_band_propagate_fwd(const bg_plan* plan, bg_dtype dtype, int32_t H, const void* E,
                          const void* W, const float* b, float* Y, void* ws, size_t ws_bytes,
                          void* stream);

/* Backward of bg_band_propagate_fwd through the transposed band (A_p^T: the diagonal tiles
 * transposed, super- and sub-diagonal exchanged):
 *   dM_p = A_p^T dY,  dE = sum_p dM_p W_p^T,  dW_p = E^T dM_p,  db_p = column sums of dM_p.
 * dY [n_pad, H] fp32; dE [n_pad, H], dW [P, H, H], db [P, H] (may be NULL) fp32, overwritten
 * unless flags has BG_ACCUM. */
int bg_band_propagate_bwd(const bg_plan* plan, bg_dtype dtype, int32_t H, const void* E,
                          const void* W, const float* dY, float* dE, float* dW, float* db,
                          uint32_t flags, void* ws, size_t ws_bytes, void* stream);

/* Same result as bg_band_propagate_fwd, for callers that cannot allocate device memory while they
 * run (no allocator of their own for the workspace, or cudaMalloc forbidden at that point): the
 * scratch comes from a fixed 32 MiB array inside the library (static device memory, reserved on
 * every GPU where this part of the library's device code is loaded, until the process exits)
 * instead of a caller workspace, and the call itself allocates nothing -- no cudaMalloc, cudaFree
 * or allocating library routine.  The paper has no counterpart; this is a deployment variant.
 * Set-up: bg_plan_upload (which allocates anyway, and must precede this call on the same device)
 * resolves the array's device address (cudaGetSymbolAddress with that device current, which also
 * reserves the array there), creates the library's status word and loads the forward kernels of
 * the plan's block size, so no set-up is left for the first call.
 * Scratch needed: the tensor-core path (bg_band_uses_tensor_cores = 1) needs about
 * n_pad H 2 + P H^2 4 bytes plus the split-tile partials; the SIMT path n_pad P H 4 bytes.  A plan
 * that needs more than 32 MiB is refused with BG_ECAPACITY and a message giving both sizes.
 * All calls share the array, which keeps the previous call's contents (every byte a call reads is
 * written earlier in the same call): calls that overlap on the GPU (different streams, or
 * different host threads without ordering) race and corrupt each other's results; serialise them.
 * Bounded device waits that give up are recorded in the library's status word, as for every other
 * entry point: bg_check_device reports them (BG_ETIMEOUT) and clears the word. */
int bg_band_propagate_fwd_noalloc(const bg_plan* plan, bg_dtype dtype, int32_t H, const void* E,
                                  const void* W, const float* b, float* Y, void* stream);

/* ---- GGNN steps (device) --------------------------------------------------------------------
 * T steps of E(t+1) = GRU(sum_p A_p (E(t) W_p + b_p), E(t)) (Eq. 1; GRU of Cho et al.:
 * r = sigma(W_ir x + b_ir + W_hr h + b_hr), z likewise, n = tanh(W_in x + b_in + r (W_hn h + b_hn)),
 * h' = (1 - z) n + z h, with x the summed messages and h the state; padding rows stay 0). */
typedef struct bg_params {
  const void* W;     /* [P, H, H] dtype */
  const float* b;    /* [P, H] or NULL */
  const void* W_ih;  /* [3H, H] dtype, gate rows r, z, n */
  const void* W_hh;  /* [3H, H] dtype */
  const float* b_ih; /* [3H] */
  const float* b_hh; /* [3H] */
} bg_params;

typedef struct bg_grads {
  float* dW;    /* [P, H, H] */
  float* db;    /* [P, H] or NULL */
  float* dW_ih; /* [3H, H] */
  float* dW_hh; /* [3H, H] */
  float* db_ih; /* [3H] */
  float* db_hh; /* [3H] */
} bg_grads;

/* Bytes of the activation buffer the forward fills and the backward reads: E(0..T) in dtype and
 * the messages Y(0..T-1) in fp32 (the (T+1) N H embeddings of Appendix A.1 plus T message sums);
 * on the tensor-core paths (bf16 with a band kernel for the plan's S and H) the messages are kept
 * in bf16 and transposed bf16 copies of E(0..T-1) and Y(0..T-1) are added, the backward's
 * operands.  The layout is the library's own: callers pass the buffer through unchanged. */
size_t bg_ggnn_saved_bytes(const bg_plan* plan, bg_dtype dtype, int32_t H, int32_t T);
/* E0 [n_pad, H] dtype; ET [n_pad, H] dtype or NULL; saved: device buffer of
 * bg_ggnn_saved_bytes. */
int bg_ggnn_step(const bg_plan* plan, bg_dtype dtype, int32_t H, int32_t T, const bg_params* prm,
                 const void* E0, void* ET, void* saved, size_t saved_bytes, void* ws,
                 size_t ws_bytes, void* stream);
/* dET [n_pad, H] fp32 -> dE0 [n_pad, H] fp32 and parameter gradients (overwritten unless
 * BG_ACCUM).  `saved` must come from bg_ggnn_step with the same plan, prm, H and T. */
int bg_ggnn_step_bwd(const bg_plan* plan, bg_dtype dtype, int32_t H, int32_t T,
                     const bg_params* prm, const void* saved, size_t saved_bytes,
                     const float* dET, float* dE0, const bg_grads* grads, uint32_t flags,
                     void* ws, size_t ws_bytes, void* stream);

/* ---- training-step extras (device) -------------------------------------------------------
 * Per-graph mean-pool readout with a linear output and squared loss:
 *   pool_g = mean over graph g's positions of ET,  pred_g = w_out . pool_g,
 *   loss = 1/2 sum_g (pred_g - target_g)^2.
 * ET [n_pad, H] dtype; w_out [H] fp32; target [n_packed] fp32; loss [1] fp32; dET [n_pad, H]
 * fp32 (overwritten; padding rows 0); dw_out [H] fp32 (overwritten). */
int bg_readout_loss(const bg_plan* plan, bg_dtype dtype, int32_t H, const void* ET,
                    const float* w_out, const float* target, float* loss, float* dET,
                    float* dw_out, void* ws, size_t ws_bytes, void* stream);

/* One bias-corrected Adam step (Kingma & Ba) on n fp32 master parameters with fp32 moments m, v;
 * `working` (n elements of working_dtype, or NULL) receives the updated parameters rounded to
 * the working dtype.  step >= 1. */
int bg_adam_step(int64_t n, float* master, void* working, bg_dtype working_dtype, float* m,
                 float* v, const float* grad, float lr, float beta1, float beta2, float eps,
                 int32_t step, void* stream);

/* ---- diagnostics --------------------------------------------------------------------------- */
const char* bg_last_error(void);
/* Synchronise `stream` and read the device status word that bounded waits and in-kernel checks
 * write: BG_OK, BG_ETIMEOUT or BG_EDEVICE (the word is then cleared). */
int bg_check_device(void* stream);
/* Failure-path self test: launches (asynchronously, on `stream`) one block whose bounded
 * mbarrier wait is never satisfied, so that it gives up after its poll cap (a fraction of a
 * second), records BG_ETIMEOUT (site 901) in the status word and returns, as a stalled pipeline
 * role would.  The next bg_check_device reports BG_ETIMEOUT and clears the word; the context stays
 * usable.  Nothing faults or hangs. */
int bg_selftest_device_wait(void* stream);
/* Kernel timing with CUDA events recorded on the launching stream around every launch of the
 * listed kernels while enabled (adds two event records per launch). */
#define BG_KID_BAND_FWD 0
#define BG_KID_BAND_BWD 1
#define BG_KID_GRU_FWD 2
#define BG_KID_GRU_BWD 3
#define BG_KID_DW 4
#define BG_KID_COUNT 5
int bg_profile_enable(int32_t on);
/* Total milliseconds and launches recorded for kernel `kid` since the last reset (synchronises
 * on the recorded events); reset != 0 clears the record afterwards. */
int bg_profile_read(int32_t kid, double* ms_total, int64_t* launches, int32_t reset);
/* Number of kernels this library has launched since load (all kinds). */
int64_t bg_launch_count(void);
/* 1 when band propagation for (plan, dtype, H) runs on the fused tcgen05 tensor-core kernels,
 * 0 when it runs on the SIMT kernels (fp32 path and shapes the tensor-core kernels do not cover:
 * H not in {32, 64, 128, 256}, H = 256 at S >= 256, P > 32, a padded size that is not a whole
 * number of 128-row tiles); negative status on error.  The plan must be uploaded. */
int bg_band_uses_tensor_cores(const bg_plan* plan, bg_dtype dtype, int32_t H);

#ifdef __cplusplus
}
#endif
#endif /* BANDGGNN_H_ */
