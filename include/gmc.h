/*
 * gmc.h -- C ABI of libgmc.so, the GB300 (sm_103a) implementation of the
 * layer-boundary compression step of Grounded Message Coreset Pruning (GMC,
 * "Messages, Not Tokens: Grounded Coresets for Faithful VLM Compression",
 * arXiv 2608.02134).
 *
 * One call compresses B independent image boundaries.  For each image it
 *   1. builds the grounded message clients from the native causal attention
 *      of the text queries (Sec. 3.2, Eq. (1)-(2); appendix Eq.
 *      (cond-native-message) .. (cond-head-weight)), the appearance clients
 *      and the spatial clients (appendix Eq. (cond-aux-clients),
 *      (cond-coverage));
 *   2. selects K carriers with the batched responsibility solver (Sec. 3.3,
 *      Eq. (4); appendix Eq. (cond-responsibility) and its totality rule);
 *   3. assigns every visual token to a carrier and transports the population
 *      into it (Sec. 3.4, Eq. (5); appendix Eq. (cond-assignment),
 *      (cond-transport), (cond-grounded-energy), (cond-population-gate));
 *   4. physically compacts hidden states, K/V and position ids (Algorithm 1
 *      step 6 and the appendix paragraph on the index map).
 *
 * Conventions shared by every entry point
 *   - Every tensor pointer is a DEVICE pointer owned by the caller, except
 *     the gmc_problem / gmc_params structs themselves, which are host memory
 *     read during the call only.
 *   - The library allocates no device memory.  Scratch lives in the caller's
 *     workspace, sized by the matching *_workspace_size function; its
 *     address must be 256-byte aligned.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream).  The return value reports argument validation and
 *     launch errors only (GMC_OK or a GMC_ERR_* code); nothing is printed.
 *     Conditions the GPU detects (non-finite values when params->check_mode
 *     is 1, a bounded wait that gave up, text lengths above T) set bits of a
 *     status word inside the workspace; gmc_read_status() returns them.
 *   - Inputs are never written.  Outputs may not alias inputs or workspace.
 *   - Calls that share a workspace must not overlap in time.
 *   - Layouts are row-major and dense.  bf16 tensors hold IEEE bfloat16
 *     bit patterns; fp32 tensors IEEE binary32.
 *
 * Sequence layout of one image b: N visual tokens followed by T_b text
 * tokens (source rows 0..N-1 visual in raster order i = r*grid_w + c, then
 * N..N+T_b-1 text).  Text query t sits at sequence position N+t; its native
 * causal softmax covers all N visual keys and text keys 0..t.
 */
#ifndef GMC_H
#define GMC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* gmc_stream_t; /* identical to cudaStream_t */

/* return codes */
#define GMC_OK 0
#define GMC_ERR_ARG 1         /* a pointer is NULL/misaligned or a size is out of range */
#define GMC_ERR_UNSUPPORTED 2 /* valid request this build does not implement (shape limits below) */
#define GMC_ERR_WORKSPACE 3   /* ws_bytes smaller than the matching *_workspace_size() */
#define GMC_ERR_CUDA 4        /* a CUDA launch or query failed; cudaGetLastError() was cleared */

/* element types of hidden / keys / queries / out_hidden / out_kv */
#define GMC_F32 0
#define GMC_BF16 1

/* device status bits (gmc_read_status) */
#define GMC_STATUS_NONFINITE 0x1u  /* check_mode: a client, gain, mass or output was not finite */
#define GMC_STATUS_TIMEOUT 0x2u    /* a bounded device wait gave up; outputs are not valid */
#define GMC_STATUS_TEXT_LEN 0x4u   /* text_offsets gave some T_b < 1 or T_b > T */
#define GMC_STATUS_INTERNAL 0x8u   /* a device-side consistency check failed */

/* Shape limits of this build (GMC_ERR_UNSUPPORTED beyond them). */
#define GMC_MAX_N 8192            /* visual tokens per image */
#define GMC_MAX_POOL 128          /* pool_mult * batch_b */
#define GMC_MAX_HEADS 64          /* H */
#define GMC_MAX_VIEWS 4           /* message views: the current one and up to 3 historical ones */
#define GMC_MAX_PREFIX_LAYERS 64  /* dense prefix layers gathered by gmc_compress_ex */
#define GMC_MAX_N_LONG 16384      /* visual tokens per image on the long-prefix path */
#define GMC_MAX_POOL_WIDE 4096    /* pool_mult * batch_b on the long-prefix path and gmc_select */
#define GMC_MAX_RANK 256          /* rows of the long-prefix Rademacher map */

/*
 * Method constants.  gmc_default_params() fills the values of the paper's
 * Table "Shared GMC configuration" (fixed-token settings).  Where the paper
 * gives no number (resp_eps, beta_G for a current-view-only run, rms_eps,
 * norm_eps) the default is this library's choice, stated beside the field.
 */
typedef struct gmc_params {
  int batch_b;             /* 16:  responsibility batch b (Eq. (4)) */
  int pool_mult;           /* 4:   candidate pool = pool_mult * batch_b largest gains */
  float resp_temp;         /* 0.1: responsibility temperature factor */
  float resp_eps;          /* 1e-12 (not given in the paper): epsilon of Eq. (4) */
  float tau_v;             /* 0.2: appearance temperature */
  float tau_s;             /* 0.02: spatial temperature (clients and assignment) */
  float beta_G;            /* 0.5: grounded bank mass; the paper's current-view share */
  float beta_V;            /* 0.5: appearance bank mass */
  float beta_S;            /* 0.25: spatial bank mass */
  int landmarks;           /* 16:  landmarks x landmarks spatial clients */
  int max_head_clusters;   /* 4:   farthest-first head clusters */
  float head_eps;          /* 0.05: (d_h + head_eps)^-1 head weights */
  float terminal_q_weight; /* 2:   weight of the terminal prompt query */
  float lambda_mass;       /* 1:   lambda_mass of Eq. (1) */
  float eps_mass;          /* 1e-8: epsilon_mass of Eq. (1) */
  float assign_spatial_w;  /* 0.5: lambda_p, spatial weight of the assignment */
  float gate_scale;        /* 0.08: separability gate scale */
  float gate_pow;          /* 8:    separability gate power */
  float ambig_margin;      /* 0.05: local ambiguity margin */
  float pop_strength;      /* 0.5: alpha, grounded population strength */
  float rms_eps;           /* 1e-6 (not given; a common RMSNorm epsilon): epsilon of R_j */
  float norm_eps;          /* 1e-12 (not given): epsilon of h / max(||h||, eps) */
  int check_mode;          /* 0: off; 1: finite-value checks -> GMC_STATUS_NONFINITE */
} gmc_params;

/* Fill *p with the defaults above.  Never fails. */
void gmc_default_params(gmc_params* p);

/*
 * Problem description shared by gmc_compress / gmc_transport and the sizing
 * functions.
 */
typedef struct gmc_problem {
  int B;                       /* boundaries (prompts) in the call, >= 1 */
  int grid_h, grid_w;          /* source grid of every image; N == images * grid_h * grid_w */
  int Hkv;                     /* key/value heads; H % Hkv == 0, query head h reads h / (H/Hkv) */
  int dtype;                   /* GMC_F32 or GMC_BF16 */
  const int32_t* text_offsets; /* DEVICE int32[B+1]: offsets[0] = 0, T_b = offsets[b+1]-offsets[b],
                                  1 <= T_b <= T; or NULL: every image has exactly T text tokens */
  int images;                  /* images of every prompt, 0 or 1 = one (Sec. 3.1 I): the visual
                                  segment holds them one after another, grid_h x grid_w tokens
                                  each in raster order; the budget is min(N, max(K, images)), the
                                  support starts with each image's best singleton-gain token,
                                  appearance and spatial clients (one landmark grid per image)
                                  cover their own image, and every token is assigned to a
                                  carrier of its own image (appendix "Appearance and spatial
                                  clients", "Batched complementary support", Eq.
                                  (cond-assignment)).  gmc_transport* ignore it. */
} gmc_problem;

/* Bytes of workspace gmc_compress needs for this problem (0 on invalid arguments). */
size_t gmc_workspace_size(const gmc_problem* prob, int N, int T, int H, int d, int D, int K);

/*
 * Completed historical message views (appendix "Native message clients"):
 * earlier layers' text queries, keys/values and value-output probes of the
 * same images.  Each view adds its own grounded client rows (beta_hist is
 * shared equally by the views; the current view keeps params->beta_G), the
 * head patterns concatenate every view (Eq. (cond-head-pattern)), and the
 * message energy stays the current view's.  Every pointer has the layout of
 * the corresponding gmc_compress argument.
 */
typedef struct gmc_views {
  int n;                                     /* historical views, 0 .. GMC_MAX_VIEWS-1 */
  float beta_hist;                           /* their total grounded mass (0.5) */
  const void* keys[GMC_MAX_VIEWS - 1];       /* per view: keys then values, as `keys` */
  const void* queries[GMC_MAX_VIEWS - 1];    /* per view: text queries, as `queries` */
  const float* vo_probe[GMC_MAX_VIEWS - 1];  /* per view: W_h = O_h P of that layer */
} gmc_views;

/* Workspace of gmc_compress_views with n_views historical views (0 on invalid arguments). */
size_t gmc_workspace_size_views(const gmc_problem* prob, int n_views, int N, int T, int H, int d,
                                int D, int K);

/*
 * gmc_compress -- one GMC boundary compression per image (Algorithm 1, steps 2-6).
 *
 * Let Tb = T_b, Rb = N + T_b, Kb = K (after the budget rule), with per-image
 * row offsets  s_b = b*N + off_b  and  o_b = b*Kb + off_b, where off_b =
 * text_offsets[b] (or b*T when text_offsets is NULL).
 *
 *   hidden    [rows s_b .. s_b+Rb-1][D]          boundary residual states h (visual first)
 *   keys      [2*s_b .. : K block Rb rows then V block Rb rows][Hkv][d]
 *             i.e. image b occupies 2*Rb*Hkv*d elements starting at element
 *             2*s_b*Hkv*d: its post-RoPE keys, then its values
 *   queries   [rows off_b .. off_b+Tb-1][H][d]    post-RoPE text queries
 *   pos_ids   int32 [3*s_b ..: 3 rows of Rb]     (t, h, w) position ids (1-D models repeat one id)
 *   vo_probe  fp32 [H][d][4]                      W_h = O_h P, the value->output block of head h
 *                                                 times the rank-4 orthonormal probe P (Eq. (1));
 *                                                 shared by all images
 *   N, T, H, d, D, K                              visual tokens, text tokens (max over images when
 *                                                 ragged), query heads, head dim, hidden dim,
 *                                                 requested budget K_r
 * Outputs (K below is the realized budget min(N, max(K_r, 1))):
 *   out_idx    int32 [b*K .. +K]                  kept source visual indices, ascending
 *   out_hidden [rows o_b .. o_b+K+Tb-1][D]        transported carriers (ascending source order)
 *                                                 then the text rows, bit-exact copies
 *   out_kv     image b at element 2*o_b*Hkv*d:    K rows then V rows, each (K+Tb) x Hkv x d,
 *                                                 gathered at the kept sequence rows (bit-exact)
 *   out_pos    int32 [3*o_b ..: 3 rows of K+Tb]   original position ids of the kept rows
 *   trace      NULL, or gmc_trace_size() bytes per image of diagnostics (layout below)
 * K == N (after clamping) copies every input row unchanged (identity).
 *
 * Limits: 1 <= N <= GMC_MAX_N, N == grid_h*grid_w, T >= 1, 1 <= H <= GMC_MAX_HEADS,
 * H % Hkv == 0, d <= 1024 and D <= 8192, d a multiple of 8 (bf16) or 4 (fp32),
 * and H <= 56 in this build (the head-pattern statistics of one token block
 * must fit a block's 227 KB of shared memory; GMC_ERR_UNSUPPORTED above),
 * D a multiple of 8.  hidden/keys/queries/vo_probe/out_hidden/out_kv must be
 * 16-byte aligned, trace 16-byte aligned.
 *
 * Selection runs on one thread-block cluster per image while its state (a
 * copy of every token's gain, bucket and pool slot, and a share of the M
 * client rows per CTA) fits a CTA's shared memory; beyond that (with the
 * default parameters, N above about 7,700 at H = 28 and T = 128) every round runs
 * on the whole GPU, with the same decisions.  A multi-image prompt
 * (images > 1) that does not fit the cluster returns GMC_ERR_UNSUPPORTED.
 */
int gmc_compress(const gmc_problem* prob, const gmc_params* params, const void* hidden,
                 const void* keys, const void* queries, const int32_t* pos_ids,
                 const float* vo_probe, int N, int T, int H, int d, int D, int K,
                 int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                 void* workspace, size_t ws_bytes, void* trace, gmc_stream_t stream);

/*
 * gmc_compress_host -- gmc_compress from and to HOST memory (a deployment
 * variant; the paper has no counterpart).  The caller passes its inputs in
 * page-locked host memory, device buffers to copy them into (the layouts and
 * alignment of gmc_compress's inputs), the device outputs and page-locked
 * host buffers for them.  The call enqueues, on `stream` and the library's
 * side stream:
 *   - the copies of keys, queries, vo_probe and pos_ids on `stream`;
 *   - the copy of the hidden states on the side stream, after everything
 *     enqueued on `stream` before the call (so a previous call that still
 *     reads `d_hidden` is not overwritten), beside the probe, the message
 *     slice and the heads, which do not read the hidden states; the row norms
 *     and the cosine Gram follow it there, and `stream` joins the side stream
 *     before the first kernel on it that reads them;
 *   - gmc_compress on the device buffers;
 *   - the copies of the four outputs back to the host buffers on `stream`.
 * It returns once that is enqueued: synchronise `stream` before reading the
 * host outputs or reusing the host inputs.  Byte counts are the caller's
 * (every input and output of the call, e.g. hidden: (B*N + sum_b T_b) * D *
 * element size).  Returns GMC_OK or the error gmc_compress returns
 * (GMC_ERR_ARG also for a NULL pointer or a zero byte count).
 */
typedef struct gmc_host_io {
  /* inputs: page-locked HOST memory, then the DEVICE buffers they are copied to */
  const void* hidden;    void* d_hidden;    size_t hidden_bytes;
  const void* keys;      void* d_keys;      size_t keys_bytes;
  const void* queries;   void* d_queries;   size_t queries_bytes;
  const int32_t* pos_ids; int32_t* d_pos_ids; size_t pos_ids_bytes;
  const float* vo_probe; float* d_vo_probe; size_t vo_probe_bytes;
  /* outputs: DEVICE buffers of gmc_compress, then the page-locked HOST copies */
  int32_t* d_out_idx;    int32_t* out_idx;  size_t out_idx_bytes;
  void* d_out_hidden;    void* out_hidden;  size_t out_hidden_bytes;
  void* d_out_kv;        void* out_kv;      size_t out_kv_bytes;
  int32_t* d_out_pos;    int32_t* out_pos;  size_t out_pos_bytes;
} gmc_host_io;

int gmc_compress_host(const gmc_problem* prob, const gmc_params* params, const gmc_host_io* io,
                      int N, int T, int H, int d, int D, int K, void* workspace, size_t ws_bytes,
                      void* trace, gmc_stream_t stream);

/* gmc_compress with historical message views (views NULL or n == 0: gmc_compress). */
int gmc_compress_views(const gmc_problem* prob, const gmc_params* params, const gmc_views* views,
                       const void* hidden, const void* keys, const void* queries,
                       const int32_t* pos_ids, const float* vo_probe, int N, int T, int H, int d,
                       int D, int K, int32_t* out_idx, void* out_hidden, void* out_kv,
                       int32_t* out_pos, void* workspace, size_t ws_bytes, void* trace,
                       gmc_stream_t stream);

/*
 * Dense prefix layers for the cached path (appendix "Index map and physical
 * token accounting"): the prompt K/V that blocks 0 .. p-1 already computed are
 * kept, unchanged, at the retained sequence rows -- the selected visual rows
 * in ascending order, then every text row, the rows out_kv uses -- while the
 * boundary layer and the layers after it see the transported states.  Layer
 * l's input has the layout of `keys` ([B][2][N+T_b][Hkv][d], K then V) and
 * its output the layout of `out_kv` ([B][2][K+T_b][Hkv][d]); the gather is
 * bit-exact and runs in the same kernel as the compaction.
 */
typedef struct gmc_prefix_kv {
  int n_layers;                              /* p, 0 .. GMC_MAX_PREFIX_LAYERS */
  const void* keys[GMC_MAX_PREFIX_LAYERS];   /* per layer: device input, as `keys` */
  void* out_kv[GMC_MAX_PREFIX_LAYERS];       /* per layer: device output, as `out_kv` */
} gmc_prefix_kv;

/*
 * gmc_compress_ex -- gmc_compress with historical message views and dense
 * prefix layers (either may be NULL; both NULL is gmc_compress).  Workspace:
 * gmc_workspace_size_views with views->n (the prefix layers need none).  The
 * prefix outputs may not alias any input or other output.
 */
int gmc_compress_ex(const gmc_problem* prob, const gmc_params* params, const gmc_views* views,
                    const gmc_prefix_kv* prefix, const void* hidden, const void* keys,
                    const void* queries, const int32_t* pos_ids, const float* vo_probe, int N,
                    int T, int H, int d, int D, int K, int32_t* out_idx, void* out_hidden,
                    void* out_kv, int32_t* out_pos, void* workspace, size_t ws_bytes,
                    void* trace, gmc_stream_t stream);

/*
 * Long prefixes: the bounded appearance bank (appendix "Appearance and spatial
 * clients", last paragraph; the cost notes after Algorithm 1; Table "Shared
 * GMC configuration", long-prefix row: rank 128, Rademacher seed 104729,
 * M_V <= 4096, b = 512).  The appearance states are the boundary states under a
 * fixed rank-r map R with entries +-1, normalised after the map:
 * x~_i = R h_i / max(||R h_i||, norm_eps).  The appearance clients are the
 * M_V = min(N, max_clients) uniformly spaced tokens c(m) = floor(m N / M_V);
 * row m is softmax_i(x~_{c(m)} . x~_i / tau_v), beta_V / M_V each.  The
 * assignment uses the cosines of the unprojected states against the support
 * only (an N x K product), and every solver round runs on the whole GPU.
 */
typedef struct gmc_long_prefix {
  int rank;                /* r, a multiple of 8, 8 .. GMC_MAX_RANK (128 in the paper) */
  int max_clients;         /* M_V cap, >= 1 (4096 in the paper) */
  const void* rademacher;  /* DEVICE bf16 [r][D], entries -1 or +1 (exact in bf16); 16-byte
                              aligned; read only */
} gmc_long_prefix;

/* Workspace of gmc_compress_long with n_views historical views (0 on invalid
 * arguments).  Unlike gmc_workspace_size it depends on params (the pool size). */
size_t gmc_workspace_size_long(const gmc_problem* prob, const gmc_params* params,
                               const gmc_long_prefix* lp, int n_views, int N, int T, int H, int d,
                               int D, int K);

/*
 * gmc_compress_long -- gmc_compress_ex with the bounded appearance bank of long
 * prefixes (lp must not be NULL; views and prefix may be NULL).  Arguments,
 * layouts, outputs and the trace are those of gmc_compress_ex; the trace's
 * appearance bank values F_S[1] / F_V[1] are the bounded bank's.  params may
 * set pool_mult * batch_b up to GMC_MAX_POOL_WIDE (the paper's b = 512 gives a
 * pool of 2048).
 * Limits: bf16 states, one image per prompt (images 0 or 1), 256 <= N <=
 * GMC_MAX_N_LONG, and the limits of gmc_compress otherwise; GMC_ERR_UNSUPPORTED
 * beyond them, GMC_ERR_ARG for a NULL, misaligned or out-of-range lp.
 */
int gmc_compress_long(const gmc_problem* prob, const gmc_params* params,
                      const gmc_long_prefix* lp, const gmc_views* views,
                      const gmc_prefix_kv* prefix, const void* hidden, const void* keys,
                      const void* queries, const int32_t* pos_ids, const float* vo_probe, int N,
                      int T, int H, int d, int D, int K, int32_t* out_idx, void* out_hidden,
                      void* out_kv, int32_t* out_pos, void* workspace, size_t ws_bytes,
                      void* trace, gmc_stream_t stream);

/*
 * gmc_clients_long -- gmc_clients with the bounded appearance bank: out_clients
 * receives float[B][M][N] with M = (1 + views->n) * H * T + M_V + landmarks^2
 * (grounded rows, then the M_V appearance rows, then the spatial rows).
 * Workspace: gmc_workspace_size_long.
 */
int gmc_clients_long(const gmc_problem* prob, const gmc_params* params, const gmc_long_prefix* lp,
                     const gmc_views* views, const void* hidden, const void* keys,
                     const void* queries, const int32_t* pos_ids, const float* vo_probe, int N,
                     int T, int H, int d, int D, int K, float* out_clients, void* workspace,
                     size_t ws_bytes, void* trace, gmc_stream_t stream);

/*
 * Diagnostics trace (optional).  Image b's record starts at byte
 * b * gmc_trace_size(...) / B.  All fields are 4-byte words.
 */
typedef struct gmc_trace_header {
  int32_t K;          /* realized budget */
  int32_t rounds;     /* selection rounds run, a final zero-gain fill included */
  int32_t n_clusters; /* nonempty head clusters C */
  int32_t filled;     /* tokens added by the zero-gain fill */
  float s_x;          /* separability gate */
  float delta_bar;    /* mean best-minus-second-best selected cosine over discarded tokens */
  float F_S[3];       /* F_b(S) for the grounded, appearance, spatial banks */
  float F_V[3];       /* F_b(V) */
  float c_B;          /* batched certificate 1 - prod_t (1 - q_t) over the rounds with U_t > 0,
                         q_t = [F(S_t u B_t) - F(S_t)] / U_t, U_t the sum of the K largest
                         singleton gains of unselected tokens (Sec. 4.1 Eq. (6); appendix Eq.
                         (cond-batched-bound)), from the round gains and coverage below */
  int32_t reserved[3];
} gmc_trace_header;

typedef struct gmc_trace_layout {
  size_t bytes_per_image; /* the record size; gmc_trace_size() = B * bytes_per_image */
  int rounds_max;         /* ceil(K / batch_b) + 1, + 1 for prompts of several images */
  int pool_size;          /* pool_mult * batch_b */
  /* byte offsets inside one record */
  size_t off_order;       /* int32[K]   indices in the order they entered the support */
  size_t off_round_end;   /* int32[rounds_max]  prefix count of `order` after each round */
  size_t off_pool;        /* int32[rounds_max][pool_size] pool of each round (-1 padded);
                             a fill round has an empty pool */
  size_t off_centres;     /* int32[max_head_clusters]  centre heads in farthest-first order */
  size_t off_head_assign; /* int32[H]   cluster (index into centres) of each head */
  size_t off_omega;       /* float[H]   head weights omega_h */
  size_t off_pi;          /* int32[N]   representative of every visual token */
  size_t off_ebar;        /* float[N]   normalised message energy */
  size_t off_mass;        /* float[N]   population weights m_i */
  size_t off_gains;       /* int64[rounds_max][N]  singleton gains at the start of each round,
                             fixed point (scale 2^e, e = 61 - ceil(log2(total bank mass))) */
  size_t off_cover;       /* int64[rounds_max]  F(S) after each round, same fixed point */
} gmc_trace_layout;

/* Fill *out for this problem.  Returns GMC_OK or GMC_ERR_ARG. */
int gmc_get_trace_layout(const gmc_problem* prob, const gmc_params* params, int N, int T, int H,
                         int K, gmc_trace_layout* out);
/* B * bytes_per_image, or 0 on invalid arguments. */
size_t gmc_trace_size(const gmc_problem* prob, const gmc_params* params, int N, int T, int H,
                      int K);

/*
 * gmc_select -- the batched responsibility solver alone (Sec. 3.3, Eq. (4);
 * appendix Eq. (cond-responsibility)) on caller-built client matrices.
 *   clients  fp32 [B][M][N], every entry >= 0 (the preweighted Cbar of Eq. (cond-coverage));
 *            read only
 *   out_idx  int32 [B][K] the support, ascending
 *   trace    NULL or B records laid out as gmc_get_trace_layout with H = 0
 *            (order, round_end, pool and the header's K / rounds / filled are written)
 * 1 <= K <= N <= GMC_MAX_N, M >= 1.  The clients are copied into the workspace
 * first, so `clients` is never written.  A pool pool_mult * batch_b above
 * GMC_MAX_POOL (up to GMC_MAX_POOL_WIDE) runs every round on the whole GPU, the
 * solver of gmc_compress_long, and allows N up to GMC_MAX_N_LONG; so does a
 * problem whose cluster-solver state does not fit a CTA's shared memory (as in
 * gmc_compress).
 */
size_t gmc_select_workspace_size(int B, int M, int N, int K, const gmc_params* params);
int gmc_select(const float* clients, int B, int M, int N, int K, const gmc_params* params,
               int32_t* out_idx, void* workspace, size_t ws_bytes, void* trace,
               gmc_stream_t stream);

/*
 * gmc_cosine -- the cosine matrix of the visual boundary states alone,
 * cos_ij = h_i . h_j / (max(||h_i||, eps) max(||h_j||, eps)) (appendix Eq.
 * (cond-aux-clients), (cond-assignment)), as gmc_compress computes it: bf16
 * states on the tcgen05 tensor cores with fp32 accumulation, fp32 states on
 * CUDA cores.  hidden as gmc_compress (only the visual rows are read);
 * out_cos fp32 [B][N][N].  d is not used.
 */
size_t gmc_cosine_workspace_size(const gmc_problem* prob, int N);
int gmc_cosine(const gmc_problem* prob, const gmc_params* params, const void* hidden, int N,
               int T, int D, float* out_cos, void* workspace, size_t ws_bytes,
               gmc_stream_t stream);

/*
 * gmc_transport -- population transport and physical compaction for a given
 * support and assignment (Sec. 3.4, Eq. (5); appendix Eq. (cond-transport);
 * Algorithm 1 step 6).  Inputs as gmc_compress, plus
 *   support  int32 [B][K]  ascending selected visual indices
 *   assign   int32 [B][N]  pi(i), an element of the image's support; pi(j) = j on the support
 *   weights  fp32  [B][N]  population weights m_i > 0
 * Outputs out_idx / out_hidden / out_kv / out_pos exactly as gmc_compress.
 * Here K is the support size (1 <= K <= N), not a request.
 */
size_t gmc_transport_workspace_size(const gmc_problem* prob, int N, int T, int K);
int gmc_transport(const gmc_problem* prob, const gmc_params* params, const void* hidden,
                  const void* keys, const int32_t* pos_ids, const int32_t* support,
                  const int32_t* assign, const float* weights, int N, int T, int d, int D, int K,
                  int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                  void* workspace, size_t ws_bytes, gmc_stream_t stream);

/*
 * gmc_transport_noalloc -- gmc_transport for callers that cannot allocate
 * device memory.  The paper has no counterpart: this is a deployment variant.
 *
 * Who needs it: code that may only launch work into memory someone else
 * already owns -- an inference-engine plugin inside its enqueue(), a caller
 * that is inside a CUDA graph capture (an allocation there breaks or
 * invalidates the capture), a server whose device pool is fixed at start-up.
 * Such callers pass inputs and outputs exactly as for gmc_transport, but no
 * workspace: the scratch (a status word and one float per visual row) lives
 * in a fixed array inside libgmc.so, sized for GMC_NOALLOC_MAX_ROWS visual
 * rows (B * N) plus 256 bytes.  Every GPU that loads the library keeps that
 * array (about 256 KiB) until the process exits.
 *
 *   - Larger problems (B * N > GMC_NOALLOC_MAX_ROWS) are rejected with
 *     GMC_ERR_UNSUPPORTED before anything is launched.
 *   - It calls no cudaMalloc, cudaFree or other allocating routine.
 *   - The first call made in a CUDA context (normally the device's primary
 *     context) looks up the array's device address (cudaGetSymbolAddress)
 *     and caches it for that context; make that first call before any
 *     stream capture that includes this entry point.  After cudaDeviceReset
 *     the new primary context gets a fresh look-up on its first call.
 *   - All calls share the one array.  Calls that overlap on the GPU (other
 *     streams, other host threads) race on it; serialise them.  The status
 *     word is cleared at the start of every call; the rest is overwritten.
 *   - device_status: NULL, or a caller-owned device uint32 that receives the
 *     GMC_STATUS_* bits of this call (cleared first); with NULL the bits stay
 *     in the library's array and cannot be read back.
 *   - Its kernels are not counted by gmc_launch_count().
 * Arguments, layouts and results are those of gmc_transport.
 */
#define GMC_NOALLOC_MAX_ROWS 65536
int gmc_transport_noalloc(const gmc_problem* prob, const gmc_params* params, const void* hidden,
                          const void* keys, const int32_t* pos_ids, const int32_t* support,
                          const int32_t* assign, const float* weights, int N, int T, int d, int D,
                          int K, int32_t* out_idx, void* out_hidden, void* out_kv,
                          int32_t* out_pos, uint32_t* device_status, gmc_stream_t stream);

/*
 * gmc_clients -- the client matrix alone (steps 1 of gmc_compress): grounded
 * message clients (Sec. 3.2, Eq. (1)-(2); appendix Eq. (cond-native-message)
 * .. (cond-head-weight)), appearance and spatial clients (appendix Eq.
 * (cond-aux-clients), (cond-coverage)), written to out_clients as
 * float[B][M][N] with M = (1 + views->n) * H * T + N + landmarks^2.  Image b's
 * rows: grounded (view, head, text query) view-major then head-major for its
 * own T_b, then N appearance rows, then landmarks^2 spatial rows; rows past
 * that (ragged images) are left unspecified.  Arguments, workspace (sized by
 * gmc_workspace_size / gmc_workspace_size_views) and trace are those of
 * gmc_compress_views (views may be NULL); the trace receives the head
 * clustering fields.  The selection, assignment, transport and compaction do
 * not run.  Returns GMC_OK or a GMC_ERR_* code.
 */
int gmc_clients(const gmc_problem* prob, const gmc_params* params, const gmc_views* views,
                const void* hidden, const void* keys, const void* queries, const int32_t* pos_ids,
                const float* vo_probe, int N, int T, int H, int d, int D, int K,
                float* out_clients, void* workspace, size_t ws_bytes, void* trace,
                gmc_stream_t stream);

/*
 * gmc_selftest_bounded_wait -- checks the failure path of the bounded device
 * waits (no counterpart in the paper).  A one-block kernel waits, with the
 * library's clock-bounded mbarrier wait, on a barrier phase that nothing ever
 * completes; after `cycles` SM clocks (0 .. 4e9) it sets GMC_STATUS_TIMEOUT
 * in the status word at the start of `workspace` (256-byte aligned, >= 4
 * bytes; cleared first) and returns.  The context stays usable.  Read the
 * bit with gmc_read_status.  Returns GMC_OK, GMC_ERR_ARG or GMC_ERR_CUDA.
 */
int gmc_selftest_bounded_wait(long long cycles, void* workspace, size_t ws_bytes,
                              gmc_stream_t stream);

/*
 * Synchronise `stream`, then copy the device status word of `workspace`
 * (as passed to the last call that used it) into *status.  The word is
 * cleared at the start of every gmc_compress / gmc_select / gmc_transport
 * call.  Returns GMC_OK or GMC_ERR_ARG / GMC_ERR_CUDA.
 */
int gmc_read_status(const void* workspace, uint32_t* status, gmc_stream_t stream);

/*
 * Benchmark instrumentation (no counterpart in the paper).
 * gmc_profile_enable(1): later gmc_compress calls record a CUDA event on
 *   their stream before the first and after every stage (9 stages: row
 *   norms, probe, message slice, head weights, cosine Gram, client matrix,
 *   selection, assignment, transport + compaction).  0 turns it off.  Not for
 *   use during stream capture.
 * gmc_profile_read(ms, names, max): waits for the last profiled call and
 *   writes up to `max` per-stage durations in milliseconds (and, if `names`
 *   is not NULL, static stage names); returns the number of stages, or -1 if
 *   no profiled call has run.
 * gmc_launch_count(): total kernels this library has launched in the process
 *   (memsets and copies not counted).
 */
int gmc_profile_enable(int on);
int gmc_profile_read(float* ms, const char** names, int max);
uint64_t gmc_launch_count(void);

/* Static string naming a return code. */
const char* gmc_error_string(int code);

/* Library version, e.g. "gmc 0.1.0 sm_103a". */
const char* gmc_version(void);

#ifdef __cplusplus
}
#endif
#endif /* GMC_H */
