/*
 * bitlogic.h -- C ABI of the GB300 (sm_103a) LUT-network hot path.
 *
 * The library implements the data-parallel hot path of BitLogic's
 * gradient-based LUT networks (arXiv 2602.07400): the thermometer encoder
 * (with the quantile fit of its thresholds), the soft forward/backward of a
 * LUT layer (LightLUT soft or straight-through hard node; fixed connectivity
 * or learnable routing over candidate pools), the group-sum head with
 * temperature and cross-entropy, the AdamW update of the logits, and the
 * hard bit-packed evaluation mode with a popcount group-sum.  Every call is
 * a hand-written CUDA kernel sequence enqueued on the caller's stream.
 *
 * Conventions shared by all calls
 *   - Pointers marked "device" are caller-owned device memory; the library
 *     never allocates, frees or synchronizes inside a compute call.  Arrays
 *     marked "host" are read before the call returns.
 *   - Every compute call enqueues its kernels on `stream` and returns a
 *     status code (bitlogic_status_t).  Arguments are validated on the host
 *     before any launch; a rejected call launches nothing.  No kernel traps
 *     or asserts: a connectivity or CSR index that is out of range is read as
 *     index 0 and recorded in a device-side flag that
 *     bitlogic_device_error() reports.
 *   - Layouts:
 *       raw samples      x[s*d + j]             uint8, sample-major
 *       soft activations X[row*B + s]           fp32, feature-major
 *       connectivity     conn[j*k + i]          int32, slot i of node j
 *       table logits     theta[j*2^k + a]       fp32
 *       hard tables      table[j], bit a        uint64 = entry a of node j
 *       packed bits      xp[row*W + s/32], bit s%32, W = ceil(N/32)
 *     Slot i of a node is bit i of its table index a.
 *   - Vectorised (16-byte) paths are taken when B % 4 == 0 and the arrays are
 *     16-byte aligned; otherwise a scalar path runs.  Integer, byte and bit
 *     results are identical on both; floating-point results agree within
 *     rounding (the soft forward evaluates its table in another order on the
 *     vector path), and each path is deterministic from run to run.
 */
#ifndef BITLOGIC_H
#define BITLOGIC_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    BITLOGIC_OK = 0,
    BITLOGIC_ERR_NULL = -1,       /* a required pointer is NULL */
    BITLOGIC_ERR_SHAPE = -2,      /* size <= 0, overflow, or w % C != 0 */
    BITLOGIC_ERR_FANIN = -3,      /* k outside 1..6, or k > w_in */
    BITLOGIC_ERR_ALIGN = -4,      /* workspace not 16-byte aligned */
    BITLOGIC_ERR_WORKSPACE = -5,  /* workspace smaller than the query result */
    BITLOGIC_ERR_CUDA = -6,       /* a CUDA launch or copy failed */
    BITLOGIC_ERR_INDEX = -7,      /* index out of range (host-side check) */
    BITLOGIC_ERR_DEVICE = -8,     /* device-side index check tripped */
    BITLOGIC_ERR_THRESH = -9,     /* thresholds: b outside 1..32 */
    BITLOGIC_ERR_TOO_LARGE = -10, /* sizes beyond bitlogic_head_loss_noalloc's fixed scratch */
    BITLOGIC_ERR_HYPER = -11,     /* optimizer hyperparameter out of range */
    BITLOGIC_ERR_NODE = -12       /* unknown node form */
} bitlogic_status_t;

/* Node forms of the LightLUT parameterization (§2 "Gradient-based LUT
 * methods"; the node sweep of §4 lists both):
 *   BITLOGIC_NODE_SOFT  table entry t_a = sigmoid(theta_a) in the forward.
 *   BITLOGIC_NODE_ST    straight-through hard sampling: the forward uses the
 *                       discretized entry t_a = [theta_a > 0] (the value
 *                       bitlogic_binarize_tables deploys; theta = 0 gives 0),
 *                       the input gradient is that of the hard-table forward,
 *                       and the table gradient reaches theta through the
 *                       sigmoid slope as if t_a were sigmoid(theta_a). */
typedef enum {
    BITLOGIC_NODE_SOFT = 0,
    BITLOGIC_NODE_ST = 1
} bitlogic_node_t;

/* Thermometer encoder E: R^d -> {0,1}^{db} (paper §3, "Encoders and heads";
 * linear thermometer with b thresholds, b+1 levels on b wires).
 *   x        device uint8 [B][d]   raw samples
 *   thr_host host uint8 [b]        thresholds, 1 <= b <= 32
 *   bits     device fp32 [d*b][B]  bits[(j*b+i)*B + s] = (x[s][j] > thr[i])
 * B == 0 is a no-op. */
int bitlogic_encode_thermometer(const uint8_t* x, int64_t B, int32_t d,
                                const uint8_t* thr_host, int32_t b,
                                float* bits, cudaStream_t stream);

/* The same wires as bytes (0 or 1): bits device uint8 [d*b][B], for
 * consumers that gather the encoder rows and want a quarter of the bytes
 * (bitlogic_route_forward_u8). */
int bitlogic_encode_thermometer_u8(const uint8_t* x, int64_t B, int32_t d,
                                   const uint8_t* thr_host, int32_t b,
                                   uint8_t* bits, cudaStream_t stream);

/* Both forms in one pass: bits device fp32 [d*b][B] and bits8 device uint8
 * [d*b][B], the same wires (for a step whose forward reads fp32 rows and
 * whose backward gathers bytes).  BITLOGIC_ERR_NULL when bits8 is NULL. */
int bitlogic_encode_thermometer_both(const uint8_t* x, int64_t B, int32_t d,
                                     const uint8_t* thr_host, int32_t b,
                                     float* bits, uint8_t* bits8, cudaStream_t stream);

/* The same wires at one bit per sample ("wire bit rows"), for the soft
 * layer-1 kernels on binary wires (bitlogic_lut_forward_bitrows,
 * bitlogic_lut_backward_bitrows): an eighth of the bytes of byte rows.  The
 * batch is cut into blocks of 1024 samples; each wire row holds 32 words
 * per block, W = 32 * ceil(B / 1024) words in all, and bit 8m + r of word L
 * of block q is the wire of sample 1024q + 128r + 4L + m (r < 8, m < 4), the
 * order in which those kernels' lanes visit the samples.  Samples past B
 * read 0.
 *   bits  device uint32 [d*b][W]
 * Any B and alignment of x; B == 0 is a no-op.  Returns BITLOGIC_ERR_NULL,
 * BITLOGIC_ERR_SHAPE, BITLOGIC_ERR_THRESH, BITLOGIC_ERR_CUDA. */
int bitlogic_encode_thermometer_bitrows(const uint8_t* x, int64_t B, int32_t d,
                                        const uint8_t* thr_host, int32_t b,
                                        uint32_t* bits, cudaStream_t stream);

/* Distributive (quantile) thermometer fit (§3 "Encoders and heads"; App. A
 * "Initialization": thresholds fit once from the empirical pixel quantiles
 * of the training split, over the globally flattened pixels, App. B).  Two
 * steps, so that a training split larger than device memory can be streamed
 * through in pieces and the library never synchronizes:
 *   bitlogic_pixel_histogram   device: hist[v] += number of bytes of x equal
 *                              to v (x device uint8 [n], any alignment; hist
 *                              device uint64 [256], zeroed by the caller
 *                              before the first piece).  n == 0 is a no-op.
 *   bitlogic_quantile_thresholds  host: from the finished histogram (copied
 *                              to the host, hist_host uint64 [256]), threshold
 *                              i = 1..b is the quantile at level i/(b+1) with
 *                              linear interpolation between order statistics,
 *                              floored to the integer that the encoder's
 *                              strict compare needs (pixel > floor(q) equals
 *                              pixel > q on integer pixels); exact integer
 *                              arithmetic.  thr_host uint8 [b], ascending and
 *                              possibly repeated (a point mass collapses
 *                              neighbouring thresholds).  1 <= b <= 32
 *                              (BITLOGIC_ERR_THRESH); an empty histogram gives
 *                              BITLOGIC_ERR_SHAPE. */
int bitlogic_pixel_histogram(const uint8_t* x, int64_t n, uint64_t* hist, cudaStream_t stream);
int bitlogic_quantile_thresholds(const uint64_t* hist_host, int32_t b, uint8_t* thr_host);

/* Soft LUT layer forward: one logic layer L_M(f_theta^(n)) of the paper's
 * Eq. (1) (§3), with the LightLUT node of §2 (Kronecker-indicator basis,
 * 2^k parameters per node) read as
 *   t = sigmoid(theta_j),  y_j(s) = sum_a t_a prod_i x_i^{a_i} (1-x_i)^{1-a_i},
 * x_i = X[conn[j][i]][s].  Evaluated as a 2^k-1 step lerp tree.
 *   X     device fp32 [w_in][B]     layer input
 *   conn  device int32 [w][k]       fixed connectivity (§3 "Connectivity")
 *   theta device fp32 [w][2^k]      table logits
 *   Y     device fp32 [w][B]        output, overwritten
 * 1 <= k <= 6, k <= w_in.  B == 0 is a no-op. */
int bitlogic_lut_forward(const float* X, int32_t w_in, int64_t B,
                         const int32_t* conn, const float* theta,
                         int32_t w, int32_t k, float* Y, cudaStream_t stream);

/* bitlogic_lut_forward for either node form: node is a bitlogic_node_t
 * (BITLOGIC_ERR_NODE otherwise); BITLOGIC_NODE_SOFT is bitlogic_lut_forward.
 * With BITLOGIC_NODE_ST and binary inputs every output is 0 or 1: the
 * deployed network's value, as bitlogic_hard_forward computes it. */
int bitlogic_lut_forward_node(const float* X, int32_t w_in, int64_t B,
                              const int32_t* conn, const float* theta,
                              int32_t w, int32_t k, int32_t node, float* Y,
                              cudaStream_t stream);

/* Bytes of workspace bitlogic_lut_backward needs (0 when want_dx == 0). */
size_t bitlogic_lut_backward_workspace(int32_t w_in, int64_t B, int32_t w,
                                       int32_t k, int32_t want_dx);

/* Soft LUT layer backward (chain rule through the forward above):
 *   dtheta[j][a] = t_a (1-t_a) sum_s dY[j][s] w_a(x(s))     (reduced over the
 *                  batch inside the kernel, deterministic order)
 *   dX[i][s]     = sum over edges (j, slot) with conn[j][slot] == i of
 *                  dY[j][s] * dy_j/dx_slot(s)
 * The input gradient uses the inverse-connectivity CSR map (off, edge) from
 * bitlogic_build_csr(): per-edge terms are written to the workspace and
 * summed per input in increasing edge order, so no atomics are used.
 *   X, conn, theta  as in bitlogic_lut_forward
 *   dY     device fp32 [w][B]
 *   csr_off  device int32 [w_in+1], csr_edge device int32 [w*k]
 *            (edge id = j*k + slot); required only when dX != NULL
 *   dtheta device fp32 [w][2^k]   overwritten (not accumulated)
 *   dX     device fp32 [w_in][B] or NULL (skips the input gradient)
 *   workspace device, 16-byte aligned, >= bitlogic_lut_backward_workspace() */
int bitlogic_lut_backward(const float* X, int32_t w_in, int64_t B,
                          const int32_t* conn, const float* theta,
                          int32_t w, int32_t k, const float* dY,
                          const int32_t* csr_off, const int32_t* csr_edge,
                          float* dtheta, float* dX,
                          void* workspace, size_t ws_bytes, cudaStream_t stream);

/* The two phases of bitlogic_lut_backward, for callers that time them
 * separately or consume the per-edge terms themselves.
 * bitlogic_lut_backward_edges: dtheta as above and, when edge_terms is not
 *   NULL, edge_terms[(j*k + i)*B + s] = dY[j][s] * dy_j/dx_i(s)
 *   (device fp32 [w*k][B], 16-byte aligned for the vector path).
 * bitlogic_csr_reduce: dX[i][s] = sum of edge_terms[csr_edge[p]][s] over the
 *   CSR positions p of input i, in increasing p (n_edges = w*k).  csr_edge
 *   may be NULL when the term rows are already stored in CSR order (row p,
 *   see edge_pos of bitlogic_lut_backward_ex): the sum then reads each
 *   input's rows as one contiguous block. */
int bitlogic_lut_backward_edges(const float* X, int32_t w_in, int64_t B,
                                const int32_t* conn, const float* theta,
                                int32_t w, int32_t k, const float* dY,
                                float* dtheta, float* edge_terms, cudaStream_t stream);
int bitlogic_csr_reduce(const float* edge_terms, int64_t B, const int32_t* csr_off,
                        const int32_t* csr_edge, int32_t w_in, int32_t n_edges,
                        float* dX, cudaStream_t stream);

/* bitlogic_lut_forward_node on byte rows (binary wires, each byte 0 or 1,
 * e.g. from bitlogic_encode_thermometer_u8; a byte is read by its lowest
 * bit).  On binary inputs the corner weights prod_i x_i^{a_i}(1-x_i)^{1-a_i}
 * are 1 for a = sum_i x_i 2^i and 0 for every other corner (§2: a soft node
 * on binary inputs returns its table entry), so
 *   Y[j][s] = t_a,  a = sum_i X[conn[j][i]][s] 2^i,
 * with t_a = sigmoid(theta_j[a]) (BITLOGIC_NODE_SOFT) or [theta_j[a] > 0]
 * (BITLOGIC_NODE_ST): a gather of k bytes and one table read per output.
 *   X     device uint8 [w_in][B];  conn, theta, Y, k, node as in
 *         bitlogic_lut_forward_node.
 * Any B and alignment (B % 4 == 0 with 4-byte aligned X and 16-byte aligned
 * Y takes the vector form).  Out-of-range connectivity raises the device
 * flag and reads row 0.  Returns BITLOGIC_ERR_NULL, BITLOGIC_ERR_SHAPE,
 * BITLOGIC_ERR_FANIN, BITLOGIC_ERR_NODE, BITLOGIC_ERR_CUDA. */
int bitlogic_lut_forward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                            const float* theta, int32_t w, int32_t k, int32_t node, float* Y,
                            cudaStream_t stream);

/* bitlogic_lut_forward_u8 on wire bit rows (the layout of
 * bitlogic_encode_thermometer_bitrows): X device uint32 [w_in][W], W = 32 *
 * ceil(B / 1024), 4-byte aligned (BITLOGIC_ERR_ALIGN otherwise).  Every
 * other argument, the result and the errors as bitlogic_lut_forward_u8: the
 * same wires give the same Y bit for bit.  B % 4 == 0 with 16-byte aligned
 * Y takes vector stores. */
int bitlogic_lut_forward_bitrows(const uint32_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                 const float* theta, int32_t w, int32_t k, int32_t node, float* Y,
                                 cudaStream_t stream);

/* General form of the layer backward, with the output gradient taken from
 * one of two sources (exactly one of dY and up_terms is non-NULL):
 *   dY rows:  node j reads row j / dy_group of dY ([w / dy_group][B]);
 *             dy_group = 1 is an ordinary dY [w][B]; dy_group = w / C takes
 *             the per-class gradient of bitlogic_head_loss_ex (the nodes of
 *             a class share one gradient row), so the full dY is never stored.
 *   up terms: dY[j][s] = sum over p in [up_off[j], up_off[j+1]) of
 *             up_terms[up_edge[p]][s], in increasing p -- the input gradient
 *             of the next layer (its per-edge terms and the CSR map of its
 *             connectivity, up_edges = w_next * k_next), reduced on the fly;
 *             the result equals bitlogic_csr_reduce of those terms bit for bit.
 *             up_edge may be NULL when the terms are stored in CSR order.
 * dtheta, edge_terms as in bitlogic_lut_backward_edges (edge_terms may be
 * NULL).  edge_pos (device int32 [w*k] or NULL): when given, the term of
 * edge e = j*k + i is stored at row edge_pos[e] instead of row e; with the
 * positions of bitlogic_csr_positions the rows come out in CSR order, so
 * their consumer reads each input's rows contiguously (a position outside
 * [0, w*k) raises the device flag and stores at row e).  dY_out (device fp32
 * [w][B] or NULL) receives the gradient used. */
int bitlogic_lut_backward_ex(const float* X, int32_t w_in, int64_t B,
                             const int32_t* conn, const float* theta,
                             int32_t w, int32_t k,
                             const float* dY, int32_t dy_group,
                             const float* up_terms, const int32_t* up_off,
                             const int32_t* up_edge, int32_t up_edges,
                             float* dtheta, float* edge_terms, const int32_t* edge_pos,
                             float* dY_out, cudaStream_t stream);

/* bitlogic_lut_backward_ex for either node form (node as in
 * bitlogic_lut_forward_node).  For BITLOGIC_NODE_ST:
 *   dtheta[j][a] = s_a (1 - s_a) sum_s dY[j][s] w_a(x(s)),  s_a = sigmoid(theta)
 *   (the straight-through estimate: the same expression as the soft node),
 *   and the edge terms use the hard entries [theta > 0]. */
int bitlogic_lut_backward_node(const float* X, int32_t w_in, int64_t B,
                               const int32_t* conn, const float* theta,
                               int32_t w, int32_t k, int32_t node,
                               const float* dY, int32_t dy_group,
                               const float* up_terms, const int32_t* up_off,
                               const int32_t* up_edge, int32_t up_edges,
                               float* dtheta, float* edge_terms, const int32_t* edge_pos,
                               float* dY_out, cudaStream_t stream);

/* Table gradient of a layer whose output gradient is recomputed through a
 * next layer of small fan-in (chain rule on the node of §2, the
 * multilinear form of the relaxed table): output row j of this layer is an
 * input of the next layer, and its gradient
 *   g[j][s] = sum over the CSR positions p in [up_off[j], up_off[j+1]) (in
 *             increasing p) of up_dY[j2 / up_group][s] * d y_j2 / d x_slot (s),
 *             edge up_edge[p] = j2 * up_k + slot,
 * where the derivative of next-layer node j2 with respect to its input slot
 * is a multilinear function of its other up_k - 1 inputs, read from Y.  So
 * neither the next layer's per-edge terms nor g is stored (g goes to dY_out
 * when that is given).  dtheta is then as in bitlogic_lut_backward_node
 * with g as the output gradient (overwritten, not accumulated).  `node`
 * applies to both layers (the next layer's table entries in the derivative;
 * the slope of the sigmoid in this layer's dtheta).
 *   X         device fp32 [w_in][B]: this layer's input
 *   conn      device int32 [w][k];  theta device fp32 [w][2^k]
 *   Y         device fp32 [w][B]: this layer's output (the next layer's input)
 *   up_conn   device int32 [up_w][up_k], entries in [0, w); up_theta fp32 [up_w][2^up_k]
 *   up_dY     device fp32 [up_w / up_group][B]: the next layer's output
 *             gradient, one row per group of up_group nodes
 *   up_off    device int32 [w + 1], up_edge device int32 [up_w * up_k] or
 *             NULL (identity): the CSR map of up_conn (bitlogic_build_csr)
 *   dtheta    device fp32 [w][2^k];  dY_out device fp32 [w][B] or NULL
 * Needs 1 <= up_k <= 3 (BITLOGIC_ERR_FANIN otherwise), B % 4 == 0 and
 * 16-byte aligned X, Y, up_dY and dY_out (BITLOGIC_ERR_ALIGN otherwise); B = 0
 * zeroes dtheta.  Out-of-range CSR positions, edge ids or rows raise the
 * device flag and contribute nothing.  Returns BITLOGIC_ERR_NULL,
 * BITLOGIC_ERR_SHAPE (up_w % up_group != 0), BITLOGIC_ERR_NODE,
 * BITLOGIC_ERR_CUDA. */
int bitlogic_lut_backward_through(const float* X, int32_t w_in, int64_t B, const int32_t* conn,
                                  const float* theta, int32_t w, int32_t k, int32_t node,
                                  const float* Y, const int32_t* up_conn, const float* up_theta,
                                  int32_t up_w, int32_t up_k, const float* up_dY, int32_t up_group,
                                  const int32_t* up_off, const int32_t* up_edge, float* dtheta,
                                  float* dY_out, cudaStream_t stream);

/* bitlogic_lut_backward_through with the layer input as byte rows (binary
 * wires, each byte 0 or 1, e.g. from bitlogic_encode_thermometer_u8; a byte
 * is read by its lowest bit): X device uint8 [w_in][B]; every other argument
 * as above.  On binary wires the corner weights are one-hot (§2), so each
 * sample adds its gradient to the one table entry its input bits select, in
 * the sample order of the fp32 form: the result equals the fp32-row call on
 * the same wires bit for bit. */
int bitlogic_lut_backward_through_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                     const float* theta, int32_t w, int32_t k, int32_t node,
                                     const float* Y, const int32_t* up_conn, const float* up_theta,
                                     int32_t up_w, int32_t up_k, const float* up_dY, int32_t up_group,
                                     const int32_t* up_off, const int32_t* up_edge, float* dtheta,
                                     float* dY_out, cudaStream_t stream);

/* Table gradient (no input gradient) of a layer whose input is byte rows
 * (binary wires, each byte 0 or 1; a byte is read by its lowest bit):
 * gathering bytes moves a quarter of the data of fp32 rows, and on binary
 * wires the corner weights are one-hot (§2), so each sample adds its
 * gradient to the one table entry its input bits select instead of 2^k
 * multiply-adds.  The output gradient comes from exactly one of
 *   dY rows:  node j reads row j / dy_group of dY ([w / dy_group][B]);
 *   up terms: the next layer's per-edge terms up_terms [up_edges][B] summed
 *             over p in [up_off[j], up_off[j+1]) in increasing p (row
 *             up_edge[p], or p when up_edge is NULL): the same sum, bit for
 *             bit, as bitlogic_csr_reduce.
 *   X         device uint8 [w_in][B];  conn, theta, dtheta, node as in
 *             bitlogic_lut_backward_node;  dY_out device fp32 [w][B] or NULL
 *             (the gradient used).
 * The result equals bitlogic_lut_backward_node without edge terms on the
 * same wires as fp32 rows, bit for bit.  Needs B % 4 == 0 and 16-byte
 * aligned X, the source and dY_out (BITLOGIC_ERR_ALIGN otherwise); B = 0
 * zeroes dtheta.  Out-of-range indices raise the device flag and read as
 * zero.  Returns BITLOGIC_ERR_NULL (no source or two), BITLOGIC_ERR_SHAPE,
 * BITLOGIC_ERR_FANIN, BITLOGIC_ERR_NODE, BITLOGIC_ERR_CUDA. */
int bitlogic_lut_backward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                             const float* theta, int32_t w, int32_t k, int32_t node,
                             const float* dY, int32_t dy_group, const float* up_terms,
                             const int32_t* up_off, const int32_t* up_edge, int32_t up_edges,
                             float* dtheta, float* dY_out, cudaStream_t stream);

/* bitlogic_lut_backward_u8 on wire bit rows: X device uint32 [w_in][W]
 * (the layout of bitlogic_encode_thermometer_bitrows), 16-byte aligned.
 *   order  device int32 [w] or NULL: the order in which the kernel's warps
 *          take the nodes (a permutation of 0 .. w-1; bitlogic_degree_order
 *          over the CSR offsets puts the nodes with the most term rows
 *          first, which shortens the launch's tail); NULL takes them in
 *          index order.  With an order, up_off and up_edge are the CSR map
 *          in the order's sequence: the rows of node order[p] are the CSR
 *          positions up_off[p] .. up_off[p+1] - 1 (bitlogic_build_csr over
 *          the next layer's connectivity with node i renamed to its
 *          position in the order).  An entry outside [0, w) raises the
 *          device flag and is skipped; a repeated entry leaves another
 *          node's dtheta unwritten.  The order changes no result.
 * Every other argument, the result and the errors as
 * bitlogic_lut_backward_u8: the same wires give the same dtheta and dY_out
 * bit for bit (the samples are visited in the same order). */
int bitlogic_lut_backward_bitrows(const uint32_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                  const float* theta, int32_t w, int32_t k, int32_t node,
                                  const float* dY, int32_t dy_group, const float* up_terms,
                                  const int32_t* up_off, const int32_t* up_edge, int32_t up_edges,
                                  const int32_t* order, float* dtheta, float* dY_out,
                                  cudaStream_t stream);

/* Learnable routing (§3, the paragraph on connectivity: a per-slot
 * candidate pool whose selection is differentiable in training and snapped
 * to a sparse mapping at discretization; App. A "Initialization": pools
 * drawn uniformly, logits zero).  Slot e = j*k + i of
 * a layer of w nodes (slots = w*k) has candidates cand[e][m] and logits
 * r[e][m], m < Kc, 1 <= Kc <= 32:
 *   p_e = softmax(r_e),   Xr[e][s] = sum_m p_e[m] X[cand[e][m]][s].
 * The rows Xr [slots][B] are the layer's slot inputs: the LUT calls read
 * them through the identity connectivity conn[j][i] = j*k + i, and the LUT
 * backward's per-edge terms over them are G = dL/dXr.
 *   X     device fp32 [w_in][B];   cand device int32 [slots][Kc] in [0, w_in)
 *   r     device fp32 [slots][Kc]
 *   Xr    device fp32 [slots][B], overwritten (may be NULL when B == 0)
 *   prob  device fp32 [slots][Kc] or NULL: receives p
 * bitlogic_route_backward, with G device fp32 [slots][B]:
 *   dr[e][m] = p_e[m] (A_m - sum_m' p_e[m'] A_m'),  A_m = sum_s G[e][s] X[cand[e][m]][s]
 *   (device fp32 [slots][Kc], overwritten; batch sums in a fixed order), and
 *   when dX is not NULL
 *   dX[c][s] = sum of prob[id] G[id / Kc][s] over the CSR positions of input
 *   c in increasing order (csr_off/csr_edge from bitlogic_build_csr over cand
 *   as a [slots][Kc] connectivity, so id = e*Kc + m; prob as written by
 *   bitlogic_route_forward), device fp32 [w_in][B], overwritten.
 * bitlogic_route_snap: conn[e] = cand[e][argmax_m r[e][m]] (first maximum),
 *   device int32 [slots]: the fixed connectivity of the discretized layer.
 * A candidate index outside [0, w_in) is read as 0 and raises the device flag. */
int bitlogic_route_forward(const float* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r,
                           int32_t slots, int32_t Kc, float* Xr, float* prob, cudaStream_t stream);
int bitlogic_route_backward(const float* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r,
                            int32_t slots, int32_t Kc, const float* G, float* dr, const float* prob,
                            const int32_t* csr_off, const int32_t* csr_edge, float* dX,
                            cudaStream_t stream);
int bitlogic_route_snap(const int32_t* cand, const float* r, int32_t slots, int32_t Kc, int32_t* conn,
                        cudaStream_t stream);

/* Routing over a layer input held as bytes (X device uint8 [w_in][B], the
 * values as numbers, e.g. the 0/1 wires of bitlogic_encode_thermometer_u8):
 * the same Xr, prob and dr as the fp32 calls on the same values (bit for
 * bit); no input gradient (a byte input is not trained). */
int bitlogic_route_forward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r,
                              int32_t slots, int32_t Kc, float* Xr, float* prob, cudaStream_t stream);
int bitlogic_route_backward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r,
                               int32_t slots, int32_t Kc, const float* G, float* dr, cudaStream_t stream);

/* Bytes of workspace bitlogic_head_loss needs. */
size_t bitlogic_head_loss_workspace(int64_t B, int32_t C);

/* Group-sum head with temperature and softmax cross-entropy (§3 "Encoders
 * and heads": popcount GroupSum; §4 "Training": cross-entropy on the raw
 * head logits).  Class c owns the contiguous nodes [c*g, (c+1)*g), g = w/C:
 *   logits[s][c] = (sum_{j in group c} Y[j][s]) / tau
 *   loss         = mean_s ( logsumexp(logits[s]) - logits[s][labels[s]] )
 *   dY[j][s]     = (softmax(logits[s])[c(j)] - [c(j) == labels[s]]) / (B tau)
 *   Y      device fp32 [w][B];  labels device int32 [B], values in [0, C)
 *   logits device fp32 [B][C] or NULL;  loss device fp32 [1]
 *   dY     device fp32 [w][B] or NULL
 *   workspace device, 16-byte aligned, >= bitlogic_head_loss_workspace()
 * Requires B >= 1, C >= 1, w % C == 0, tau > 0. */
int bitlogic_head_loss(const float* Y, int32_t w, int64_t B, int32_t C, float tau,
                       const int32_t* labels, float* logits, float* loss, float* dY,
                       void* workspace, size_t ws_bytes, cudaStream_t stream);

/* bitlogic_head_loss with one more optional output: dY_grouped, device fp32
 * [C][B], row c = the gradient shared by every node of class c
 * (dY_grouped[c][s] == dY[j][s] for every j in group c).  Either or both of
 * dY and dY_grouped may be requested. */
int bitlogic_head_loss_ex(const float* Y, int32_t w, int64_t B, int32_t C, float tau,
                          const int32_t* labels, float* logits, float* loss, float* dY,
                          float* dY_grouped, void* workspace, size_t ws_bytes,
                          cudaStream_t stream);

/* bitlogic_head_loss without a workspace argument, for callers that cannot
 * allocate device memory: code hosted inside another runtime that owns the
 * device allocator, or loops with a fixed memory budget where cudaMalloc /
 * cudaFree (which may synchronize the device or fail) are not allowed.  The
 * paper has no counterpart; this is a convenience of the library.
 *   Same arguments and results as bitlogic_head_loss; the caller still
 *   passes every input and output.
 *   Scratch: a fixed 8 MiB device array inside the library, reserved on
 *   every GPU that loads it until the process exits.  The call requires
 *   bitlogic_head_loss_workspace(B, C) <= 8 MiB (about B * C <= 340K) and
 *   returns BITLOGIC_ERR_TOO_LARGE otherwise, launching nothing.
 *   The first call on a device looks up the array's device address (a
 *   runtime query, not an allocation); make that first call before any
 *   stream capture.  All calls share the array: calls that overlap on the
 *   GPU (on different streams, or from different threads) race.  The array
 *   keeps the last call's contents; nothing in it needs to start at zero. */
int bitlogic_head_loss_noalloc(const float* Y, int32_t w, int64_t B, int32_t C, float tau,
                               const int32_t* labels, float* logits, float* loss, float* dY,
                               cudaStream_t stream);

/* One AdamW step on the table logits (§4 "Training": AdamW with beta1 0.9,
 * beta2 0.999, eps 1e-8, constant learning rate 0.01, weight decay 0),
 * weight decay decoupled, step number `step` >= 1, for every parameter i:
 *   m_i     = beta1 m_i + (1 - beta1) g_i
 *   v_i     = beta2 v_i + (1 - beta2) g_i^2
 *   theta_i = theta_i - lr ( (m_i / (1 - beta1^step))
 *                            / (sqrt(v_i / (1 - beta2^step)) + eps) + wd theta_i )
 *   theta, m, v  device fp32 [n], updated in place (m, v start at zero)
 *   grad         device fp32 [n] (e.g. the dtheta of bitlogic_lut_backward)
 * Returns BITLOGIC_ERR_HYPER unless 0 <= beta1, beta2 < 1, eps > 0, lr >= 0
 * and wd >= 0. */
int bitlogic_adamw_update(float* theta, float* m, float* v, const float* grad, int64_t n,
                          int64_t step, float lr, float beta1, float beta2, float eps,
                          float weight_decay, cudaStream_t stream);

/* Table discretization (§3: every surrogate discretizes to a 2^n-entry
 * truth table; App. C.1 extracts it once per layer): bit a of table[j] is 1
 * exactly when theta[j][a] > 0 (sigmoid > 1/2); bits >= 2^k are 0.
 *   theta device fp32 [w][2^k];  table device uint64 [w] */
int bitlogic_binarize_tables(const float* theta, int32_t w, int32_t k,
                             uint64_t* table, cudaStream_t stream);

/* Encoder fused with bit packing for the hard path (App. C.1 "Bit-packed
 * inference": samples packed along the batch into words; here 32 samples
 * per uint32): bit s%32 of xp[(j*b+i)*W + s/32] = (x[s][j] > thr[i]).
 *   x device uint8 [N][d];  thr_host host uint8 [b], 1 <= b <= 32
 *   xp device uint32 [d*b][W], W = ceil(N/32); tail bits (s >= N) are 0.
 * N == 0 is a no-op. */
int bitlogic_pack_bits(const uint8_t* x, int64_t N, int32_t d,
                       const uint8_t* thr_host, int32_t b,
                       uint32_t* xp, cudaStream_t stream);

/* Hard LUT layer on packed bits (App. C.1: each layer's LUT evaluation
 * becomes a bitwise operation on packed tensors): per node j and word,
 * the k input words select table bits by a bit-sliced Shannon mux tree, so
 * bit s of yp[j] = bit a_s of table[j] with a_s = sum_i bit_s(xp[conn[j][i]]) << i.
 * With C > 0 the popcount GroupSum head is fused: counts[s][c] = number of
 * ones among the nodes of group c (contiguous, g = w/C) for sample s, and
 * pred[s] = the first class with the largest count.
 *   xp    device uint32 [w_in][W];  conn device int32 [w][k]
 *   table device uint64 [w]
 *   yp    device uint32 [w][W], or NULL when C > 0 (then not written);
 *         tail bits (s >= N) are written as 0
 *   C     0 (no head) or the number of classes (w % C == 0)
 *   counts device int32 [N][C] (required when C > 0); pred device int32 [N]
 *         or NULL
 * N == 0 is a no-op. */
int bitlogic_hard_forward(const uint32_t* xp, int32_t w_in, int64_t N,
                          const int32_t* conn, const uint64_t* table,
                          int32_t w, int32_t k, uint32_t* yp,
                          int32_t C, int32_t* counts, int32_t* pred,
                          cudaStream_t stream);

/* Inverse connectivity (host): for each input i, the edges e = j*k + slot
 * with conn[j][slot] == i, in increasing e.  off_host [w_in+1],
 * edge_host [w*k].  Returns BITLOGIC_ERR_INDEX when an index is outside
 * [0, w_in).  Not part of the per-step path: built once per connectivity. */
int bitlogic_build_csr(const int32_t* conn_host, int32_t w, int32_t k, int32_t w_in,
                       int32_t* off_host, int32_t* edge_host);

/* Host: the CSR position of every edge, the inverse permutation of
 * edge_host: pos_host[edge_host[p]] = p for p < n_edges.  Returns
 * BITLOGIC_ERR_INDEX unless edge_host is a permutation of [0, n_edges). */
int bitlogic_csr_positions(const int32_t* edge_host, int32_t n_edges, int32_t* pos_host);

/* Host: the nodes 0 .. n-1 by decreasing CSR degree off_host[i+1] -
 * off_host[i] (ties in increasing i), the order in which
 * bitlogic_lut_backward_bitrows can take the nodes of a layer whose output
 * gradient it sums from the next layer's terms, so that the nodes with the
 * most term rows start first and the launch ends on short ones.
 * off_host [n+1] (off_host[0] == 0, non-decreasing: BITLOGIC_ERR_INDEX
 * otherwise), order_host [n]. */
int bitlogic_degree_order(const int32_t* off_host, int32_t n, int32_t* order_host);

/* Synchronizes `stream`, then reports (and clears) the device-side index
 * flag: BITLOGIC_OK, or BITLOGIC_ERR_DEVICE when a kernel met an index out of
 * range since the last call, or BITLOGIC_ERR_CUDA. */
int bitlogic_device_error(cudaStream_t stream);

/* Issue-throughput probe (measurement support, not part of the method): the
 * roofline of the hard layer counts its mux operations against the rate at
 * which this GPU issues the instructions the mux tree is made of; this launch
 * measures those rates.  One block of 1024 threads per SM
 * (bitlogic_issue_probe_blocks() blocks, bitlogic_issue_probe_threads()
 * threads) runs `iters` x bitlogic_issue_probe_ops_per_iter() instructions
 * of one kind per thread, in independent dependency chains.  Kinds: LOP3, a
 * mux with one loop-invariant operand; IMAD; FFMA (FP32 reference); MUX3, a
 * LOP3 mux of three varying registers (the tree's upper levels); MIX, IMAD
 * and MUX3 interleaved one to one (the tree's mix).
 *   sink:   device, >= bitlogic_issue_probe_threads() uint32 (one per
 *           thread, written so the work is kept);
 *   cycles: device, >= bitlogic_issue_probe_blocks() int64 or NULL: the SM
 *           clock cycles each block ran (clock64), so that
 *           threads per block x iters x ops per iter / cycles is the rate per
 *           SM and clock.
 * Returns BITLOGIC_ERR_NULL, BITLOGIC_ERR_SHAPE (iters outside [0, 2^20],
 * sink too short, unknown kind) or BITLOGIC_ERR_CUDA. */
typedef enum {
    BITLOGIC_PROBE_LOP3 = 0,
    BITLOGIC_PROBE_IMAD = 1,
    BITLOGIC_PROBE_FFMA = 2,
    BITLOGIC_PROBE_MUX3 = 3,
    BITLOGIC_PROBE_MIX = 4
} bitlogic_probe_t;
int64_t bitlogic_issue_probe_blocks(void);
int64_t bitlogic_issue_probe_threads(void);
int64_t bitlogic_issue_probe_ops_per_iter(void);
int bitlogic_issue_probe(int32_t kind, int64_t iters, uint32_t seed, uint32_t* sink,
                         int64_t sink_len, int64_t* cycles, cudaStream_t stream);

/* Static text for a status code. */
const char* bitlogic_status_string(int code);

/* ABI version (major*100 + minor). */
int bitlogic_version(void);

#ifdef __cplusplus
}
#endif

#endif /* BITLOGIC_H */
