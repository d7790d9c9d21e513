/*
 * oracle.c -- plain, slow, single-threaded CPU oracle for the doubly
 * pipelined, dual-root reduction-to-all (Traff, arXiv 2109.12626).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, includes
 * or calls this file; only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg load it.  It shares no code, header, table or helper with
 * the CUDA path.
 *
 * What it computes, each part citing the passage it follows:
 *   O1  orc_trees        dual post-order trees (Sec. 1.1, first paragraph and
 *                        the description of the subtree intervals)
 *   O2  orc_tree_fold    y by the post-order bracketing of Sec. 1.1 and the
 *                        dual-root rule of Algorithm 1
 *   O3  orc_left_fold    the plain definition y = x_0 (.) x_1 (.) ... (.) x_{p-1}
 *                        (problem statement, Sec. 1)
 *   O4  orc_simulate     event-level simulation of Algorithm 1: explicit
 *                        per-processor lists of bidirectional exchanges,
 *                        paired by a rendezvous matcher, unit-step clock
 *   O5  orc_simulate_rb  event-level simulation of the alternative that
 *                        Sec. 1.2 analyses and Sec. 2 measures (item 3,
 *                        "User-Allreduce1"): a pipelined reduction to the
 *                        root of one binary tree, then a pipelined
 *                        broadcast from it, the same b blocks in both
 *
 * Element types: int32 sum (wrapping two's complement, computed as uint32),
 * float32 sum (IEEE round-to-nearest-even, no contraction), 2x2 uint32 matrix
 * product mod 2^32 (row-major a b / c d, lower rank on the left), 2x2
 * float32 matrix product (each entry two rounded products and a rounded
 * sum: non-commutative and, in rounding, non-associative), and an
 * oracle-only "interval witness" whose elements are rank intervals [lo,hi]:
 * [a,b] (.) [b+1,c] = [a,c], every other pair gives the absorbing value
 * bottom = (-1,-1).  The witness is associative and non-commutative and fails
 * on any misordered, dropped or repeated operand.
 *
 * Readings of the paper this file takes:
 *   - d_i is the DEPTH of processor i (the correctness argument of Sec. 1.1
 *     uses depth; the caption of Algorithm 1 says height).
 *   - tree 0 = ranks [0, floor(p/2)), tree 1 = [floor(p/2), p), both
 *     complete binary trees (all levels full but the last, which fills from
 *     the left), numbered in post-order.
 *   - a node with one child has child_0 = i-1 and no child_1.
 *   - an exchange whose send block and receive block are both outside
 *     [0,b) is void and is skipped (the zero-size blocks of Sec. 1.3).
 *   - block j covers [j*(m/b) + min(j, m%b), ...): the first m%b blocks hold
 *     one element more.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { ORC_I32 = 0, ORC_F32 = 1, ORC_MAT = 2, ORC_WIT = 3, ORC_MATF = 4 };

enum {
    ORC_OK = 0,
    ORC_EINVAL = 1,
    ORC_ENOMEM = 2,
    ORC_EMISMATCH = 3, /* two partners met with disagreeing block indices */
    ORC_EDEADLOCK = 4  /* no pair of processors can make progress       */
};

/* Planted mistakes, used only by the tests that show the pins catch them.
 * 0 = none. 1 = swap the operands of the child_0 combine in the tree fold.
 * 2 = drop the child_1 term in the tree fold. 3 = use node height instead of
 * depth for d_i in the simulation. 4 = both roots apply t (.) Y in the
 * simulation (ignores the non-commutative rule of Algorithm 1).
 * 5 = in the reduce-then-broadcast simulation the root starts broadcasting
 * each block as soon as child_0's part of it has arrived, before child_1's
 * part and before its reduction phase has ended. */
static int g_mutation = 0;
void orc_set_mutation(int k) { g_mutation = k; }

static size_t esize(int dt)
{
    switch (dt) {
    case ORC_I32: return 4;
    case ORC_F32: return 4;
    case ORC_MAT: return 16;
    case ORC_WIT: return 8;
    case ORC_MATF: return 16;
    default: return 0;
    }
}

/* out = a (.) b for one element.  out may alias a or b. */
static void op1(int dt, const void* a, const void* b, void* out)
{
    switch (dt) {
    case ORC_I32: {
        uint32_t u, v;
        memcpy(&u, a, 4);
        memcpy(&v, b, 4);
        u = u + v; /* wraps mod 2^32 */
        memcpy(out, &u, 4);
        break;
    }
    case ORC_F32: {
        float u, v;
        memcpy(&u, a, 4);
        memcpy(&v, b, 4);
        volatile float s = u + v; /* one IEEE single add, nothing fused */
        float r = s;
        memcpy(out, &r, 4);
        break;
    }
    case ORC_MAT: {
        uint32_t A[4], B[4], C[4];
        memcpy(A, a, 16);
        memcpy(B, b, 16);
        /* [A0 A1; A2 A3] * [B0 B1; B2 B3] mod 2^32 */
        C[0] = A[0] * B[0] + A[1] * B[2];
        C[1] = A[0] * B[1] + A[1] * B[3];
        C[2] = A[2] * B[0] + A[3] * B[2];
        C[3] = A[2] * B[1] + A[3] * B[3];
        memcpy(out, C, 16);
        break;
    }
    case ORC_MATF: {
        /* [A0 A1; A2 A3] * [B0 B1; B2 B3] in float32: each entry is two
         * rounded products and one rounded sum, nothing fused */
        float A[4], B[4], C[4];
        memcpy(A, a, 16);
        memcpy(B, b, 16);
        for (int r = 0; r < 2; r++)
            for (int c = 0; c < 2; c++) {
                volatile float u = A[2 * r] * B[c];
                volatile float v = A[2 * r + 1] * B[2 + c];
                volatile float w = u + v;
                C[2 * r + c] = w;
            }
        memcpy(out, C, 16);
        break;
    }
    case ORC_WIT: {
        int32_t A[2], B[2], C[2];
        memcpy(A, a, 8);
        memcpy(B, b, 8);
        if (A[0] >= 0 && B[0] >= 0 && A[1] + 1 == B[0]) {
            C[0] = A[0];
            C[1] = B[1];
        } else {
            C[0] = -1;
            C[1] = -1;
        }
        memcpy(out, C, 8);
        break;
    }
    }
}

/* out[e] = a[e] (.) b[e] for e < n. */
static void opv(int dt, const char* a, const char* b, char* out, int64_t n)
{
    size_t s = esize(dt);
    for (int64_t e = 0; e < n; e++)
        op1(dt, a + e * s, b + e * s, out + e * s);
}

/* ------------------------------------------------------------------ O1 ---
 * Dual post-order trees (Sec. 1.1).  Each tree of n nodes is a complete
 * binary tree built by heap indexing (node k has children 2k and 2k+1,
 * k = 1..n) and then numbered in post-order: left subtree, right subtree,
 * node.  The left subtree therefore holds the lower ranks [i', i''] and its
 * root is child_1 = i''; the right subtree [i''+1, i-1] has root
 * child_0 = i-1, as the paper fixes.  With only a left child, that child is
 * i-1 and is child_0.  d_i = depth (root 0).  Roots: r0 = floor(p/2)-1 and
 * r1 = p-1, duals of each other.  p = 1 gives one root with no dual. */

typedef struct {
    int n;
    int* post; /* post[k] = post-order index of heap node k (1-based) */
    int next;
} heapwalk;

static void postorder(heapwalk* w, int k)
{
    if (k > w->n) return;
    postorder(w, 2 * k);
    postorder(w, 2 * k + 1);
    w->post[k] = w->next++;
}

static int build_tree(int lo, int n, int* parent, int* child0, int* child1,
                      int* depth)
{
    if (n <= 0) return ORC_OK;
    heapwalk w;
    w.n = n;
    w.next = 0;
    w.post = (int*)malloc(sizeof(int) * (size_t)(n + 1));
    if (!w.post) return ORC_ENOMEM;
    postorder(&w, 1);
    for (int k = 1; k <= n; k++) {
        int i = lo + w.post[k];
        int d = 0;
        for (int t = k; t > 1; t >>= 1) d++;
        depth[i] = d;
        parent[i] = (k == 1) ? -1 : lo + w.post[k / 2];
        int l = 2 * k, r = 2 * k + 1;
        if (l <= n && r <= n) {
            child0[i] = lo + w.post[r];
            child1[i] = lo + w.post[l];
        } else if (l <= n) {
            child0[i] = lo + w.post[l];
            child1[i] = -1;
        } else {
            child0[i] = -1;
            child1[i] = -1;
        }
    }
    free(w.post);
    return ORC_OK;
}

/* topo 0: the dual trees of Sec. 1.1.  topo 1: one complete post-order tree
 * over all p ranks, root p-1, no dual (the single doubly pipelined tree
 * discussed in Sec. 1.2). */
int orc_trees_topo(int p, int topo, int* parent, int* child0, int* child1,
                   int* dual, int* depth)
{
    if (p < 1 || topo < 0 || topo > 1) return ORC_EINVAL;
    if (topo == 1) {
        int rc = build_tree(0, p, parent, child0, child1, depth);
        for (int i = 0; i < p; i++) dual[i] = -1;
        return rc;
    }
    int n0 = p / 2, n1 = p - n0;
    int rc = build_tree(0, n0, parent, child0, child1, depth);
    if (rc) return rc;
    rc = build_tree(n0, n1, parent, child0, child1, depth);
    if (rc) return rc;
    for (int i = 0; i < p; i++) dual[i] = -1;
    if (n0 > 0) {
        dual[n0 - 1] = p - 1;
        dual[p - 1] = n0 - 1;
    }
    return ORC_OK;
}

int orc_trees(int p, int* parent, int* child0, int* child1, int* dual,
              int* depth)
{
    return orc_trees_topo(p, 0, parent, child0, child1, dual, depth);
}

/* ------------------------------------------------------------------ O3 ---
 * The plain definition of the result (Sec. 1): y = x_0 (.) x_1 (.) ... (.)
 * x_{p-1}, folded left to right.  x is row-major [p][m], y is [m]. */
int orc_left_fold(int p, int64_t m, int dt, const void* x, void* y)
{
    size_t s = esize(dt);
    if (p < 1 || m < 0 || s == 0) return ORC_EINVAL;
    const char* X = (const char*)x;
    memcpy(y, X, (size_t)m * s);
    for (int i = 1; i < p; i++)
        opv(dt, (const char*)y, X + (size_t)i * (size_t)m * s, (char*)y, m);
    return ORC_OK;
}

/* Float32 inputs folded left to right in double, with sum_i |x_i| per
 * element: context for a re-bracketed float32 error bound. */
int orc_left_fold_f64(int p, int64_t m, const float* x, double* y,
                      double* abs_sum)
{
    if (p < 1 || m < 0) return ORC_EINVAL;
    for (int64_t e = 0; e < m; e++) {
        double acc = 0.0, a = 0.0;
        for (int i = 0; i < p; i++) {
            double v = (double)x[(size_t)i * (size_t)m + (size_t)e];
            acc += v;
            a += v < 0 ? -v : v;
        }
        y[e] = acc;
        if (abs_sum) abs_sum[e] = a;
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------ O2 ---
 * The bracketing the method produces (Sec. 1.1): the node value of processor
 * i is v(i) = v(child_1) (.) ( v(child_0) (.) x_i ), the lower subtree on the
 * left, and both roots end with v(r0) (.) v(r1) (Algorithm 1, dual-root step:
 * the lower-numbered root applies Y (.) t, the other t (.) Y).  Written as a
 * recursion over whole m-vectors. */
typedef struct {
    int p;
    int64_t m;
    int dt;
    size_t s;
    const char* X;
    const int* c0;
    const int* c1;
} foldctx;

static int subtree_value(const foldctx* f, int i, char* out)
{
    size_t bytes = (size_t)f->m * f->s;
    memcpy(out, f->X + (size_t)i * bytes, bytes);
    if (f->c0[i] >= 0 || f->c1[i] >= 0) {
        char* tmp = (char*)malloc(bytes ? bytes : 1);
        if (!tmp) return ORC_ENOMEM;
        if (f->c0[i] >= 0) {
            int rc = subtree_value(f, f->c0[i], tmp);
            if (rc) { free(tmp); return rc; }
            if (g_mutation == 1)
                opv(f->dt, out, tmp, out, f->m);      /* planted: swapped */
            else
                opv(f->dt, tmp, out, out, f->m);      /* v(c0) (.) x_i    */
        }
        if (f->c1[i] >= 0 && g_mutation != 2) {
            int rc = subtree_value(f, f->c1[i], tmp);
            if (rc) { free(tmp); return rc; }
            opv(f->dt, tmp, out, out, f->m);          /* v(c1) (.) (...)  */
        }
        free(tmp);
    }
    return ORC_OK;
}

/* One tree (topo 1): y = v(p-1). */
int orc_tree_fold_topo(int p, int topo, int64_t m, int dt, const void* x,
                       void* y)
{
    size_t s = esize(dt);
    if (p < 1 || m < 0 || s == 0) return ORC_EINVAL;
    int* T = (int*)malloc(sizeof(int) * 5 * (size_t)p);
    if (!T) return ORC_ENOMEM;
    int *par = T, *c0 = T + p, *c1 = T + 2 * p, *du = T + 3 * p,
        *dep = T + 4 * p;
    int rc = orc_trees_topo(p, topo, par, c0, c1, du, dep);
    if (rc) { free(T); return rc; }
    foldctx f = {p, m, dt, s, (const char*)x, c0, c1};
    int n0 = topo == 1 ? 0 : p / 2;
    if (n0 == 0) {
        rc = subtree_value(&f, p - 1, (char*)y); /* one root: y = v(p-1) */
    } else {
        size_t bytes = (size_t)m * s;
        char* v1 = (char*)malloc(bytes ? bytes : 1);
        if (!v1) { free(T); return ORC_ENOMEM; }
        rc = subtree_value(&f, n0 - 1, (char*)y);
        if (!rc) rc = subtree_value(&f, p - 1, v1);
        if (!rc) opv(dt, (const char*)y, v1, (char*)y, m); /* v(r0) (.) v(r1) */
        free(v1);
    }
    free(T);
    return rc;
}

int orc_tree_fold(int p, int64_t m, int dt, const void* x, void* y)
{
    return orc_tree_fold_topo(p, 0, m, dt, x, y);
}

/* The full reduction-to-all contract on the CPU: the tree fold, then the
 * result copied to each of the p output rows (y is row-major [p][m]). */
int orc_allreduce(int p, int64_t m, int dt, const void* x, void* y)
{
    size_t s = esize(dt);
    if (p < 1 || m < 0 || s == 0) return ORC_EINVAL;
    size_t bytes = (size_t)m * s;
    char* Y = (char*)y;
    int rc = orc_tree_fold(p, m, dt, x, Y);
    if (rc) return rc;
    for (int i = 1; i < p; i++) memcpy(Y + (size_t)i * bytes, Y, bytes);
    return ORC_OK;
}

/* ------------------------------------------------------------------ O4 ---
 * Event-level simulation of Algorithm 1.  Every processor i gets the explicit
 * list of bidirectional exchanges it performs in rounds j = 0..b+d_i, in the
 * order of the algorithm: child_0, child_1, then dual (roots) or parent.
 *   child_k : send Y[j-(d_i+1)], receive t = the child's Y[j], Y[j] = t (.) Y[j]
 *   dual    : send Y[j], receive t = the dual's Y[j];
 *             lower root Y[j] = Y[j] (.) t, higher root Y[j] = t (.) Y[j]
 *   parent  : send Y[j], receive Y[j-d_i] (overwrites the own block)
 * Blocks outside [0,b) have zero elements; an exchange that is empty in both
 * directions is void and skipped.  A rendezvous matcher repeatedly looks for
 * two processors whose next exchanges name each other, checks that each
 * one's send index is the other's receive index, performs both transfers
 * from the blocks as they were before the exchange, and advances a unit-step
 * clock to max(clock_a, clock_b) + 1 for both.
 *
 * x is [p][m]; y ([p][m]) receives every processor's final Y.
 * stats[0] total steps (largest clock)
 * stats[1] step at which the last processor holds final block 0
 * stats[2] number of exchanges performed
 * stats[3] largest number of (.) applications by a non-root in one round
 * stats[4] largest number of (.) applications by a root in one round
 * stats[5] number of void exchanges skipped
 * last_round[i] = round of processor i's last non-void exchange (-1: none).
 */
typedef struct {
    int partner;
    int kind; /* 0 child_0, 1 child_1, 2 parent, 3 dual */
    int send_blk;
    int recv_blk;
    int round;
} xop;

static int64_t blk_start(int64_t m, int b, int j)
{
    int64_t q = m / b, r = m % b;
    return (int64_t)j * q + (j < r ? j : r);
}

static int valid_blk(int b, int j) { return j >= 0 && j < b; }

int orc_simulate_topo(int p, int topo, int64_t m, int b, int dt,
                      const void* x, void* y, int64_t* stats, int* last_round)
{
    size_t s = esize(dt);
    if (p < 1 || m < 1 || b < 1 || b > m || s == 0) return ORC_EINVAL;
    int rc = ORC_OK;
    size_t bytes = (size_t)m * s;
    int* T = (int*)malloc(sizeof(int) * 6 * (size_t)p);
    if (!T) return ORC_ENOMEM;
    int *par = T, *c0 = T + p, *c1 = T + 2 * p, *du = T + 3 * p,
        *dep = T + 4 * p, *hgt = T + 5 * p;
    rc = orc_trees_topo(p, topo, par, c0, c1, du, dep);
    if (rc) { free(T); return rc; }
    /* node height, only for the planted mistake that confuses it with depth */
    for (int i = 0; i < p; i++) {
        int hl = (c1[i] >= 0) ? hgt[c1[i]] + 1 : 0;
        int hr = (c0[i] >= 0) ? hgt[c0[i]] + 1 : 0;
        hgt[i] = hl > hr ? hl : hr; /* children have lower ranks */
    }

    xop** L = (xop**)calloc((size_t)p, sizeof(xop*));
    int64_t* nops = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* cur = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* clk = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* arr0 = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    char* Y = (char*)y;
    char* sa = (char*)malloc(bytes / (size_t)b * 2 + 2 * s + 16);
    char* sb = (char*)malloc(bytes / (size_t)b * 2 + 2 * s + 16);
    int* ops_round = (int*)calloc((size_t)p, sizeof(int));
    int* ops_round_id = (int*)malloc(sizeof(int) * (size_t)p);
    if (!L || !nops || !cur || !clk || !arr0 || !sa || !sb ||
        !ops_round || !ops_round_id) { rc = ORC_ENOMEM; goto done; }
    memcpy(Y, x, bytes * (size_t)p); /* Y <- x_i */
    int64_t skipped = 0;

    for (int i = 0; i < p; i++) {
        int d = (g_mutation == 3) ? hgt[i] : dep[i];
        int64_t cap = 3 * ((int64_t)b + d + 1);
        L[i] = (xop*)malloc(sizeof(xop) * (size_t)cap);
        if (!L[i]) { rc = ORC_ENOMEM; goto done; }
        int64_t k = 0;
        for (int j = 0; j <= b + d; j++) {
            int ch[2] = {c0[i], c1[i]};
            for (int q = 0; q < 2; q++) {
                if (ch[q] < 0) continue;
                xop o = {ch[q], q, j - (d + 1), j, j};
                if (!valid_blk(b, o.send_blk)) o.send_blk = -1;
                if (!valid_blk(b, o.recv_blk)) o.recv_blk = -1;
                if (o.send_blk < 0 && o.recv_blk < 0) { skipped++; continue; }
                L[i][k++] = o;
            }
            if (du[i] >= 0) {
                xop o = {du[i], 3, j, j, j};
                if (!valid_blk(b, j)) { skipped++; continue; }
                L[i][k++] = o;
            } else if (par[i] >= 0) {
                xop o = {par[i], 2, j, j - d, j};
                if (!valid_blk(b, o.send_blk)) o.send_blk = -1;
                if (!valid_blk(b, o.recv_blk)) o.recv_blk = -1;
                if (o.send_blk < 0 && o.recv_blk < 0) { skipped++; continue; }
                L[i][k++] = o;
            }
        }
        nops[i] = k;
        last_round[i] = k ? L[i][k - 1].round : -1;
        arr0[i] = -1;
        ops_round_id[i] = -1;
    }
    /* a root without a dual holds final block 0 once round 0's child
     * exchanges are done; with no children at all, from the start */
    for (int i = 0; i < p; i++)
        if (par[i] < 0 && du[i] < 0 && c0[i] < 0) arr0[i] = 0;

    int64_t done_ops = 0, total_ops = 0, nex = 0;
    int64_t max_nonroot = 0, max_root = 0;
    for (int i = 0; i < p; i++) total_ops += nops[i];
    while (done_ops < total_ops) {
        int progress = 0;
        for (int a = 0; a < p; a++) {
            if (cur[a] >= nops[a]) continue;
            xop* oa = &L[a][cur[a]];
            int bb = oa->partner;
            if (bb < a) continue; /* each pair is looked at from its lower end */
            if (cur[bb] >= nops[bb]) continue;
            xop* ob = &L[bb][cur[bb]];
            if (ob->partner != a) continue;
            if (oa->send_blk != ob->recv_blk || oa->recv_blk != ob->send_blk) {
                rc = ORC_EMISMATCH;
                goto done;
            }
            /* snapshot both outgoing blocks, then apply both receives */
            int64_t la = 0, lb = 0;
            if (oa->send_blk >= 0) {
                int64_t s0 = blk_start(m, b, oa->send_blk);
                la = blk_start(m, b, oa->send_blk + 1) - s0;
                memcpy(sa, Y + (size_t)a * bytes + (size_t)s0 * s, (size_t)la * s);
            }
            if (ob->send_blk >= 0) {
                int64_t s0 = blk_start(m, b, ob->send_blk);
                lb = blk_start(m, b, ob->send_blk + 1) - s0;
                memcpy(sb, Y + (size_t)bb * bytes + (size_t)s0 * s, (size_t)lb * s);
            }
            int64_t step = (clk[a] > clk[bb] ? clk[a] : clk[bb]) + 1;
            clk[a] = clk[bb] = step;
            for (int side = 0; side < 2; side++) {
                int me = side ? bb : a;
                int other = side ? a : bb;
                xop* o = side ? ob : oa;
                const char* t = side ? sa : sb;
                if (o->recv_blk < 0) continue;
                int64_t s0 = blk_start(m, b, o->recv_blk);
                int64_t len = blk_start(m, b, o->recv_blk + 1) - s0;
                char* Yb = Y + (size_t)me * bytes + (size_t)s0 * s;
                if (o->kind == 2) {
                    memcpy(Yb, t, (size_t)len * s); /* final block from parent */
                    if (o->recv_blk == 0) arr0[me] = step;
                } else {
                    if (o->kind == 3 && me < other && g_mutation != 4)
                        opv(dt, Yb, t, Yb, len); /* lower root: Y (.) t */
                    else
                        opv(dt, t, Yb, Yb, len); /* t (.) Y              */
                    if (o->kind == 3 && o->recv_blk == 0) arr0[me] = step;
                    if (o->kind <= 1 && o->recv_blk == 0 && par[me] < 0 &&
                        du[me] < 0)
                        arr0[me] = step; /* lone root: block 0 final after its children */
                    if (ops_round_id[me] != o->round) {
                        ops_round_id[me] = o->round;
                        ops_round[me] = 0;
                    }
                    ops_round[me]++;
                    int64_t c = ops_round[me];
                    if (du[me] >= 0) { if (c > max_root) max_root = c; }
                    else if (c > max_nonroot) max_nonroot = c;
                }
            }
            cur[a]++;
            cur[bb]++;
            done_ops += 2;
            nex++;
            progress = 1;
        }
        if (!progress) { rc = ORC_EDEADLOCK; goto done; }
    }
    int64_t tot = 0, a0 = 0;
    for (int i = 0; i < p; i++) {
        if (clk[i] > tot) tot = clk[i];
        if (arr0[i] > a0) a0 = arr0[i];
    }
    stats[0] = tot;
    stats[1] = a0;
    stats[2] = nex;
    stats[3] = max_nonroot;
    stats[4] = max_root;
    stats[5] = skipped;

done:
    if (L) for (int i = 0; i < p; i++) free(L[i]);
    free(L); free(nops); free(cur); free(clk); free(arr0);
    free(sa); free(sb); free(ops_round); free(ops_round_id); free(T);
    return rc;
}

int orc_simulate(int p, int64_t m, int b, int dt, const void* x, void* y,
                 int64_t* stats, int* last_round)
{
    return orc_simulate_topo(p, 0, m, b, dt, x, y, stats, last_round);
}

/* ------------------------------------------------------------------ O5 ---
 * Pipelined reduce, then pipelined broadcast, on one binary tree (the
 * alternative of Sec. 1.2 whose cost is 2(2h + 2(b-1))(alpha + beta m/b),
 * and the "pipelined reduce followed by a pipelined broadcast with the same
 * pipeline block size using a single binary tree" of Sec. 2, item 3).  The
 * tree is the one-tree topology (topo 1): complete, post-order, root p-1.
 *
 * Communication model: every processor has one send port and one receive
 * port (it can send one block and receive another in the same step, as in
 * the bidirectional model of Sec. 1.2); a transfer of one block takes one
 * unit step on the sender's send port and the receiver's receive port.
 * Each port works through a fixed list of transfers in order:
 *   reduction phase, blocks j = 0..b-1:
 *     receive port: child_0's partial block j, then child_1's;
 *                   Y[j] = t (.) Y[j] for each, so Y[j] = v(c1) (.) (v(c0) (.) x_i)
 *     send port:    Y[j] to the parent, once both children's blocks j arrived
 *   broadcast phase, blocks j = 0..b-1:
 *     receive port: final block j from the parent, Y[j] = t
 *     send port:    Y[j] to child_0, then to child_1, once held
 * The two phases are two collective operations called one after the other:
 * a processor takes part in the broadcast only when all its reduction
 * transfers (on both ports) are done, and the root broadcasts only after it
 * has reduced all b blocks.  A transfer happens when the sender's next send
 * and the receiver's next receive name each other (with equal block index
 * and phase, else ORC_EMISMATCH), at step max(send port free, receive port
 * free, data ready) + 1.
 *
 * x is [p][m]; y ([p][m]) receives every processor's final Y.
 * stats[0] total steps (largest port clock)
 * stats[1] step at which the root holds all b reduced blocks
 * stats[2] number of transfers
 * stats[3] step at which the last processor holds final block 0
 * stats[4] largest number of (.) applications on one block at one processor
 * stats[5] step at which the root's first broadcast transfer starts
 */
typedef struct {
    int partner;
    int blk;
    int phase; /* 0 reduction, 1 broadcast */
} rbop;

int orc_simulate_rb(int p, int64_t m, int b, int dt, const void* x, void* y,
                    int64_t* stats)
{
    size_t s = esize(dt);
    if (p < 1 || m < 1 || b < 1 || b > m || s == 0) return ORC_EINVAL;
    int rc = ORC_OK;
    size_t bytes = (size_t)m * s;
    char* Y = (char*)y;
    int* T = (int*)malloc(sizeof(int) * 5 * (size_t)p);
    rbop** snd = (rbop**)calloc((size_t)p, sizeof(rbop*));
    rbop** rcv = (rbop**)calloc((size_t)p, sizeof(rbop*));
    int64_t* nsnd = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* nrcv = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* sp = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* rp = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* sfree = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* rfree = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    int64_t* red_left = (int64_t*)calloc((size_t)p, sizeof(int64_t)); /* reduction transfers to go */
    int64_t* red_end = (int64_t*)calloc((size_t)p, sizeof(int64_t));
    /* per processor and block: children's blocks still to come, the step at
     * which the block is reduced (-1: not yet), the step at which the final
     * block is held (-1: not yet) */
    int* left = (int*)malloc(sizeof(int) * (size_t)p * (size_t)b);
    int64_t* ready = (int64_t*)malloc(sizeof(int64_t) * (size_t)p * (size_t)b);
    int64_t* fin = (int64_t*)malloc(sizeof(int64_t) * (size_t)p * (size_t)b);
    char* early = (char*)malloc(bytes); /* planted mistake 5: the root's early copies */
    if (!T || !snd || !rcv || !nsnd || !nrcv || !sp || !rp || !sfree || !rfree ||
        !red_left || !red_end || !left || !ready || !fin || !early) {
        rc = ORC_ENOMEM;
        goto done;
    }
    int *par = T, *c0 = T + p, *c1 = T + 2 * p, *du = T + 3 * p, *dep = T + 4 * p;
    rc = orc_trees_topo(p, 1, par, c0, c1, du, dep);
    if (rc) goto done;
    memcpy(Y, x, bytes * (size_t)p); /* Y <- x_i */
    int root = p - 1;
    int64_t ntransfers = 0, max_ops = 0;
    for (int i = 0; i < p; i++) {
        int nch = (c0[i] >= 0) + (c1[i] >= 0);
        snd[i] = (rbop*)malloc(sizeof(rbop) * (size_t)b * 3);
        rcv[i] = (rbop*)malloc(sizeof(rbop) * (size_t)b * 3);
        if (!snd[i] || !rcv[i]) { rc = ORC_ENOMEM; goto done; }
        int64_t ks = 0, kr = 0;
        for (int j = 0; j < b; j++) { /* reduction */
            if (c0[i] >= 0) rcv[i][kr++] = (rbop){c0[i], j, 0};
            if (c1[i] >= 0) rcv[i][kr++] = (rbop){c1[i], j, 0};
            if (par[i] >= 0) snd[i][ks++] = (rbop){par[i], j, 0};
        }
        red_left[i] = ks + kr;
        for (int j = 0; j < b; j++) { /* broadcast */
            if (par[i] >= 0) rcv[i][kr++] = (rbop){par[i], j, 1};
            if (c0[i] >= 0) snd[i][ks++] = (rbop){c0[i], j, 1};
            if (c1[i] >= 0) snd[i][ks++] = (rbop){c1[i], j, 1};
        }
        nsnd[i] = ks;
        nrcv[i] = kr;
        ntransfers += ks;
        for (int j = 0; j < b; j++) {
            left[(size_t)i * b + j] = nch;
            ready[(size_t)i * b + j] = nch ? -1 : 0; /* a leaf's block is x_i */
            fin[(size_t)i * b + j] = -1;
        }
        if (nch > max_ops) max_ops = nch;
    }
    int64_t done_tr = 0, first_bcast = -1;
    while (done_tr < ntransfers) {
        int progress = 0;
        for (int a = 0; a < p; a++) {
            while (sp[a] < nsnd[a]) {
                rbop* o = &snd[a][sp[a]];
                int B = o->partner;
                if (rp[B] >= nrcv[B]) break;
                rbop* q = &rcv[B][rp[B]];
                if (q->partner != a) break; /* the receiver expects someone else first */
                if (q->blk != o->blk || q->phase != o->phase) { rc = ORC_EMISMATCH; goto done; }
                int j = o->blk;
                int64_t rdy;
                const char* src = Y + (size_t)a * bytes;
                if (o->phase == 0) {
                    rdy = ready[(size_t)a * b + j];
                    if (rdy < 0) break;
                } else {
                    /* both ends have finished their reduction transfers */
                    if (red_left[B] > 0) break;
                    if (a == root && g_mutation == 5) {
                        /* planted: broadcast once child_0's part has arrived */
                        rdy = fin[(size_t)a * b + j];
                        if (rdy < 0) break;
                        src = early;
                    } else {
                        if (red_left[a] > 0) break;
                        rdy = (a == root) ? ready[(size_t)a * b + j] : fin[(size_t)a * b + j];
                        if (rdy < 0) break;
                        if (red_end[a] > rdy) rdy = red_end[a];
                    }
                    if (red_end[B] > rdy) rdy = red_end[B];
                }
                int64_t t = sfree[a] > rfree[B] ? sfree[a] : rfree[B];
                if (rdy > t) t = rdy;
                t += 1;
                sfree[a] = rfree[B] = t;
                sp[a]++;
                rp[B]++;
                done_tr++;
                progress = 1;
                int64_t s0 = blk_start(m, b, j);
                int64_t len = blk_start(m, b, j + 1) - s0;
                char* dst = Y + (size_t)B * bytes + (size_t)s0 * s;
                const char* t_blk = src + (size_t)s0 * s;
                if (o->phase == 0) {
                    opv(dt, t_blk, dst, dst, len); /* Y[j] = t (.) Y[j] */
                    size_t k = (size_t)B * b + j;
                    if (--left[k] == 0) ready[k] = t;
                    /* planted mistake 5 keeps the root's block as it is
                     * after child_0's part */
                    if (g_mutation == 5 && B == root && a == c0[root]) {
                        memcpy(early + (size_t)s0 * s, dst, (size_t)len * s);
                        fin[k] = t;
                    }
                    if (--red_left[a] == 0) red_end[a] = t;
                    if (--red_left[B] == 0) red_end[B] = t;
                } else {
                    memcpy(dst, t_blk, (size_t)len * s); /* final block */
                    fin[(size_t)B * b + j] = t;
                    if (a == root && (first_bcast < 0 || t - 1 < first_bcast)) first_bcast = t - 1;
                }
            }
        }
        if (!progress) { rc = ORC_EDEADLOCK; goto done; }
    }
    int64_t tot = 0, f0 = 0;
    for (int i = 0; i < p; i++) {
        if (sfree[i] > tot) tot = sfree[i];
        if (rfree[i] > tot) tot = rfree[i];
        int64_t h0 = (i == root) ? ready[(size_t)i * b] : fin[(size_t)i * b];
        if (h0 > f0) f0 = h0;
    }
    int64_t rend = 0;
    for (int j = 0; j < b; j++)
        if (ready[(size_t)root * b + j] > rend) rend = ready[(size_t)root * b + j];
    stats[0] = tot;
    stats[1] = rend;
    stats[2] = ntransfers;
    stats[3] = f0;
    stats[4] = max_ops;
    stats[5] = first_bcast;

done:
    if (snd) for (int i = 0; i < p; i++) free(snd[i]);
    if (rcv) for (int i = 0; i < p; i++) free(rcv[i]);
    free(snd); free(rcv); free(nsnd); free(nrcv); free(sp); free(rp); free(sfree);
    free(rfree); free(red_left); free(red_end); free(left); free(ready); free(fin);
    free(early); free(T);
    return rc;
}
