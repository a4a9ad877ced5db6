/*
 * _ppasfast: a CPython extension with the two calls a serving loop makes on
 * every layer of every scheduler iteration, ppas_kv_append and
 * ppas_attention_step, forwarding to the C ABI of libppas.so (include/ppas.h)
 * with argument marshalling only.
 *
 * ctypes spends ~12 us of host time converting the 19 arguments of one
 * attention call; a decode-only step of a few rows takes less than that on
 * the GPU per layer, so with ctypes such steps are bound by the host.  Here
 * the arguments are parsed by PyArg_ParseTuple (pointers as Python ints,
 * the per-row length arrays through the buffer protocol: contiguous int32).
 */
#define PY_SSIZE_T_CLEAN
#include <Python.h>

#include "ppas.h"

static int int32_buffer(const Py_buffer *b, const char *what) {
    if (b->len % 4 != 0 || b->itemsize != 4 || !PyBuffer_IsContiguous(b, 'C')) {
        PyErr_Format(PyExc_TypeError, "%s must be a contiguous int32 buffer", what);
        return 0;
    }
    return 1;
}

/* attention_step(q, k_cache, v_cache, num_blocks, d_block_tables,
 *                max_blocks_per_seq, q_lens, ctx_lens, n_q_heads, n_kv_heads,
 *                head_dim, scale, out, out_is_fp32, workspace,
 *                workspace_bytes, d_err_flag, stream) -> ppas_status */
static PyObject *py_attention_step(PyObject *self, PyObject *args) {
    unsigned long long q, k, v, tables, out, ws, ws_bytes, err, stream;
    int num_blocks, width, hq, hk, d, out_fp32;
    float scale;
    Py_buffer ql, cl;
    (void)self;
    if (!PyArg_ParseTuple(args, "KKKiKiy*y*iiifKiKKKK", &q, &k, &v, &num_blocks, &tables, &width, &ql, &cl, &hq,
                          &hk, &d, &scale, &out, &out_fp32, &ws, &ws_bytes, &err, &stream))
        return NULL;
    PyObject *res = NULL;
    if (int32_buffer(&ql, "q_lens") && int32_buffer(&cl, "ctx_lens")) {
        if (ql.len != cl.len) {
            PyErr_SetString(PyExc_ValueError, "q_lens and ctx_lens differ in length");
        } else {
            const ppas_status st = ppas_attention_step(
                (const void *)(uintptr_t)q, (const void *)(uintptr_t)k, (const void *)(uintptr_t)v, num_blocks,
                (const int32_t *)(uintptr_t)tables, width, (const int32_t *)ql.buf, (const int32_t *)cl.buf,
                (int32_t)(ql.len / 4), hq, hk, d, scale, (void *)(uintptr_t)out, out_fp32, (void *)(uintptr_t)ws,
                (size_t)ws_bytes, (int32_t *)(uintptr_t)err, (void *)(uintptr_t)stream);
            res = PyLong_FromLong((long)st);
        }
    }
    PyBuffer_Release(&ql);
    PyBuffer_Release(&cl);
    return res;
}

/* kv_append(k_new, v_new, d_slot_mapping, n_tokens, k_cache, v_cache,
 *           num_blocks, n_kv_heads, head_dim, d_err_flag, stream) -> ppas_status */
static PyObject *py_kv_append(PyObject *self, PyObject *args) {
    unsigned long long kn, vn, slots, kc, vc, err, stream;
    int n_tokens, num_blocks, hk, d;
    (void)self;
    if (!PyArg_ParseTuple(args, "KKKiKKiiiKK", &kn, &vn, &slots, &n_tokens, &kc, &vc, &num_blocks, &hk, &d, &err,
                          &stream))
        return NULL;
    const ppas_status st = ppas_kv_append((const void *)(uintptr_t)kn, (const void *)(uintptr_t)vn,
                                          (const int32_t *)(uintptr_t)slots, n_tokens, (void *)(uintptr_t)kc,
                                          (void *)(uintptr_t)vc, num_blocks, hk, d, (int32_t *)(uintptr_t)err,
                                          (void *)(uintptr_t)stream);
    return PyLong_FromLong((long)st);
}

static PyMethodDef methods[] = {
    {"attention_step", py_attention_step, METH_VARARGS, "ppas_attention_step (see include/ppas.h)"},
    {"kv_append", py_kv_append, METH_VARARGS, "ppas_kv_append (see include/ppas.h)"},
    {NULL, NULL, 0, NULL},
};

static struct PyModuleDef module = {PyModuleDef_HEAD_INIT, "_ppasfast", NULL, -1, methods, NULL, NULL, NULL, NULL};

PyMODINIT_FUNC PyInit__ppasfast(void) { return PyModule_Create(&module); }
